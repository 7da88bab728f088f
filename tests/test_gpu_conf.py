"""GPU parity of visual-head identification (Sec. 4.4: head confidence C^h over
the critical text rows, the N_vis most confident heads) and of pruning with
those heads, against the fp64 oracle; and of the all-heads variant used at the
middle pruning layer.

Inputs: the in-LLM workloads with planted visual heads (synth.in_llm_inputs
with visual_heads=True), on a few samples per workload, each with a seeded
critical-row mask (one sample takes every text row).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_25332_gb300 import synth
from paper_2608_25332_gb300 import provip as P
from parity import assert_close_rel, check_topk_band, rtol_for

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
N_VIS = 6  # visual heads per pruning layer in the paper's evaluation (Sec. 5.1)
BATCH = {"llava15_7b_f32_b1": 1, "llava15_7b_bf16_b16": 4, "llava15_13b_bf16_b32": 3,
         "llava_next_7b_bf16_b8": 3, "video_gqa_bf16_b1": 1}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


def crit_masks(cpu, B, N_t_max, seed):
    """Seeded critical-row masks; sample 0 keeps every text row."""
    rng = np.random.default_rng(seed)
    m = (rng.random((B, N_t_max)) < 0.4).astype(np.uint8)
    m[0, :] = 1
    for b in range(B):
        m[b, int(cpu["text_len"][b]):] = 0
        if m[b].sum() == 0:
            m[b, 0] = 1
    return m


_cache = {}


def case(name):
    if name not in _cache:
        w = synth.BY_NAME[name]
        B = BATCH[name]
        cpu = synth.in_llm_inputs(w, batch=B, visual_heads=True)
        gpu = {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
        mask = crit_masks(cpu, B, w.n_t[1], w.seed)
        gpu["crit_mask"] = torch.from_numpy(mask).to(DEV)
        Q = cpu["Q"].float().numpy()
        K = cpu["K"].float().numpy()
        C = []
        for b in range(B):
            sl, ts = int(cpu["seq_len"][b]), int(cpu["text_start"][b])
            rows = ts + np.flatnonzero(mask[b])
            C.append(oracle.head_confidence(Q[b, :sl], K[b, :sl], rows, cpu["vis_start"], cpu["N_v"]))
        _cache.clear()
        _cache[name] = (w, B, cpu, gpu, mask, np.stack(C))
    return _cache[name]


def conf_tol(dtype):
    return rtol_for(dtype)


def check_conf(conf_gpu, C_ref, rtol, what):
    # C is a sum of non-negative variances: relative per head, with a floor at
    # a small fraction of the sample's largest C for near-zero heads
    for b in range(C_ref.shape[0]):
        assert_close_rel(conf_gpu[b], C_ref[b], rtol, f"{what} sample {b}", atol=rtol * 1e-2 * C_ref[b].max())


TC_ALGOS = [P.ALGO_TCGEN05_STREAM, P.ALGO_TCGEN05_CLUSTER, P.ALGO_TCGEN05_TWOPASS]
CASES = [(w.name, a) for w in synth.WORKLOADS
         for a in ([P.ALGO_SIMT] if w.dtype == "f32" else [P.ALGO_SIMT] + TC_ALGOS)]


@pytest.mark.parametrize("name,algo", CASES)
def test_confidence_and_visual_heads_match_oracle(name, algo):
    w, B, cpu, g, mask, C_ref = case(name)
    vis, conf = P.provip_head_confidence(g["Q"], g["K"], g["text_start"], g["text_len"], g["seq_len"],
                                         g["vis_start"], g["N_v"], N_VIS, crit_mask=g["crit_mask"],
                                         algo=algo, N_t_max=w.n_t[1])
    torch.cuda.synchronize()
    rt = conf_tol(w.dtype)
    check_conf(conf.cpu().numpy(), C_ref, rt, f"{name} algo={algo} C")
    vis = vis.cpu().numpy()
    for b in range(B):
        check_topk_band(vis[b], C_ref[b], N_VIS, rt, f"{name} algo={algo} visual heads sample {b}")


def test_confidence_paths_agree_on_the_selection():
    """The three kernel families pick the same heads wherever the oracle's
    margin is clear, and the one-pass path is deterministic."""
    name = "llava_next_7b_bf16_b8"
    w, B, cpu, g, mask, C_ref = case(name)
    runs = [P.provip_head_confidence(g["Q"], g["K"], g["text_start"], g["text_len"], g["seq_len"],
                                     g["vis_start"], g["N_v"], N_VIS, crit_mask=g["crit_mask"], algo=a,
                                     N_t_max=w.n_t[1])
            for a in (P.ALGO_TCGEN05, P.ALGO_TCGEN05, P.ALGO_TCGEN05_STREAM, P.ALGO_TCGEN05_CLUSTER,
                      P.ALGO_TCGEN05_TWOPASS, P.ALGO_SIMT)]
    torch.cuda.synchronize()
    assert torch.equal(runs[0][1], runs[1][1]) and torch.equal(runs[0][0], runs[1][0])
    for vis, _ in runs[2:]:
        for b in range(B):
            check_topk_band(vis[b].cpu().numpy(), C_ref[b], N_VIS, 2e-3, f"{name} sample {b}")


def test_uniform_attention_gives_zero_confidence():
    """Q = 0: every attention row is uniform over its causal keys, so every
    variance is zero and the ties go to the lowest heads."""
    w = synth.BY_NAME["llava15_7b_bf16_b16"]
    cpu = synth.in_llm_inputs(w, batch=2)
    g = {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
    Q = torch.zeros_like(g["Q"])
    for algo in (P.ALGO_TCGEN05_STREAM, P.ALGO_TCGEN05_CLUSTER, P.ALGO_TCGEN05_TWOPASS, P.ALGO_SIMT):
        vis, conf = P.provip_head_confidence(Q, g["K"], g["text_start"], g["text_len"], g["seq_len"],
                                             g["vis_start"], g["N_v"], 4, algo=algo, N_t_max=w.n_t[1])
        torch.cuda.synchronize()
        assert float(conf.abs().max()) < 1e-12, algo
        assert vis.cpu().tolist() == [[0, 1, 2, 3]] * 2


def test_empty_critical_set_selects_the_first_heads():
    w = synth.BY_NAME["llava15_7b_bf16_b16"]
    cpu = synth.in_llm_inputs(w, batch=2, visual_heads=True)
    g = {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
    empty = torch.zeros((2, w.n_t[1]), dtype=torch.uint8, device=DEV)
    vis, conf = P.provip_head_confidence(g["Q"], g["K"], g["text_start"], g["text_len"], g["seq_len"],
                                         g["vis_start"], g["N_v"], 3, crit_mask=empty, N_t_max=w.n_t[1])
    torch.cuda.synchronize()
    assert float(conf.abs().max()) == 0.0
    assert vis.cpu().tolist() == [[0, 1, 2]] * 2


E2E = [(w.name, a) for w in synth.WORKLOADS
       for a in ([P.ALGO_SIMT] if w.dtype == "f32" else [P.ALGO_TCGEN05_STREAM, P.ALGO_TCGEN05_CLUSTER])]


@pytest.mark.parametrize("name,algo", E2E)
def test_prune_visual_heads_end_to_end(name, algo):
    """Visual heads within the tie band of the oracle's C; v of the chosen heads
    within tolerance of the oracle's; keep set exact outside the band;
    compaction exact; and, for the cluster and CUDA-core forms, bit-identical
    to provip_prune (same form) on each sample alone with head_list = its
    visual heads."""
    w, B, cpu, g, mask, C_ref = case(name)
    n_vis = min(N_VIS, w.H_q)
    step = P.VisualHeadsPruneStep(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], w.n_t[1], g["N_v"],
                                  w.keep, n_vis, algo=algo)
    out = step(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], g["text_start"], g["text_len"],
               g["seq_len"], g["vis_start"], crit_mask=g["crit_mask"])
    torch.cuda.synchronize()
    rt = rtol_for(w.dtype)
    vis = out["vis_heads"].cpu().numpy()
    scores = out["scores"].cpu().numpy()
    idx = out["idx"].cpu().numpy()
    check_conf(out["conf"].cpu().numpy(), C_ref, rt, f"{name} C")
    Q = cpu["Q"].float().numpy()
    K = cpu["K"].float().numpy()
    for b in range(B):
        check_topk_band(vis[b], C_ref[b], n_vis, rt, f"{name} visual heads sample {b}")
        sl, ts, tl = int(cpu["seq_len"][b]), int(cpu["text_start"][b]), int(cpu["text_len"][b])
        v_ref = oracle.head_scores(Q[b, :sl], K[b, :sl], vis[b], np.arange(ts, ts + tl),
                                   cpu["vis_start"], cpu["N_v"])
        assert_close_rel(scores[b], v_ref, rt, f"{name} v sample {b}")
        check_topk_band(idx[b], v_ref, w.keep, rt, f"{name} keep sample {b}")
        n = sl - cpu["N_v"] + w.keep
        src = np.r_[np.arange(cpu["vis_start"]), cpu["vis_start"] + idx[b],
                    np.arange(cpu["vis_start"] + cpu["N_v"], sl)]
        for key in ("hidden", "K", "V"):
            exp = oracle.gather_rows(cpu[key][b].view(torch.int16 if w.dtype == "bf16" else torch.int32).numpy(), src)
            got = out[key][b, :n].cpu().view(torch.int16 if w.dtype == "bf16" else torch.int32).numpy()
            np.testing.assert_array_equal(got, exp)
        # the same sample pruned alone with its visual heads as an explicit list
        one = {k: (v[b:b + 1].contiguous() if isinstance(v, torch.Tensor) and v.dim() >= 1 and k != "pos"
                   else v) for k, v in g.items()}
        one["pos"] = g["pos"][:, b:b + 1].contiguous()
        ref = P.provip_prune(one["Q"], one["K"], one["V"], one["hidden"], one["pos"], vis[b].tolist(),
                             one["text_start"], one["text_len"], one["seq_len"], g["vis_start"], g["N_v"],
                             w.keep, algo=algo, N_t_max=w.n_t[1])
        torch.cuda.synchronize()
        # every form computes a head's partial scores with the same arithmetic
        # whether or not it keeps confidence statistics: the same bits
        assert torch.equal(ref["scores"][0], out["scores"][b]), f"{name} sample {b}: scores differ"
        assert torch.equal(ref["idx"][0], out["idx"][b])


def test_prune_visual_heads_overlapped_calls_match_serial():
    """PROVIP_PRUNE_OVERLAP_PREVIOUS over rotating independent batches gives the
    bits of serial calls."""
    w = synth.BY_NAME["llava_next_7b_bf16_b8"]
    copies = []
    for s in range(3):
        cpu = synth.in_llm_inputs(w, seed=w.seed + 77 * s, visual_heads=True)
        copies.append({k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()})
    g0 = copies[0]
    mk = lambda fl: P.VisualHeadsPruneStep(g0["Q"], g0["K"], g0["V"], g0["hidden"], g0["pos"], w.n_t[1],
                                           g0["N_v"], g0["keep"], N_VIS, flags=fl)
    serial, ov = mk(0), mk(P.PRUNE_OVERLAP_PREVIOUS)
    keys = ("idx", "scores", "vis_heads", "conf", "hidden", "K", "V", "pos", "seq_len")
    call = lambda st, c: st(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"],
                            c["seq_len"], c["vis_start"])
    ref = []
    for i in range(3):
        o = call(serial, copies[i])
        ref.append({k: o[k].clone() for k in keys})
    torch.cuda.synchronize()
    snaps = []
    for i in range(6):
        o = call(ov, copies[i % 3])
        snaps.append({k: o[k].clone() for k in keys})  # ordered on the stream after the call
    torch.cuda.synchronize()
    for i, s in enumerate(snaps):
        for k in keys:
            assert torch.equal(s[k], ref[i % 3][k]), f"call {i}: {k} differs"


@pytest.mark.parametrize("name", ["llava15_7b_bf16_b16", "llava_next_7b_bf16_b8", "video_gqa_bf16_b1",
                                  "llava15_7b_f32_b1"])
def test_all_heads_prune_matches_oracle(name):
    """The middle-layer variant (every head; Sec. 4.4): a null head list equals
    the explicit list of all heads bit for bit, and matches the oracle."""
    w = synth.BY_NAME[name]
    B = min(BATCH[name], 2)
    cpu = synth.in_llm_inputs(w, batch=B)
    g = {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
    args = (g["text_start"], g["text_len"], g["seq_len"], g["vis_start"], g["N_v"], g["keep"])
    a = P.provip_prune(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], None, *args, N_t_max=w.n_t[1])
    b_ = P.provip_prune(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], list(range(w.H_q)), *args,
                        N_t_max=w.n_t[1])
    torch.cuda.synchronize()
    assert torch.equal(a["scores"], b_["scores"]) and torch.equal(a["idx"], b_["idx"])
    Q = cpu["Q"].float().numpy()
    K = cpu["K"].float().numpy()
    rt = rtol_for(w.dtype)
    for b in range(B):
        sl, ts, tl = int(cpu["seq_len"][b]), int(cpu["text_start"][b]), int(cpu["text_len"][b])
        v_ref = oracle.head_scores(Q[b, :sl], K[b, :sl], np.arange(w.H_q), np.arange(ts, ts + tl),
                                   cpu["vis_start"], cpu["N_v"])
        assert_close_rel(a["scores"][b].cpu().numpy(), v_ref, rt, f"{name} all heads sample {b}")
        check_topk_band(a["idx"][b].cpu().numpy(), v_ref, g["keep"], rt, f"{name} keep sample {b}")


@pytest.mark.parametrize("seed", range(5))
def test_confidence_random_shapes(seed):
    """Seeded random shapes for head confidence and the visual heads: batch,
    GQA ratio, heads, prefix, visual count (ragged against the 128-key tiles),
    ragged text lengths with a random critical-row mask, N_vis; every form."""
    rng = np.random.default_rng(5000 + seed)
    B = int(rng.integers(1, 4))
    Hkv = int(rng.choice([1, 2, 4]))
    Hq = Hkv * int(rng.choice([2, 4]))
    nsys = int(rng.integers(0, 40))
    nv = int(rng.integers(16, 600))
    tls = rng.integers(1, 200, B).astype(np.int32)
    n_vis = int(rng.integers(1, Hq + 1))
    Ntm = int(tls.max())
    Lm = nsys + nv + Ntm
    Q = rng.standard_normal((B, Lm, Hq, 128)).astype(np.float32)
    K = rng.standard_normal((B, Lm, Hkv, 128)).astype(np.float32)
    Q[:, :, 0] *= 3.0  # one sharp query head: confidences spread out
    sl = (nsys + nv + tls).astype(np.int32)
    ts = np.full(B, nsys + nv, np.int32)
    mask = (rng.random((B, Ntm)) < 0.5).astype(np.uint8)
    for b in range(B):
        Q[b, sl[b]:] = np.nan
        K[b, sl[b]:] = np.nan
        mask[b, tls[b]:] = 0
        if mask[b].sum() == 0:
            mask[b, 0] = 1
    Qt, Kt = torch.from_numpy(Q).to(torch.bfloat16), torch.from_numpy(K).to(torch.bfloat16)
    Qn, Kn = Qt.float().numpy(), Kt.float().numpy()
    C_ref = np.stack([oracle.head_confidence(Qn[b, :sl[b]], Kn[b, :sl[b]], ts[b] + np.flatnonzero(mask[b]), nsys, nv)
                      for b in range(B)])
    g = [torch.from_numpy(x).to(DEV) for x in (ts, tls, sl, mask)]
    for algo in (P.ALGO_TCGEN05_STREAM, P.ALGO_TCGEN05_CLUSTER, P.ALGO_TCGEN05_TWOPASS, P.ALGO_SIMT):
        vis, conf = P.provip_head_confidence(Qt.to(DEV), Kt.to(DEV), g[0], g[1], g[2], nsys, nv, n_vis,
                                             crit_mask=g[3], algo=algo, N_t_max=Ntm)
        torch.cuda.synchronize()
        what = f"seed {seed} (B={B} Hq={Hq} Hkv={Hkv} nsys={nsys} nv={nv} tl={tls.tolist()} n_vis={n_vis}) algo {algo}"
        check_conf(conf.cpu().numpy(), C_ref, 2e-3, what + " C")
        vis = vis.cpu().numpy()
        for b in range(B):
            check_topk_band(vis[b], C_ref[b], n_vis, 2e-3, what + f" visual heads sample {b}")
