"""GPU parity of the in-LLM pruning step (Sec. 4.4) against the fp64 oracle.

Every workload runs at its full size; the oracle computes every sample (each
sample takes it well under a second). Both kernel families (CUDA-core and
tcgen05) are checked for bf16.
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


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


_cache = {}


def inputs(name):
    if name not in _cache:
        w = synth.BY_NAME[name]
        cpu = synth.in_llm_inputs(w)
        gpu = {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
        _cache.clear()
        _cache[name] = (w, cpu, gpu)
    return _cache[name]


def oracle_scores(w, cpu):
    Q = cpu["Q"].float().numpy()
    K = cpu["K"].float().numpy()
    heads = cpu["head_list"].numpy()
    out = []
    for b in range(Q.shape[0]):
        sl = int(cpu["seq_len"][b])
        ts, tl = int(cpu["text_start"][b]), int(cpu["text_len"][b])
        out.append(oracle.head_scores(Q[b, :sl], K[b, :sl], heads, np.arange(ts, ts + tl),
                                      cpu["vis_start"], cpu["N_v"]))
    return np.stack(out)


_ref = {}


def ref_scores(name):
    if name not in _ref:
        w, cpu, _ = inputs(name)
        _ref.clear()
        _ref[name] = oracle_scores(w, cpu)
    return _ref[name]


CASES = [(w.name, a) for w in synth.WORKLOADS
         for a in ([P.ALGO_SIMT] if w.dtype == "f32" else
                   [P.ALGO_SIMT, P.ALGO_TCGEN05, P.ALGO_TCGEN05_TWOPASS, P.ALGO_TCGEN05_STREAM,
                    P.ALGO_TCGEN05_CLUSTER])]


@pytest.mark.parametrize("name,algo", CASES)
def test_head_scores_match_oracle(name, algo):
    w, cpu, g = inputs(name)
    s = P.provip_head_scores(g["Q"], g["K"], g["head_list"], g["text_start"], g["text_len"],
                             g["seq_len"], g["vis_start"], g["N_v"], algo=algo, N_t_max=w.n_t[1])
    torch.cuda.synchronize()
    assert_close_rel(s.cpu().numpy(), ref_scores(name), rtol_for(w.dtype), f"{name} algo={algo}")


@pytest.mark.parametrize("name", [w.name for w in synth.WORKLOADS])
def test_prune_end_to_end(name):
    """scores within tolerance, keep set exact outside the tie band, compaction exact."""
    w, cpu, g = inputs(name)
    ref = ref_scores(name)
    out = P.provip_prune(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], g["head_list"], g["text_start"],
                         g["text_len"], g["seq_len"], g["vis_start"], g["N_v"], g["keep"], N_t_max=w.n_t[1])
    torch.cuda.synchronize()
    rt = rtol_for(w.dtype)
    assert_close_rel(out["scores"].cpu().numpy(), ref, rt, f"{name} fused scores")
    idx = out["idx"].cpu().numpy()
    hid, Kc, Vc = (out[k].cpu() for k in ("hidden", "K", "V"))
    pos = out["pos"].cpu().numpy()
    slo = out["seq_len"].cpu().numpy()
    for b in range(w.B):
        check_topk_band(idx[b], ref[b], w.keep, rt, f"{name} sample {b}")
        sl = int(cpu["seq_len"][b])
        ref_idx = oracle.topk(ref[b], w.keep)
        n = sl - g["N_v"] + w.keep
        assert slo[b] == n
        if np.array_equal(ref_idx, idx[b]):
            src = oracle.compact_map(sl, g["vis_start"], g["N_v"], ref_idx)
        else:  # inside the tie band: the kept rows must still be those the GPU reports
            src = np.r_[np.arange(g["vis_start"]), g["vis_start"] + idx[b],
                        np.arange(g["vis_start"] + g["N_v"], sl)]
        for got, full in ((hid, cpu["hidden"]), (Kc, cpu["K"]), (Vc, cpu["V"])):
            exp = oracle.gather_rows(full[b].view(torch.int16).numpy(), src)
            np.testing.assert_array_equal(got[b, :n].view(torch.int16).numpy(), exp)
        for p in range(pos.shape[0]):
            np.testing.assert_array_equal(pos[p, b, :n], cpu["pos"][p, b].numpy()[src])


def test_fused_and_standalone_scores_are_identical():
    name = "llava15_7b_bf16_b16"
    w, cpu, g = inputs(name)
    s = P.provip_head_scores(g["Q"], g["K"], g["head_list"], g["text_start"], g["text_len"],
                             g["seq_len"], g["vis_start"], g["N_v"], N_t_max=w.n_t[1])
    out = P.provip_prune(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], g["head_list"], g["text_start"],
                         g["text_len"], g["seq_len"], g["vis_start"], g["N_v"], g["keep"], N_t_max=w.n_t[1])
    torch.cuda.synchronize()
    assert torch.equal(s, out["scores"])
    idx2 = P.provip_topk(s, g["keep"])
    assert torch.equal(idx2, out["idx"])


@pytest.mark.parametrize("algo", ["ALGO_AUTO", "ALGO_TCGEN05_STREAM", "ALGO_TCGEN05_CLUSTER"])
@pytest.mark.parametrize("name", ["llava_next_7b_bf16_b8", "video_gqa_bf16_b1"])
def test_overlapped_calls_match_serial_calls(name, algo):
    """PROVIP_PRUNE_OVERLAP_PREVIOUS: back-to-back calls on three different batches
    sharing one workspace give the same bits as calls separated by a sync, for
    each tensor-core form of the head scores."""
    algo = getattr(P, algo)
    w, cpu, g0 = inputs(name)
    batches = [g0] + [{k: (v.to(DEV) if isinstance(v, torch.Tensor) else v)
                       for k, v in synth.in_llm_inputs(w, seed=w.seed + 77 + i).items()} for i in range(2)]
    ws = P.workspace(P.lib().provip_prune_workspace_size(w.B, w.L_max, w.H_sel, w.n_t[1], w.keep_pre,
                                                         algo, P.BF16), DEV)
    def run(flags, sync):
        outs = []
        for c in batches:
            st = P.PruneStep(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["head_list"], w.n_t[1], c["N_v"],
                             c["keep"], algo=algo, flags=flags, ws=ws)
            outs.append(st(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"],
                           c["seq_len"], c["vis_start"]))
            if sync:
                torch.cuda.synchronize()
        torch.cuda.synchronize()
        return [{k: v.clone() for k, v in o.items() if v is not None} for o in outs]
    serial = run(0, True)
    for rep in range(3):
        over = run(P.PRUNE_OVERLAP_PREVIOUS, False)
        for a, b in zip(serial, over):
            for k in a:
                assert torch.equal(a[k], b[k]), f"overlapped call differs in {k} (rep {rep})"


def _small_case(seed, B=3, Hq=6, Hkv=2, nsys=5, nv=37, tls=(1, 9, 130), dtype=torch.bfloat16):
    """ragged: 37 visual columns, a one-row sample and a 130-row sample (two row blocks)."""
    rng = np.random.default_rng(seed)
    Ntm = max(tls)
    Lm = nsys + nv + Ntm
    Q = rng.standard_normal((B, Lm, Hq, 128)).astype(np.float32)
    K = rng.standard_normal((B, Lm, Hkv, 128)).astype(np.float32)
    K[:, 0] *= 6.0
    tl = np.array(tls, np.int32)
    sl = (nsys + nv + tl).astype(np.int32)
    for b in range(B):
        Q[b, sl[b]:] = np.nan
        K[b, sl[b]:] = np.nan
    Qt = torch.from_numpy(Q).to(dtype)
    Kt = torch.from_numpy(K).to(dtype)
    return dict(Q=Qt, K=Kt, tl=tl, sl=sl, ts=np.full(B, nsys + nv, np.int32), nsys=nsys, nv=nv, Ntm=Ntm)


@pytest.mark.parametrize("algo", [P.ALGO_SIMT, P.ALGO_TCGEN05, P.ALGO_TCGEN05_TWOPASS, P.ALGO_TCGEN05_STREAM,
                                  P.ALGO_TCGEN05_CLUSTER])
def test_head_scores_ragged_and_masked_rows(algo):
    c = _small_case(7)
    heads = [1, 2, 5]
    B = c["Q"].shape[0]
    mask = (np.random.default_rng(3).random((B, c["Ntm"])) < 0.5).astype(np.uint8)
    mask[:, 0] = 1
    Qd, Kd = c["Q"].to(DEV), c["K"].to(DEV)
    ts, tl, sl = (torch.from_numpy(x).to(DEV) for x in (c["ts"], c["tl"], c["sl"]))
    for rm in (None, mask):
        s = P.provip_head_scores(Qd, Kd, heads, ts, tl, sl, c["nsys"], c["nv"], algo=algo, N_t_max=c["Ntm"],
                                 row_mask=None if rm is None else torch.from_numpy(rm).to(DEV))
        torch.cuda.synchronize()
        Qn, Kn = c["Q"].float().numpy(), c["K"].float().numpy()
        for b in range(B):
            rows = [c["ts"][b] + j for j in range(c["tl"][b]) if rm is None or rm[b, j]]
            ref = oracle.head_scores(Qn[b, :c["sl"][b]], Kn[b, :c["sl"][b]], heads, rows, c["nsys"], c["nv"])
            assert_close_rel(s[b].cpu().numpy(), ref, 2e-3, f"small case b={b} mask={rm is not None}")


@pytest.mark.parametrize("nv,tl", [(4000, 200), (8000, 316)])
def test_head_scores_long_sequences(nv, tl):
    # 4205 keys: 33 chunks -> clusters of 9 CTAs with 4 chunks each; 8321 keys: more
    # than 64 chunks -> the two-pass kernels take over
    c = _small_case(9, B=1, Hq=4, Hkv=2, nsys=5, nv=nv, tls=(tl,))
    heads = [0, 3]
    Qd, Kd = c["Q"].to(DEV), c["K"].to(DEV)
    ts, tlt, sl = (torch.from_numpy(x).to(DEV) for x in (c["ts"], c["tl"], c["sl"]))
    Qn, Kn = c["Q"].float().numpy(), c["K"].float().numpy()
    ref = oracle.head_scores(Qn[0, :c["sl"][0]], Kn[0, :c["sl"][0]], heads,
                             np.arange(c["ts"][0], c["ts"][0] + c["tl"][0]), c["nsys"], c["nv"])
    for algo in (P.ALGO_TCGEN05, P.ALGO_TCGEN05_TWOPASS, P.ALGO_SIMT, P.ALGO_TCGEN05_STREAM,
                 P.ALGO_TCGEN05_CLUSTER):
        s = P.provip_head_scores(Qd, Kd, heads, ts, tlt, sl, c["nsys"], c["nv"], algo=algo, N_t_max=c["Ntm"])
        torch.cuda.synchronize()
        assert_close_rel(s[0].cpu().numpy(), ref, 2e-3, f"long L={c['sl'][0]} algo={algo}")


def test_topk_matches_oracle_with_ties():
    for (B, N, k, seed) in [(4, 1000, 1, 1), (3, 960, 320, 2), (2, 9216, 2304, 3), (1, 577, 577, 4),
                            (2, 49152, 4099, 5), (5, 33, 17, 6)]:
        s = synth.random_scores(B, N, seed, ties=True)
        idx = P.provip_topk(s.to(DEV), k).cpu().numpy()
        for b in range(B):
            np.testing.assert_array_equal(idx[b], oracle.topk(s[b].numpy().astype(np.float64), k))
    # all equal: the lowest indices
    s = torch.full((2, 100), 0.25)
    assert P.provip_topk(s.to(DEV), 7).cpu().numpy().tolist() == [list(range(7))] * 2


@pytest.mark.parametrize("name", ["llava15_7b_bf16_b16", "video_gqa_bf16_b1", "llava15_7b_f32_b1"])
def test_compact_bit_exact(name):
    w, cpu, g = inputs(name)
    rng = np.random.default_rng(11)
    idx = np.stack([np.sort(rng.choice(g["N_v"], w.keep, replace=False)) for _ in range(w.B)]).astype(np.int32)
    out = P.provip_compact(torch.from_numpy(idx).to(DEV), g["hidden"], g["K"], g["V"], g["pos"], g["seq_len"],
                           g["vis_start"], g["N_v"])
    torch.cuda.synchronize()
    view = torch.int32 if w.dtype == "f32" else torch.int16
    for b in range(w.B):
        sl = int(cpu["seq_len"][b])
        src = oracle.compact_map(sl, g["vis_start"], g["N_v"], idx[b])
        n = len(src)
        assert int(out["seq_len"][b]) == n
        for key in ("hidden", "K", "V"):
            np.testing.assert_array_equal(out[key][b, :n].cpu().view(view).numpy(),
                                          oracle.gather_rows(cpu[key][b].view(view).numpy(), src))
        for p in range(w.P):
            np.testing.assert_array_equal(out["pos"][p, b, :n].cpu().numpy(),
                                          oracle.gather_rows(cpu["pos"][p, b].numpy(), src))


@pytest.mark.parametrize("name,lanes", [("llava_next_7b_bf16_b8", 2), ("video_gqa_bf16_b1", 5)])
def test_concurrent_lanes_match_serial_calls(name, lanes):
    """The bench's multi-stream configuration: independent batches on their own
    streams, each with its own outputs and workspace, several steps per lane,
    running at the same time, give the bits of the same calls made serially."""
    w = synth.BY_NAME[name]
    batches = [{k: (v.to(DEV) if isinstance(v, torch.Tensor) else v)
                for k, v in synth.in_llm_inputs(w, seed=w.seed + 31 * i).items()} for i in range(lanes)]
    steps = [P.PruneStep(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["head_list"], w.n_t[1], c["N_v"],
                         c["keep"], algo=P.ALGO_TCGEN05_STREAM, flags=P.PRUNE_OVERLAP_PREVIOUS) for c in batches]

    def call(i, stream=None):
        c = batches[i]
        return steps[i](c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"],
                        c["seq_len"], c["vis_start"], stream=stream)

    serial = []
    for i in range(lanes):
        o = call(i)
        torch.cuda.synchronize()
        serial.append({k: v.clone() for k, v in o.items() if v is not None})
    streams = [torch.cuda.Stream(device=DEV) for _ in range(lanes)]
    for rep in range(4):
        for i in range(lanes):
            call(i, streams[i])
    torch.cuda.synchronize()
    for i in range(lanes):
        for k, v in serial[i].items():
            got = getattr(steps[i], {"hidden": "hidden_out", "K": "K_out", "V": "V_out", "pos": "pos_out",
                                     "idx": "idx", "seq_len": "seq_len_out", "scores": "scores"}[k])
            assert torch.equal(got, v), f"{name} lane {i}: {k} differs under concurrency"
