"""GPU parity of the progressive schedule (Sec. 4.1: pre-LLM N_v -> N1, shallow
layer N1 -> N2 with each sample's visual heads, middle layer N2 -> N3 over all
heads) against the oracle run as the same chain on the CPU, and a check that
the three stages run without a host synchronisation (the whole schedule is
captured in one CUDA graph and replayed).

The oracle chain never takes a GPU result as input: it finds its own T, keep
sets, visual heads and compacted sequences. Where a GPU decision lies inside
the tie band of the oracle's, the two chains may part from there on; such a
sample is checked up to that stage only, and most samples must run the whole
chain.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_25332_gb300 import synth
from paper_2608_25332_gb300 import provip as P
from paper_2608_25332_gb300.schedule import ProgressiveSchedule
from parity import assert_close_rel, check_mask_band, check_topk_band, rtol_for

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
N_VIS = 6


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


def make(w, B, N3, pre_llm=True, shallow_heads="visual"):
    cpu = synth.schedule_inputs(w, batch=B)
    gpu = {k: {kk: (vv.to(DEV) if isinstance(vv, torch.Tensor) else vv) for kk, vv in v.items()}
           for k, v in cpu.items()}
    sched = ProgressiveSchedule(B, w.N_v, w.D, w.n_t[1], w.L_max, w.H_q, w.H_kv, w.D, w.P, w.keep_pre,
                                w.keep, N3, N_VIS, dtype=w.torch_dtype, device=DEV, pre_llm=pre_llm,
                                shallow_heads=shallow_heads)
    return cpu, gpu, sched


def run(sched, g):
    s = g["shallow"]
    return sched(g["pre"]["emb_v"], g["pre"]["emb_t"], g["pre"]["text_len"], s, g["middle"], s["vis_start"])


def as_bits(t):
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.view(torch.int32).numpy()


def check_chain(w, B, cpu, out, N3, pre_llm, shallow_heads, what):
    """Runs the oracle as the same chain and compares every stage; returns the
    number of samples that ran the whole chain."""
    rt = rtol_for(w.dtype)
    pre, sh, mid = cpu["pre"], cpu["shallow"], cpu["middle"]
    vis = sh["vis_start"]
    Ev = pre["emb_v"].float().numpy()
    Et = pre["emb_t"].float().numpy()
    Q1, K1 = sh["Q"].float().numpy(), sh["K"].float().numpy()
    Q2 = mid["Q"].float().numpy()
    g_mask = out["pre"]["mask"].cpu().numpy()
    o1, o2 = out["shallow"], out["middle"]
    g_idx2, g_idx3 = o1["idx"].cpu().numpy(), o2["idx"].cpu().numpy()
    full = 0
    for b in range(B):
        tl = int(pre["text_len"][b])
        # stage 1: critical text rows (and, with pre-LLM pruning, its keep set)
        r, T = oracle.crit_text(Et[b, :tl])
        check_mask_band(g_mask[b, :tl], r, rt, f"{what} T sample {b}")
        assert not g_mask[b, tl:].any()
        if not np.array_equal(g_mask[b, :tl].astype(bool), T.astype(bool)):
            continue
        rows_T = np.flatnonzero(T)
        if pre_llm:
            p = oracle.relevance(Et[b, :tl], T, Ev[b])
            check_topk_band(out["pre"]["idx"][b].cpu().numpy(), p, w.keep_pre, rt, f"{what} idx1 sample {b}")
        # stage 2: the shallow layer's heads (visual heads on the oracle's T, or all)
        sl1, ts1 = int(sh["seq_len"][b]), int(sh["text_start"][b])
        if shallow_heads == "visual":
            C = oracle.head_confidence(Q1[b, :sl1], K1[b, :sl1], ts1 + rows_T, vis, w.keep_pre)
            g_vis = o1["vis_heads"][b].cpu().numpy()
            check_topk_band(g_vis, C, N_VIS, rt, f"{what} visual heads sample {b}")
            heads = oracle.topk(C, N_VIS)
            if not np.array_equal(heads, g_vis):
                continue
        else:
            heads = np.arange(w.H_q)
        v1 = oracle.head_scores(Q1[b, :sl1], K1[b, :sl1], heads, np.arange(ts1, ts1 + tl), vis, w.keep_pre)
        assert_close_rel(o1["scores"][b].cpu().numpy(), v1, rt, f"{what} shallow v sample {b}")
        check_topk_band(g_idx2[b], v1, w.keep, rt, f"{what} idx2 sample {b}")
        idx2 = oracle.topk(v1, w.keep)
        if not np.array_equal(idx2, g_idx2[b]):
            continue
        src1 = oracle.compact_map(sl1, vis, w.keep_pre, idx2)
        sl2 = len(src1)
        assert int(o1["seq_len"][b]) == sl2
        np.testing.assert_array_equal(as_bits(o1["K"][b, :sl2].cpu()), oracle.gather_rows(as_bits(sh["K"][b]), src1))
        # stage 3: every head over the oracle's compacted keys
        K2 = oracle.gather_rows(K1[b], src1)
        ts2 = int(mid["text_start"][b])
        v2 = oracle.head_scores(Q2[b, :sl2], K2, np.arange(w.H_q), np.arange(ts2, ts2 + tl), vis, w.keep)
        assert_close_rel(o2["scores"][b].cpu().numpy(), v2, rt, f"{what} middle v sample {b}")
        check_topk_band(g_idx3[b], v2, N3, rt, f"{what} idx3 sample {b}")
        idx3 = oracle.topk(v2, N3)
        if not np.array_equal(idx3, g_idx3[b]):
            continue
        src2 = oracle.compact_map(sl2, vis, w.keep, idx3)
        n3 = len(src2)
        assert int(o2["seq_len"][b]) == n3
        for key in ("hidden", "K", "V"):
            exp = oracle.gather_rows(oracle.gather_rows(as_bits(sh[key][b]), src1), src2)
            np.testing.assert_array_equal(as_bits(o2[key][b, :n3].cpu()), exp)
        pos_exp = sh["pos"][:, b].numpy()[:, src1][:, src2]
        np.testing.assert_array_equal(o2["pos"][:, b, :n3].cpu().numpy(), pos_exp)
        full += 1
    return full


@pytest.mark.parametrize("name,B", [("llava15_7b_bf16_b16", 4), ("llava_next_7b_bf16_b8", 2)])
def test_schedule_matches_the_oracle_chain(name, B):
    w = synth.BY_NAME[name]
    N3 = w.keep // 2
    cpu, g, sched = make(w, B, N3)
    out = run(sched, g)
    torch.cuda.synchronize()
    full = check_chain(w, B, cpu, out, N3, True, "visual", name)
    assert full * 2 >= B, f"{name}: only {full} of {B} samples ran the whole chain"


@pytest.mark.parametrize("budget", synth.ABLATION_BUDGETS)
@pytest.mark.parametrize("heads", ["visual", "all"])
def test_ablation_without_pre_llm_pruning(budget, heads):
    """The ablation of Sec. 5: all 576 visual tokens reach the shallow layer;
    the paper's budgets after the shallow and the middle layer."""
    n2, n3 = budget
    w = synth.ablation_workload(n2)
    B = 2
    cpu, g, sched = make(w, B, n3, pre_llm=False, shallow_heads=heads)
    out = run(sched, g)
    torch.cuda.synchronize()
    full = check_chain(w, B, cpu, out, n3, False, heads, w.name)
    assert full >= 1, f"{w.name} {heads}: no sample ran the whole chain"


def test_schedule_needs_no_host_synchronisation():
    """The whole schedule captures into one CUDA graph (a host synchronisation
    inside it would abort the capture), and the replay gives the eager bits."""
    w = synth.BY_NAME["llava15_7b_bf16_b16"]
    cpu, g, sched = make(w, 4, w.keep // 2)
    out = run(sched, g)
    torch.cuda.synchronize()
    ref = {st: {k: v.clone() for k, v in out[st].items() if v is not None} for st in ("pre", "shallow", "middle")}
    for st in ("pre", "shallow", "middle"):
        for v in out[st].values():
            if v is not None:
                v.fill_(0) if v.dtype != torch.uint8 else v.zero_()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream(device=DEV)
    with torch.cuda.graph(graph, stream=s):
        run(sched, g)
    graph.replay()
    torch.cuda.synchronize()
    rows = ("hidden", "K", "V", "pos")  # rows past a sample's length are unspecified
    for st in ("pre", "shallow", "middle"):
        for k, v in ref[st].items():
            if k in rows:
                for b in range(v.shape[1] if k == "pos" else v.shape[0]):
                    n = int(ref[st]["seq_len"][b])
                    got, exp = (out[st][k][:, b, :n], v[:, b, :n]) if k == "pos" else (out[st][k][b, :n], v[b, :n])
                    assert torch.equal(got, exp), f"{st}.{k} sample {b} differs after the graph replay"
            else:
                assert torch.equal(out[st][k], v), f"{st}.{k} differs after the graph replay"
