"""GPU parity of the pre-LLM pass (Sec. 4.2-4.3) against the fp64 oracle.

The GPU always runs the full workload; the oracle checks the first samples in
full (crit text, relevance, top-N1, merge) and, where the exact merge would
take the oracle minutes (the anyres and video workloads), a sample of pruned
rows whose nearest centroid it recomputes on [those rows + all kept rows].
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_25332_gb300 import synth
from paper_2608_25332_gb300 import provip as P
from parity import assert_close_rel, check_mask_band, check_topk_band, rtol_for

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
N_CHECK = {"llava15_7b_f32_b1": 1, "llava15_7b_bf16_b16": 2, "llava15_13b_bf16_b32": 2,
           "llava_next_7b_bf16_b8": 1, "video_gqa_bf16_b1": 1}


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
        cpu = synth.pre_llm_inputs(w)
        gpu = {k: v.to(DEV) for k, v in cpu.items()}
        _cache.clear()
        _cache[name] = (w, cpu, gpu)
    return _cache[name]


def f64(t):
    return t.float().numpy().astype(np.float64)


@pytest.mark.parametrize("name", [w.name for w in synth.WORKLOADS])
def test_similarity_pass_matches_oracle(name):
    w, cpu, g = inputs(name)
    rt = rtol_for(w.dtype)
    mask, r = P.provip_crit_text(g["emb_t"], g["text_len"], want_r=True)
    res = P.provip_similarity_reduce(g["emb_v"], g["emb_t"], g["text_len"], w.keep_pre, want_merged=False)
    torch.cuda.synchronize()
    assert torch.equal(mask, res["mask"])
    for b in range(N_CHECK[name]):
        n = int(cpu["text_len"][b])
        Et, Ev = f64(cpu["emb_t"][b, :n]), f64(cpu["emb_v"][b])
        r_ref, m_ref = oracle.crit_text(Et)
        assert_close_rel(r[b, :n].cpu().numpy(), r_ref, rt, f"{name} r[{b}]")
        check_mask_band(mask[b, :n].cpu().numpy(), r_ref, rt, f"{name} T[{b}]")
        assert not mask[b, n:].any()
        # relevance with the GPU's own T only where T agrees with the oracle's
        m_gpu = mask[b, :n].cpu().numpy()
        p_ref = oracle.relevance(Et, m_ref, Ev)
        if np.array_equal(m_gpu, m_ref):
            assert_close_rel(res["p"][b].cpu().numpy(), p_ref, 0.0, f"{name} p[{b}]", atol=rt)
            check_topk_band(res["idx"][b].cpu().numpy(), p_ref, w.keep_pre, rt, f"{name} N1 keep[{b}]")
        # relevance given the oracle's T (a direct check of the p kernel)
        p_gpu = P.provip_relevance(g["emb_v"][b:b + 1], g["emb_t"][b:b + 1], g["text_len"][b:b + 1],
                                   torch.from_numpy(np.pad(m_ref, (0, w.n_t[1] - n))).to(DEV)[None])
        assert_close_rel(p_gpu[0].cpu().numpy(), p_ref, 0.0, f"{name} p|T_ref[{b}]", atol=rt)


def _cos_argmax_band(Ev, rows, keep, assign_gpu, tol):
    """the GPU's centroid of each sampled row is within tol of the best cosine"""
    K = Ev[keep]
    Kn = K / np.maximum(np.linalg.norm(K, axis=1, keepdims=True), 1e-300)
    X = Ev[rows]
    Xn = X / np.maximum(np.linalg.norm(X, axis=1, keepdims=True), 1e-300)
    C = Xn @ Kn.T
    best = C.max(axis=1)
    got = C[np.arange(len(rows)), assign_gpu[rows]]
    assert np.all(got >= best - tol), "a nearest-centroid choice is off by more than the tolerance"


@pytest.mark.parametrize("name", [w.name for w in synth.WORKLOADS])
def test_merge_matches_oracle(name):
    """The whole batch in one call (the launch configuration the benchmark
    times: several kept-row splits, ragged last tiles), each sample with the
    oracle's own keep set; the first and last samples checked against the
    oracle."""
    w, cpu, g = inputs(name)
    keeps = []
    for b in range(w.B):
        n = int(cpu["text_len"][b])
        Et = f64(cpu["emb_t"][b, :n])
        _, m_ref = oracle.crit_text(Et)
        keeps.append(oracle.topk(oracle.relevance(Et, m_ref, f64(cpu["emb_v"][b])), w.keep_pre))
    assign, merged = P.provip_merge(g["emb_v"], torch.from_numpy(np.stack(keeps)).to(DEV))
    torch.cuda.synchronize()
    for b in sorted({0, w.B - 1}):
        _check_merge_sample(w, f64(cpu["emb_v"][b]), keeps[b], assign[b].cpu().numpy(),
                            merged[b].float().cpu().numpy().astype(np.float64), f"{name}[{b}]")


def _check_merge_sample(w, Ev, keep, a_gpu, mg, what):
    pruned = np.setdiff1d(np.arange(w.N_v), keep)
    assert np.array_equal(a_gpu[keep], np.arange(w.keep_pre)), f"{what}: kept rows must be their own centroid"
    exact = w.N_v <= 1000
    if exact:
        a_ref, mg_ref = oracle.merge(Ev, keep)
        rows = pruned
    else:
        rows = np.sort(np.random.default_rng(5).choice(pruned, 48, replace=False))
        sub = np.r_[rows, keep]
        order = np.argsort(sub)
        sub_sorted = sub[order]
        kpos = np.searchsorted(sub_sorted, keep)
        a_sub, _ = oracle.merge(Ev[sub_sorted], kpos)
        a_ref = np.full(w.N_v, -1)
        a_ref[sub_sorted] = a_sub
    tol = 1e-4 if w.dtype == "bf16" else 1e-6
    same = a_gpu[rows] == a_ref[rows]
    if not same.all():
        _cos_argmax_band(Ev, rows[~same], keep, a_gpu, tol)
    assert same.mean() > 0.95, what
    if exact:
        # centroids whose member set is identical: within one output ulp
        ok = np.array([np.array_equal(np.flatnonzero(a_gpu == a), np.flatnonzero(a_ref == a))
                       for a in range(w.keep_pre)])
        ulp = np.spacing(np.abs(mg_ref).astype(np.float32)).astype(np.float64) if w.dtype == "f32" else \
            2.0 ** (np.floor(np.log2(np.maximum(np.abs(mg_ref), 1e-30))) - 7)
        err = np.abs(mg - mg_ref)
        assert np.all(err[ok] <= ulp[ok] * 1.0001 + 1e-37), f"{what}: merged rows beyond one ulp"
    else:
        # at full size: every merged row is the mean of its GPU-assigned members
        for a in np.random.default_rng(6).choice(w.keep_pre, 16, replace=False):
            mem = np.flatnonzero(a_gpu == a)
            expect = Ev[mem].mean(axis=0)
            np.testing.assert_allclose(mg[a], expect, rtol=8e-3, atol=1e-6)


@pytest.mark.parametrize("name", [w.name for w in synth.WORKLOADS])
def test_reduce_merge_agrees_with_the_merge_call(name):
    """The merge inside provip_similarity_reduce takes its inverse norms from the
    relevance kernel; the stand-alone merge computes its own. On the same kept
    set both give the same centroids, apart from rows whose nearest kept row is
    a near tie that the two fp32 norm orders may break differently."""
    w, cpu, g = inputs(name)
    res = P.provip_similarity_reduce(g["emb_v"], g["emb_t"], g["text_len"], w.keep_pre, want_merged=True)
    _, merged = P.provip_merge(g["emb_v"], res["idx"])
    torch.cuda.synchronize()
    same = (res["merged"] == merged).all(dim=2).float().mean().item()
    assert same >= 0.98, f"{name}: only {same:.3f} of the merged rows agree"
