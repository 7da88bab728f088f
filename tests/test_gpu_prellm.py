"""GPU parity of the pre-LLM pass (Sec. 4.2-4.3) against the fp64 oracle.

Every sample of every workload, in the launch configuration bench.py times:
provip_similarity_reduce on the whole batch, with its own critical-text mask,
relevance, top-N1 and merge. Per sample the oracle runs the same chain from the
same inputs (r and T, p, the keep set, the nearest-centroid assignment and the
merged rows) and every stage is compared; where a GPU decision lies inside the
oracle's tie band (T, or the keep set) the two chains part, and the rest of that
sample is checked for validity against its own decisions. The merge is checked
exactly on the LLaVA-1.5 workloads (the oracle assigns every row) and, at the
anyres and video sizes, on 16 sampled centroids per sample whose GPU members
and 48 random pruned rows the oracle reassigns against every kept row.
"""
import concurrent.futures as cf
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2608_25332_gb300 import synth
from paper_2608_25332_gb300 import provip as P
from parity import assert_close_rel, check_mask_band, check_merge, check_topk_band, rtol_for

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
EXACT_MERGE_MAX_NV = 1000  # above it the oracle's merge takes minutes per sample: sampled
POOL = min(16, os.cpu_count() or 4)


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


def _pmap(fn, items):
    # the oracle releases the GIL inside its C calls
    with cf.ThreadPoolExecutor(POOL) as ex:
        return list(ex.map(fn, items))


def _oracle_front(w, cpu, b):
    """crit text, relevance and top-N1 of sample b (Sec. 4.2-4.3)"""
    n = int(cpu["text_len"][b])
    Et, Ev = f64(cpu["emb_t"][b, :n]), f64(cpu["emb_v"][b])
    r, T = oracle.crit_text(Et)
    p = oracle.relevance(Et, T, Ev)
    return dict(r=r, T=T, p=p, keep=oracle.topk(p, w.keep_pre))


def _sampled_rows(w, keep, a_gpu, seed):
    """16 centroids and their GPU members, plus 48 random pruned rows"""
    rng = np.random.default_rng(seed)
    pruned = np.setdiff1d(np.arange(w.N_v), keep)
    cents = np.sort(rng.choice(w.keep_pre, 16, replace=False))
    mem = np.flatnonzero(np.isin(a_gpu, cents))
    rows = np.union1d(np.setdiff1d(mem, keep), rng.choice(pruned, min(48, len(pruned)), replace=False))
    return cents, rows


def _oracle_assign_rows(Ev, keep, rows):
    """the oracle's centroid of each row in `rows`, against every kept row"""
    sub = np.union1d(rows, keep)
    a_sub, _ = oracle.merge(Ev[sub], np.searchsorted(sub, keep))
    a_ref = np.full(Ev.shape[0], -1)
    a_ref[sub] = a_sub
    return a_ref


def _numpy_assign_rows(Ev, keep, rows):
    """validity of a chain that parted from the oracle's: the best kept row by
    cosine (fp64 numpy), against the GPU's own keep set"""
    U = Ev[rows] / np.maximum(np.linalg.norm(Ev[rows], axis=1, keepdims=True), 1e-300)
    K = Ev[keep] / np.maximum(np.linalg.norm(Ev[keep], axis=1, keepdims=True), 1e-300)
    a_ref = np.full(Ev.shape[0], -1)
    a_ref[rows] = np.argmax(U @ K.T, axis=1)
    return a_ref


@pytest.mark.parametrize("name", [w.name for w in synth.WORKLOADS])
def test_similarity_pass_matches_oracle(name):
    w, cpu, g = inputs(name)
    rt = rtol_for(w.dtype)
    mask, r = P.provip_crit_text(g["emb_t"], g["text_len"], want_r=True)
    res = P.provip_similarity_reduce(g["emb_v"], g["emb_t"], g["text_len"], w.keep_pre, want_merged=True,
                                     want_assign=True)
    torch.cuda.synchronize()
    assert torch.equal(mask, res["mask"])
    ref = _pmap(lambda b: _oracle_front(w, cpu, b), range(w.B))
    # relevance given the oracle's T, the whole batch in one call (a direct check of the p kernel)
    T_ref = np.zeros((w.B, w.n_t[1]), np.uint8)
    for b in range(w.B):
        T_ref[b, :len(ref[b]["T"])] = ref[b]["T"]
    p_given = P.provip_relevance(g["emb_v"], g["emb_t"], g["text_len"], torch.from_numpy(T_ref).to(DEV))
    mask_h, r_h, p_h, idx_h = (mask.cpu().numpy(), r.cpu().numpy(), res["p"].cpu().numpy(),
                               res["idx"].cpu().numpy())
    a_h = res["assign"].cpu().numpy()
    mg_h = res["merged"].float().cpu().numpy().astype(np.float64)
    to_merge, parted = [], []
    for b in range(w.B):
        n = int(cpu["text_len"][b])
        o = ref[b]
        what = f"{name}[{b}]"
        assert_close_rel(r_h[b, :n], o["r"], rt, f"{what} r")
        check_mask_band(mask_h[b, :n], o["r"], rt, f"{what} T")
        assert not mask_h[b, n:].any(), f"{what}: T mask set on padding"
        assert_close_rel(p_given[b].cpu().numpy(), o["p"], 0.0, f"{what} p|T_ref", atol=rt)
        if not np.array_equal(mask_h[b, :n].astype(bool), o["T"].astype(bool)):
            parted.append(b)  # T inside the band: the chains part here
            continue
        assert_close_rel(p_h[b], o["p"], 0.0, f"{what} p", atol=rt)
        check_topk_band(idx_h[b], o["p"], w.keep_pre, rt, f"{what} N1 keep")
        if np.array_equal(idx_h[b], o["keep"]):
            to_merge.append(b)
        else:
            parted.append(b)
    assert len(to_merge) >= max(1, (3 * w.B) // 4), \
        f"{name}: only {len(to_merge)} of {w.B} samples reach the oracle's merge"

    exact = w.N_v <= EXACT_MERGE_MAX_NV

    def merge_check(b, with_oracle):
        Ev = f64(cpu["emb_v"][b])
        keep = idx_h[b]
        what = f"{name}[{b}] merge" + ("" if with_oracle else " (own keep set)")
        if exact and with_oracle:
            a_ref, mg_ref = oracle.merge(Ev, keep)
            check_merge(Ev, keep, a_h[b], mg_h[b], w.dtype, what, a_ref, np.setdiff1d(np.arange(w.N_v), keep),
                        mg_ref=mg_ref)
            return
        cents, rows = _sampled_rows(w, keep, a_h[b], 100 + b)
        a_ref = (_oracle_assign_rows if with_oracle else _numpy_assign_rows)(Ev, keep, rows)
        check_merge(Ev, keep, a_h[b], mg_h[b], w.dtype, what, a_ref, rows, centroids=cents)

    _pmap(lambda b: merge_check(b, True), to_merge)
    _pmap(lambda b: merge_check(b, False), parted)


# bf16 merges run their Gram on pairs of SMs by default; pairs=0 holds the
# single-SM form to the oracle as well
MERGE_CASES = [(w.name, 1) for w in synth.WORKLOADS] + \
    [(w.name, 0) for w in synth.WORKLOADS if w.dtype == "bf16"]


@pytest.mark.parametrize("name,pairs", MERGE_CASES)
def test_merge_matches_oracle(name, pairs):
    """provip_merge on the whole batch in one call, each sample with the
    oracle's own keep set (so every sample reaches the merge): the stand-alone
    merge path, with its own inverse norms."""
    w, cpu, g = inputs(name)
    fronts = _pmap(lambda b: _oracle_front(w, cpu, b), range(w.B))
    keeps = np.stack([f["keep"] for f in fronts])
    P.provip_set_option(P.OPT_MERGE_PAIRS, pairs)
    try:
        assign, merged = P.provip_merge(g["emb_v"], torch.from_numpy(keeps).to(DEV))
        torch.cuda.synchronize()
    finally:
        P.provip_set_option(P.OPT_MERGE_PAIRS, 1)
    a_h = assign.cpu().numpy()
    mg_h = merged.float().cpu().numpy().astype(np.float64)
    exact = w.N_v <= EXACT_MERGE_MAX_NV

    def one(b):
        Ev = f64(cpu["emb_v"][b])
        keep = keeps[b]
        what = f"{name}[{b}] merge"
        if exact:
            a_ref, mg_ref = oracle.merge(Ev, keep)
            check_merge(Ev, keep, a_h[b], mg_h[b], w.dtype, what, a_ref, np.setdiff1d(np.arange(w.N_v), keep),
                        mg_ref=mg_ref)
        else:
            cents, rows = _sampled_rows(w, keep, a_h[b], 200 + b)
            check_merge(Ev, keep, a_h[b], mg_h[b], w.dtype, what, _oracle_assign_rows(Ev, keep, rows), rows,
                        centroids=cents)

    _pmap(one, range(w.B))
