"""GPU parity on the degenerate and boundary cases of the method, against the
oracle: the smallest and largest keep sizes (one kept token, nothing pruned),
one text row (T falls back to every row), zero-norm and duplicated visual rows
(cosine 0 by reading, exact cosine ties), row counts that leave ragged tiles,
text padding that holds NaN (so any read of it shows), and both dtypes.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_25332_gb300 import provip as P
from parity import assert_close_rel, check_mask_band, check_merge, check_topk_band, rtol_for

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


def _pre_case(seed, B, N_v, D, tls, dtype, smooth_text=False):
    rng = np.random.default_rng(seed)
    Ntm = max(tls)
    Ev = rng.standard_normal((B, N_v, D)).astype(np.float32)
    Ev[:, 3] = 0.0               # zero norm: cosine 0 against everything
    Ev[:, 7] = Ev[:, 5]          # an exact duplicate: ties in every cosine
    Ev[:, 11] *= 40.0            # scale does not change a cosine
    Et = rng.standard_normal((B, Ntm, D)).astype(np.float32)
    if smooth_text:
        # text logits of standard deviation 1/16 (the scale of LLM token
        # embeddings): a smooth softmax, so r and T are well separated
        Et *= 0.25 / D ** 0.25
    for b, t in enumerate(tls):
        Et[b, t:] = np.nan       # padding past each sample's text rows
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    ev, et = torch.from_numpy(Ev).to(td), torch.from_numpy(Et).to(td)
    return ev, et, np.array(tls, np.int32)


@pytest.mark.parametrize("dtype,B,N_v,D,tls,keep_pre", [
    ("bf16", 3, 37, 64, (1, 5, 17), 1),      # one kept token: every row merges into it
    ("bf16", 3, 37, 64, (1, 5, 17), 36),     # one pruned token
    ("bf16", 2, 37, 64, (3, 8), 37),         # nothing pruned: merged rows are the rows
    ("bf16", 2, 300, 128, (128, 33), 100),   # 128 text rows (the tensor-core limit), tiles 128+128+44
    ("bf16", 2, 200, 136, (129, 2), 50),     # 129 text rows: the CUDA-core relevance
    ("bf16", 2, 150, 136, (40, 7), 60),      # D = 136: the last K slice of the tensor-core Grams is partial
    ("f32", 2, 37, 64, (1, 9), 10),
])
def test_similarity_reduce_edge_cases(dtype, B, N_v, D, tls, keep_pre):
    ev, et, tl = _pre_case(17, B, N_v, D, tls, dtype)
    _check_reduce(ev, et, tl, keep_pre, dtype, f"edge {dtype} B={B} N_v={N_v} D={D} tl={tls} keep={keep_pre}")


@pytest.mark.parametrize("seed", range(6))
def test_similarity_reduce_random_shapes(seed):
    """Seeded random pre-LLM shapes: batch, visual count, width, ragged text
    lengths (one row included), keep_pre, both dtypes."""
    rng = np.random.default_rng(3000 + seed)
    dtype = "f32" if seed % 3 == 2 else "bf16"
    B = int(rng.integers(1, 5))
    N_v = int(rng.integers(20, 600))
    D = 8 * int(rng.integers(4, 64))
    tls = tuple(int(x) for x in rng.integers(1, 129, B))
    keep_pre = int(rng.integers(1, N_v + 1))
    ev, et, tl = _pre_case(4000 + seed, B, N_v, D, tls, dtype, smooth_text=True)
    _check_reduce(ev, et, tl, keep_pre, dtype, f"seed {seed} {dtype} B={B} N_v={N_v} D={D} tl={tls} keep={keep_pre}")


@pytest.mark.parametrize("pairs", [1, 0])
@pytest.mark.parametrize("B,N_v,D,keep", [
    (6, 1000, 256, 237),   # two 512-row groups, the second ending inside its first half
    (2, 700, 136, 640),    # 60 pruned rows; ten 64-column ranges, a partial last K slice
    (5, 513, 128, 1),      # one kept row; 512 pruned rows fill one group exactly
    (3, 800, 64, 130),     # the second group's second half holds 32 rows
    (40, 800, 64, 500),    # 120 tiles: two per pair of SMs, the accumulators reused
    (1, 4500, 64, 4200),   # more kept rows than 16 ranges of 256: the single-SM form either way
])
def test_merge_ragged_groups(B, N_v, D, keep, pairs):
    """provip_merge (bf16) with random keep sets over ragged row groups and
    column ranges, every sample against the oracle's merge, with the Gram on
    pairs of SMs (pairs=1) and on single SMs (pairs=0)."""
    rng = np.random.default_rng(7000 + N_v + keep)
    ev, _, _ = _pre_case(7100 + N_v, B, N_v, D, (1,), "bf16")
    keeps = np.stack([np.sort(rng.choice(N_v, keep, replace=False)) for _ in range(B)]).astype(np.int32)
    P.provip_set_option(P.OPT_MERGE_PAIRS, pairs)
    try:
        assign, merged = P.provip_merge(ev.to(DEV), torch.from_numpy(keeps).to(DEV))
        torch.cuda.synchronize()
    finally:
        P.provip_set_option(P.OPT_MERGE_PAIRS, 1)
    Evn = ev.float().numpy().astype(np.float64)
    for b in range(B):
        a_ref, mg_ref = oracle.merge(Evn[b], keeps[b])
        check_merge(Evn[b], keeps[b], assign[b].cpu().numpy(), merged[b].float().cpu().numpy().astype(np.float64),
                    "bf16", f"merge B={B} N_v={N_v} D={D} keep={keep} pairs={pairs} [{b}]", a_ref,
                    np.setdiff1d(np.arange(N_v), keeps[b]), mg_ref=mg_ref)


def _check_reduce(ev, et, tl, keep_pre, dtype, what):
    B, N_v = ev.shape[0], ev.shape[1]
    rt = rtol_for(dtype)
    res = P.provip_similarity_reduce(ev.to(DEV), et.to(DEV), torch.from_numpy(tl).to(DEV), keep_pre,
                                     want_merged=True, want_assign=True)
    torch.cuda.synchronize()
    Evn = ev.float().numpy().astype(np.float64)
    Etn = et.float().numpy().astype(np.float64)
    full = 0
    for b in range(B):
        n = int(tl[b])
        r_ref, T = oracle.crit_text(Etn[b, :n])
        mask = res["mask"][b].cpu().numpy()
        check_mask_band(mask[:n], r_ref, rt, f"{what} T[{b}]")
        assert not mask[n:].any()
        if n == 1:
            assert mask[0] == 1, "a single text row is critical"
        if not np.array_equal(mask[:n].astype(bool), T.astype(bool)):
            continue
        p_ref = oracle.relevance(Etn[b, :n], T, Evn[b])
        assert_close_rel(res["p"][b].cpu().numpy(), p_ref, 0.0, f"{what} p[{b}]", atol=rt)
        idx = res["idx"][b].cpu().numpy()
        check_topk_band(idx, p_ref, keep_pre, rt, f"{what} keep[{b}]")
        if not np.array_equal(idx, oracle.topk(p_ref, keep_pre)):
            continue
        a_ref, mg_ref = oracle.merge(Evn[b], idx)
        mg = res["merged"][b].float().cpu().numpy().astype(np.float64)
        if keep_pre == N_v:
            # nothing merged: every output row is its input row, bit for bit
            assert torch.equal(res["merged"][b].cpu(), ev[b][torch.from_numpy(idx).long()])
        # every merged row is the oracle's within one output ulp, or - where a
        # pruned row moved between two kept rows of (nearly) equal cosine - the
        # mean over the GPU's own members
        check_merge(Evn[b], idx, res["assign"][b].cpu().numpy(), mg, dtype, f"{what} merged[{b}]", a_ref,
                    np.setdiff1d(np.arange(N_v), idx), mg_ref=mg_ref)
        full += 1
    assert full >= 1, f"{what}: no sample reached the merge comparison"


def _in_llm_case(seed, B, nsys, nv, tls, Hq=4, Hkv=2, D=256, P_=3):
    rng = np.random.default_rng(seed)
    Ntm = max(tls)
    Lm = nsys + nv + Ntm
    Q = rng.standard_normal((B, Lm, Hq, 128)).astype(np.float32)
    K = rng.standard_normal((B, Lm, Hkv, 128)).astype(np.float32)
    V = rng.standard_normal((B, Lm, Hkv, 128)).astype(np.float32)
    H = rng.standard_normal((B, Lm, D)).astype(np.float32)
    tl = np.array(tls, np.int32)
    sl = (nsys + nv + tl).astype(np.int32)
    for b in range(B):
        Q[b, sl[b]:] = np.nan
        K[b, sl[b]:] = np.nan
    pos = rng.integers(0, 1 << 20, (P_, B, Lm)).astype(np.int32)
    bf = lambda x: torch.from_numpy(x).to(torch.bfloat16)
    return dict(Q=bf(Q), K=bf(K), V=bf(V), H=bf(H), pos=torch.from_numpy(pos), tl=tl, sl=sl,
                ts=np.full(B, nsys + nv, np.int32), nsys=nsys, nv=nv, Ntm=Ntm)


@pytest.mark.parametrize("keep", [1, 37])
@pytest.mark.parametrize("algo", ["ALGO_AUTO", "ALGO_TCGEN05_STREAM", "ALGO_SIMT"])
def test_prune_single_keep_and_identity(keep, algo):
    """keep = 1 keeps the single best visual token; keep = N_v is the identity
    gather (every row in place, the sequence unchanged)."""
    c = _in_llm_case(23, B=3, nsys=5, nv=37, tls=(1, 9, 130))
    heads = [0, 3]
    g = {k: c[k].to(DEV) for k in ("Q", "K", "V", "H", "pos")}
    ts, tl, sl = (torch.from_numpy(x).to(DEV) for x in (c["ts"], c["tl"], c["sl"]))
    out = P.provip_prune(g["Q"], g["K"], g["V"], g["H"], g["pos"], heads, ts, tl, sl, c["nsys"], c["nv"], keep,
                         algo=getattr(P, algo), N_t_max=c["Ntm"])
    torch.cuda.synchronize()
    Qn, Kn = c["Q"].float().numpy(), c["K"].float().numpy()
    for b in range(3):
        slb = int(c["sl"][b])
        ref = oracle.head_scores(Qn[b, :slb], Kn[b, :slb], heads, np.arange(c["ts"][b], c["ts"][b] + c["tl"][b]),
                                 c["nsys"], c["nv"])
        assert_close_rel(out["scores"][b].cpu().numpy(), ref, 2e-3, f"scores[{b}]")
        idx = out["idx"][b].cpu().numpy()
        check_topk_band(idx, ref, keep, 2e-3, f"keep[{b}]")
        if keep == c["nv"]:
            assert idx.tolist() == list(range(c["nv"]))
        n = int(out["seq_len"][b])
        assert n == slb - c["nv"] + keep
        src = oracle.compact_map(slb, c["nsys"], c["nv"], idx)
        for key, src_t in (("hidden", c["H"]), ("K", c["K"]), ("V", c["V"])):
            got = out[key][b, :n].cpu().view(torch.int16).numpy()
            exp = oracle.gather_rows(src_t[b].view(torch.int16).numpy(), src)
            np.testing.assert_array_equal(got, exp)
        for p in range(c["pos"].shape[0]):
            np.testing.assert_array_equal(out["pos"][p, b, :n].cpu().numpy(), c["pos"][p, b].numpy()[src])


def _random_case(rng):
    B = int(rng.integers(1, 5))
    Hkv = int(rng.choice([1, 2, 4]))
    Hq = Hkv * int(rng.choice([1, 2, 4]))
    H_sel = int(rng.integers(1, Hq + 1))
    nsys = int(rng.integers(0, 40))
    nv = int(rng.integers(8, 700))
    tls = tuple(int(x) for x in rng.integers(0, 260, B))
    keep = int(rng.integers(1, nv + 1))
    heads = sorted(rng.choice(Hq, H_sel, replace=False).tolist())
    return B, Hkv, Hq, heads, nsys, nv, tls, keep


@pytest.mark.parametrize("seed", range(8))
def test_prune_random_shapes(seed):
    """Seeded random shapes (batch, GQA ratio, selected heads, prefix, visual
    count, ragged text lengths including zero rows, keep) for every tensor-core
    form and the automatic choice: scores, keep sets and compaction against the
    oracle."""
    rng = np.random.default_rng(1000 + seed)
    B, Hkv, Hq, heads, nsys, nv, tls, keep = _random_case(rng)
    c = _in_llm_case(2000 + seed, B=B, nsys=nsys, nv=nv, tls=tls, Hq=Hq, Hkv=Hkv, D=128 * int(rng.integers(1, 9)))
    Qn, Kn = c["Q"].float().numpy(), c["K"].float().numpy()
    g = {k: c[k].to(DEV) for k in ("Q", "K", "V", "H", "pos")}
    ts, tl, sl = (torch.from_numpy(x).to(DEV) for x in (c["ts"], c["tl"], c["sl"]))
    for algo in (P.ALGO_AUTO, P.ALGO_TCGEN05_STREAM, P.ALGO_TCGEN05_CLUSTER, P.ALGO_TCGEN05_TWOPASS):
        out = P.provip_prune(g["Q"], g["K"], g["V"], g["H"], g["pos"], heads, ts, tl, sl, nsys, nv, keep,
                             algo=algo, N_t_max=c["Ntm"])
        torch.cuda.synchronize()
        what = f"seed {seed} (B={B} Hq={Hq} Hkv={Hkv} heads={heads} nsys={nsys} nv={nv} tl={tls} keep={keep}) algo {algo}"
        for b in range(B):
            slb = int(c["sl"][b])
            if tls[b] == 0:
                ref = np.zeros(nv)  # no text rows: nothing to score
                assert np.all(out["scores"][b].cpu().numpy() == 0.0), what
            else:
                ref = oracle.head_scores(Qn[b, :slb], Kn[b, :slb], heads,
                                         np.arange(c["ts"][b], c["ts"][b] + c["tl"][b]), nsys, nv)
                assert_close_rel(out["scores"][b].cpu().numpy(), ref, 2e-3, what + f" scores[{b}]")
            idx = out["idx"][b].cpu().numpy()
            check_topk_band(idx, ref, keep, 2e-3, what + f" keep[{b}]")
            n = int(out["seq_len"][b])
            assert n == slb - nv + keep, what
            src = oracle.compact_map(slb, nsys, nv, idx)
            for key, src_t in (("hidden", c["H"]), ("K", c["K"]), ("V", c["V"])):
                np.testing.assert_array_equal(out[key][b, :n].cpu().view(torch.int16).numpy(),
                                              oracle.gather_rows(src_t[b].view(torch.int16).numpy(), src),
                                              err_msg=what + f" {key}[{b}]")
