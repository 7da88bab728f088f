"""Comparison rules shared by the GPU parity tests.

Tolerances (written here, used everywhere):
  * floating outputs: relative 2e-3 for bf16 inputs with fp32 accumulation,
    1e-5 for the fp32 path (per element; v is a sum of positive terms, so the
    element-wise relative error is well conditioned);
  * cosine-valued outputs (p, mu) are compared absolutely with the same
    numbers, since |cos| <= 1;
  * integer decisions taken from floating point (top-k membership, the T mask,
    nearest-centroid assignment) must agree exactly wherever the oracle's
    margin exceeds the tolerance; inside that band either choice is valid and
    only validity is checked.
"""
import numpy as np

RTOL = {"f32": 1e-5, "bf16": 2e-3}


def rtol_for(dtype):
    return RTOL["f32" if str(dtype).endswith("float32") or dtype == "f32" else "bf16"]


def assert_close_rel(gpu, ref, rtol, what, atol=0.0):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    err = np.abs(gpu - ref)
    bad = err > rtol * np.abs(ref) + atol
    if bad.any():
        i = np.unravel_index(np.argmax(np.where(bad, err / (np.abs(ref) + 1e-300), 0)), ref.shape)
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} elements off; worst at {i}: "
                             f"gpu={gpu[i]!r} ref={ref[i]!r} rel={err[i] / (abs(ref[i]) + 1e-300):.3e}")


def check_topk_band(idx_gpu, scores_ref, k, rtol, what):
    """idx_gpu: ascending int indices from the GPU; scores_ref: oracle fp64 scores."""
    idx_gpu = np.asarray(idx_gpu)
    s = np.asarray(scores_ref, np.float64)
    n = s.shape[0]
    assert idx_gpu.shape == (k,), (what, idx_gpu.shape)
    assert np.all(np.diff(idx_gpu) > 0), f"{what}: indices not strictly ascending"
    assert idx_gpu.min() >= 0 and idx_gpu.max() < n, f"{what}: index out of range"
    order = np.lexsort((np.arange(n), -s))
    sk = s[order[k - 1]]
    sel = np.zeros(n, bool)
    sel[idx_gpu] = True
    band = rtol * abs(sk) + 1e-300
    if k < n:
        sk1 = s[order[k]]
        if sk - sk1 > band:
            ref = np.zeros(n, bool)
            ref[order[:k]] = True
            assert np.array_equal(sel, ref), f"{what}: keep set differs with a clear margin"
            return
    outside = np.abs(s - sk) > band
    must = outside & (s > sk)
    mustnot = outside & (s < sk)
    assert sel[must].all(), f"{what}: {(~sel[must]).sum()} clear winners dropped"
    assert not sel[mustnot].any(), f"{what}: {sel[mustnot].sum()} clear losers kept"


def check_mask_band(mask_gpu, r_ref, rtol, what):
    """T mask vs the oracle's r: rows clearly above/below mean(r) must agree."""
    r = np.asarray(r_ref, np.float64)
    m = np.asarray(mask_gpu).astype(bool)
    mean = r.mean()
    band = rtol * mean
    above = r > mean + band
    below = r < mean - band
    if above.any():
        assert m[above].all() and not m[below].any(), f"{what}: T mask differs outside the band"
    else:
        assert m.all() or not m[below].any(), f"{what}: degenerate T mask"


def merge_tol(dtype):
    """cosine tie band of the nearest-centroid choice: 1e-4 for bf16 inputs
    (fp32 accumulation of the Gram), 1e-6 for fp32 inputs"""
    return 1e-6 if dtype == "f32" else 1e-4


def out_ulp(x, dtype):
    """one unit in the last place of the output dtype at |x| (bf16: 8 bits of
    significand; fp32: numpy's spacing)"""
    x = np.abs(np.asarray(x, np.float64))
    if dtype == "f32":
        return np.spacing(x.astype(np.float32)).astype(np.float64)
    return 2.0 ** (np.floor(np.log2(np.maximum(x, 1e-30))) - 7)


def _unit_rows(X):
    n = np.linalg.norm(X, axis=1, keepdims=True)
    return np.where(n > 0, X / np.where(n > 0, n, 1.0), 0.0)


def check_merge(Ev, keep, a_gpu, mg_gpu, dtype, what, a_ref, rows, mg_ref=None, centroids=None):
    """Validity of a nearest-centroid merge (the Sec. 4.3 merge reading) against
    the oracle's decisions.

    Ev: the sample's visual rows (fp64, as given to the GPU); keep: ascending
    kept indices; a_gpu [N_v]: the GPU's centroid position of every row; mg_gpu
    [n1, d]: its merged rows (fp64 view of the output dtype). a_ref: the
    oracle's centroid positions, valid at least on `rows` (the pruned rows that
    are checked). mg_ref: the oracle's merged rows when it assigned every row
    (then every centroid is checked); otherwise `centroids` lists the centroids
    to check, and each of their GPU members must be in `rows`.

    Rules: kept rows are their own centroid; a checked row whose centroid
    differs from the oracle's must sit in the tie band (its cosine to the GPU's
    choice within merge_tol of its cosine to the oracle's, the best); a merged
    row whose member set equals the oracle's is within one output ulp of the
    oracle's mean; any other checked merged row is within one output ulp of the
    fp64 mean over the GPU's own members (a valid choice inside the band)."""
    n1 = len(keep)
    nv = Ev.shape[0]
    a_gpu = np.asarray(a_gpu)
    assert a_gpu.shape == (nv,), f"{what}: assignment shape {a_gpu.shape}"
    assert a_gpu.min() >= 0 and a_gpu.max() < n1, f"{what}: centroid position out of range"
    assert np.array_equal(a_gpu[keep], np.arange(n1)), f"{what}: a kept row is not its own centroid"
    rows = np.asarray(rows)
    moved = rows[a_gpu[rows] != a_ref[rows]]
    if moved.size:
        U = _unit_rows(Ev[moved])
        Kg = _unit_rows(Ev[keep[a_gpu[moved]]])
        Kr = _unit_rows(Ev[keep[a_ref[moved]]])
        c_gpu = np.sum(U * Kg, axis=1)
        c_ref = np.sum(U * Kr, axis=1)
        bad = c_gpu < c_ref - merge_tol(dtype)
        assert not bad.any(), (f"{what}: {bad.sum()} rows merged into a centroid clearly worse than the "
                               f"oracle's (rows {moved[bad][:8].tolist()})")
    if mg_ref is not None:
        check = np.arange(n1)
    else:
        check = np.asarray(centroids)
    members = {}
    order = np.argsort(a_gpu, kind="stable")
    bounds = np.searchsorted(a_gpu[order], np.arange(n1 + 1))
    for a in check:
        members[a] = order[bounds[a]:bounds[a + 1]]
    checked = set(rows.tolist()) | set(np.asarray(keep).tolist())
    for a in check:
        mem = members[a]
        if mg_ref is None:
            assert set(mem.tolist()) <= checked, f"{what}: centroid {a} has members that were not checked"
        same = mg_ref is not None and np.array_equal(mem, np.flatnonzero(a_ref == a))
        expect = mg_ref[a] if same else Ev[mem].mean(axis=0)
        err = np.abs(np.asarray(mg_gpu[a], np.float64) - expect)
        lim = out_ulp(expect, dtype) * 1.0001 + 1e-37
        assert np.all(err <= lim), (f"{what}: merged row {a} ({'oracle member set' if same else 'own members'}"
                                    f", {len(mem)} rows) beyond one ulp: worst "
                                    f"{np.max(err / lim):.2f} ulp at column {int(np.argmax(err / lim))}")
