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
