"""The comparison rules of the GPU parity tests reject wrong outputs.

The GPU tests are only as strong as tests/parity.py: these CPU cases hand the
rules outputs with a planted error (a value past the tolerance, a clear winner
dropped from a keep set, an unsorted or out-of-range index, a T mask that
disagrees outside the tie band, a merged row off by more than an ulp, a row
merged into a clearly worse centroid) and check that each is rejected, while
correct outputs and either choice inside a tie band are accepted.
"""
import numpy as np
import pytest

from parity import assert_close_rel, check_mask_band, check_merge, check_topk_band, out_ulp, rtol_for


def test_tolerances():
    assert rtol_for("bf16") == 2e-3 and rtol_for("f32") == 1e-5
    assert rtol_for("torch.float32") == 1e-5 and rtol_for("torch.bfloat16") == 2e-3


def test_close_rel_accepts_within_and_rejects_past_the_tolerance():
    ref = np.array([1.0, -2.0, 1e-3, 5.0])
    assert_close_rel(ref * (1 + 0.9e-3), ref, 1e-3, "inside")
    with pytest.raises(AssertionError, match="1 of 4"):
        bad = ref.copy()
        bad[2] *= 1 + 1.1e-3
        assert_close_rel(bad, ref, 1e-3, "one element")
    # an absolute floor admits small absolute errors on values near zero
    z = np.array([0.0, 1.0])
    assert_close_rel(z + np.array([5e-4, 0.0]), z, 1e-3, "floor", atol=1e-3)
    with pytest.raises(AssertionError):
        assert_close_rel(z + np.array([5e-4, 0.0]), z, 1e-3, "no floor")
    with pytest.raises(AssertionError):
        assert_close_rel(np.zeros(3), np.zeros(4), 1e-3, "shape")


def _scores(n, seed):
    s = np.random.default_rng(seed).permutation(n).astype(np.float64) + 1.0  # distinct, gaps of 1
    return s


def test_topk_exact_set_with_a_clear_margin():
    s = _scores(40, 1)
    k = 10
    ref = np.sort(np.argsort(-s)[:k])
    check_topk_band(ref, s, k, 1e-3, "exact")
    swapped = ref.copy()
    loser = int(np.argsort(-s)[k])  # the best of the rest, clearly below the k-th
    swapped[0] = loser
    with pytest.raises(AssertionError, match="clear margin"):
        check_topk_band(np.sort(swapped), s, k, 1e-3, "swap")


def test_topk_rejects_malformed_index_lists():
    s = _scores(20, 2)
    ref = np.sort(np.argsort(-s)[:5])
    with pytest.raises(AssertionError, match="ascending"):
        check_topk_band(ref[::-1], s, 5, 1e-3, "descending")
    with pytest.raises(AssertionError, match="ascending"):
        check_topk_band(np.r_[ref[:4], ref[3]], s, 5, 1e-3, "duplicate")
    with pytest.raises(AssertionError, match="range"):
        check_topk_band(np.r_[ref[:4], 20], s, 5, 1e-3, "out of range")
    with pytest.raises(AssertionError):
        check_topk_band(ref[:4], s, 5, 1e-3, "short")


def test_topk_tie_band_accepts_either_choice_but_not_clear_errors():
    # scores: five clear winners, three tied at the boundary (k = 6 takes one of them), clear losers
    s = np.array([9.0, 8.0, 7.0, 6.0, 5.0, 3.0, 3.0 * (1 + 1e-5), 3.0 * (1 - 1e-5), 1.0, 0.5])
    k = 6
    for tied in (5, 6, 7):
        check_topk_band(np.sort(np.r_[np.arange(5), tied]), s, k, 1e-3, f"tie {tied}")
    with pytest.raises(AssertionError, match="winners dropped"):
        check_topk_band(np.array([0, 1, 2, 3, 5, 6]), s, k, 1e-3, "winner dropped")
    with pytest.raises(AssertionError, match="losers kept"):
        check_topk_band(np.array([0, 1, 2, 3, 4, 8]), s, k, 1e-3, "loser kept")


def test_mask_band():
    r = np.array([0.30, 0.10, 0.25, 0.35])  # mean 0.25: row 2 sits on the mean
    good = np.array([1, 0, 0, 1])
    check_mask_band(good, r, 1e-3, "good")
    check_mask_band(np.array([1, 0, 1, 1]), r, 1e-3, "row on the mean either way")
    with pytest.raises(AssertionError):
        check_mask_band(np.array([1, 0, 0, 0]), r, 1e-3, "clear row missing")
    with pytest.raises(AssertionError):
        check_mask_band(np.array([1, 1, 0, 1]), r, 1e-3, "clear non-row included")
    # every r equal: the fallback (all rows) is valid
    flat = np.full(5, 0.2)
    check_mask_band(np.ones(5), flat, 1e-3, "fallback")


def _merge_case(seed=0, dtype="bf16"):
    """pruned rows 0..5 near kept rows 6..8; row 5 sits exactly between kept
    rows 7 and 8 (a cosine tie), so either centroid is valid for it"""
    rng = np.random.default_rng(seed)
    d = 16
    C = rng.standard_normal((3, d))
    C /= np.linalg.norm(C, axis=1, keepdims=True)
    Ev = np.zeros((9, d))
    Ev[6:9] = C * 3.0
    for j, c in enumerate([0, 0, 1, 1, 2]):
        Ev[j] = C[c] + 0.05 * rng.standard_normal(d)
    Ev[5] = C[1] + C[2]  # equidistant from kept rows 7 and 8
    keep = np.array([6, 7, 8])
    a_ref = np.array([0, 0, 1, 1, 2, 1, 0, 1, 2])  # the tie goes to the lower position
    mg = np.stack([Ev[a_ref == a].mean(axis=0) for a in range(3)])
    rnd = (lambda x: x.astype(np.float32).astype(np.float64)) if dtype == "f32" else \
        (lambda x: np.round(x * 2.0 ** 20) / 2.0 ** 20)  # well inside one bf16 ulp
    return Ev, keep, a_ref, mg, rnd


def test_merge_rule_accepts_the_oracle_and_a_tie_band_choice():
    Ev, keep, a_ref, mg, rnd = _merge_case()
    rows = np.arange(6)
    check_merge(Ev, keep, a_ref.copy(), rnd(mg), "bf16", "exact", a_ref, rows, mg_ref=mg)
    # row 5 moved to the other tied centroid: both merged rows become the means over the GPU members
    a = a_ref.copy()
    a[5] = 2
    mg2 = np.stack([Ev[a == k].mean(axis=0) for k in range(3)])
    check_merge(Ev, keep, a, rnd(mg2), "bf16", "tie move", a_ref, rows, mg_ref=mg)
    # the sampled form: only centroid 2 and its members are checked
    check_merge(Ev, keep, a, rnd(mg2), "bf16", "sampled", a_ref, np.array([4, 5]), centroids=[2])


def test_merge_rule_rejects_planted_errors():
    Ev, keep, a_ref, mg, rnd = _merge_case()
    rows = np.arange(6)
    # a merged value two ulps off with the oracle's member set
    bad = mg.copy()
    bad[1, 3] += 2 * out_ulp(mg[1, 3], "bf16")
    with pytest.raises(AssertionError, match="beyond one ulp"):
        check_merge(Ev, keep, a_ref.copy(), bad, "bf16", "value", a_ref, rows, mg_ref=mg)
    # a row merged into a clearly worse centroid (its value consistent with that choice)
    a = a_ref.copy()
    a[0] = 2
    mg2 = np.stack([Ev[a == k].mean(axis=0) for k in range(3)])
    with pytest.raises(AssertionError, match="clearly worse"):
        check_merge(Ev, keep, a, mg2, "bf16", "wrong centroid", a_ref, rows, mg_ref=mg)
    # a tie-band move whose merged row still holds the oracle's mean (inconsistent)
    a = a_ref.copy()
    a[5] = 2
    with pytest.raises(AssertionError, match="beyond one ulp"):
        check_merge(Ev, keep, a, mg, "bf16", "stale mean", a_ref, rows, mg_ref=mg)
    # a kept row that is not its own centroid
    a = a_ref.copy()
    a[6] = 1
    with pytest.raises(AssertionError, match="own centroid"):
        check_merge(Ev, keep, a, mg, "bf16", "kept row", a_ref, rows, mg_ref=mg)
    # the sampled form refuses a centroid with unchecked members
    with pytest.raises(AssertionError, match="not checked"):
        check_merge(Ev, keep, a_ref.copy(), mg, "bf16", "unchecked", a_ref, np.array([0]), centroids=[0])
    # fp32 tolerance: one fp32 ulp, not one bf16 ulp
    Ev, keep, a_ref, mg, rnd = _merge_case(dtype="f32")
    bad = rnd(mg)
    bad[2, 0] += 4 * out_ulp(mg[2, 0], "f32")
    with pytest.raises(AssertionError, match="beyond one ulp"):
        check_merge(Ev, keep, a_ref.copy(), bad, "f32", "fp32 value", a_ref, rows, mg_ref=mg)
