"""The comparison rules of the GPU parity tests reject wrong outputs.

The GPU tests are only as strong as tests/parity.py: these CPU cases hand the
rules outputs with a planted error (a value past the tolerance, a clear winner
dropped from a keep set, an unsorted or out-of-range index, a T mask that
disagrees outside the tie band) and check that each is rejected, while correct
outputs and either choice inside a tie band are accepted.
"""
import numpy as np
import pytest

from parity import assert_close_rel, check_mask_band, check_topk_band, rtol_for


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
