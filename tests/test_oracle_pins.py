"""Pins for the fp64 oracle against facts fixed by the paper and by mathematics.

None of these tests retypes the oracle's own code: each compares it with a
closed form derived by hand, an invariant of the paper's equations, a textbook
library routine, or the independent pure-Python brute force (``oracle.brute``)
on inputs small enough to enumerate. Each pin names the mistake it would catch.
"""
import math

import numpy as np
import pytest
from scipy.special import softmax

import oracle
from oracle import brute

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def rng(seed):
    return np.random.default_rng(seed)


# --------------------------------------------------------------------------
# Sec. 4.2: critical text tokens
# --------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(6))
def test_crit_text_matches_brute_force(seed):
    g = rng(seed)
    n, d = int(g.integers(1, 9)), int(g.integers(1, 7))
    E = g.normal(size=(n, d)) * g.uniform(0.1, 1.5)
    r, m = oracle.crit_text(E)
    rb, Tb = brute.crit_text(E.tolist())
    np.testing.assert_allclose(r, rb, rtol=1e-12, atol=1e-15)
    assert sorted(np.flatnonzero(m).tolist()) == Tb


@pytest.mark.parametrize("seed", range(4))
def test_crit_text_sums_and_mean(seed):
    # every softmax row sums to 1, so sum_j r_j = 1 and Mean(r) = 1/N_t
    g = rng(100 + seed)
    E = g.normal(size=(37, 19)) * 0.4
    r, m = oracle.crit_text(E)
    assert abs(r.sum() - 1.0) < 1e-12
    assert np.all((r > 1.0 / 37 + 1e-12) == (m == 1)) or m.all()


def test_crit_text_closed_form_orthogonal_rows():
    # E = diag(sqrt(a)): G = diag(a). Row-wise softmax gives R_ii = e^a_i / (e^a_i + n - 1)
    # and R_ij = 1 / (e^a_i + n - 1) for i != j, so
    # r_j = (1/n) [ e^a_j / (e^a_j + n - 1) + sum_{i != j} 1 / (e^a_i + n - 1) ].
    # A column-wise softmax (wrong axis) would give r_j = 1/n for every j.
    a = np.array([0.3, 1.7, 0.9, 2.5, 0.0])
    n = len(a)
    E = np.diag(np.sqrt(a))
    r, m = oracle.crit_text(E)
    den = np.exp(a) + n - 1
    expect = np.array([(math.exp(a[j]) / den[j] + sum(1.0 / den[i] for i in range(n) if i != j)) / n
                       for j in range(n)])
    np.testing.assert_allclose(r, expect, rtol=1e-13)
    assert np.flatnonzero(m).tolist() == np.flatnonzero(expect > 1.0 / n).tolist()


def test_crit_text_library_softmax():
    # the textbook form with scipy's softmax along the last axis, no 1/sqrt(d) scale
    g = rng(7)
    E = g.normal(size=(23, 41)) * 0.3
    r, _ = oracle.crit_text(E)
    np.testing.assert_allclose(r, softmax(E @ E.T, axis=1).mean(axis=0), rtol=1e-12)


def test_crit_text_degenerate_cases():
    # identical rows: r uniform, nothing exceeds the mean -> T falls back to all rows
    E = np.tile(np.array([[0.1, -0.2, 0.3]]), (6, 1))
    r, m = oracle.crit_text(E)
    np.testing.assert_allclose(r, 1.0 / 6, rtol=1e-12)
    assert m.all()
    # a single text token is critical
    r, m = oracle.crit_text(np.array([[1.0, 2.0]]))
    assert m.tolist() == [1] and abs(r[0] - 1.0) < 1e-15


# --------------------------------------------------------------------------
# Sec. 4.3: text-guided relevance
# --------------------------------------------------------------------------
def _mask(n, idx):
    m = np.zeros(n, np.uint8)
    m[list(idx)] = 1
    return m


@pytest.mark.parametrize("seed", range(6))
def test_relevance_matches_brute_force(seed):
    g = rng(200 + seed)
    nt, nv, d = int(g.integers(1, 7)), int(g.integers(1, 17)), int(g.integers(2, 7))
    Et, Ev = g.normal(size=(nt, d)), g.normal(size=(nv, d))
    T = sorted(g.choice(nt, size=int(g.integers(1, nt + 1)), replace=False).tolist())
    p = oracle.relevance(Et, _mask(nt, T), Ev)
    np.testing.assert_allclose(p, brute.relevance(Et.tolist(), T, Ev.tolist()), rtol=1e-12, atol=1e-14)


def test_relevance_cosine_matrix_is_textbook():
    g = rng(9)
    Et, Ev = g.normal(size=(9, 33)), g.normal(size=(50, 33))
    T = [1, 4, 5, 8]
    p, M, mu = oracle.relevance(Et, _mask(9, T), Ev, want_M=True)
    nt = Et[T] / np.linalg.norm(Et[T], axis=1, keepdims=True)
    nvv = Ev / np.linalg.norm(Ev, axis=1, keepdims=True)
    np.testing.assert_allclose(M, nt @ nvv.T, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(mu, M.mean(axis=1), rtol=1e-12)
    np.testing.assert_allclose(p, (M - M.mean(axis=1, keepdims=True)).max(axis=0), rtol=1e-12)


def test_relevance_single_row_is_demeaned_row():
    # |T| = 1: p is the de-meaned row itself, so it sums to zero
    g = rng(10)
    Et, Ev = g.normal(size=(4, 8)), g.normal(size=(30, 8))
    p = oracle.relevance(Et, _mask(4, [2]), Ev)
    assert abs(p.sum()) < 1e-12


def test_relevance_scale_invariance_and_mask():
    # cosine ignores positive row scales; rows outside T do not matter
    g = rng(11)
    Et, Ev = g.normal(size=(6, 12)), g.normal(size=(40, 12))
    m = _mask(6, [0, 3, 4])
    p = oracle.relevance(Et, m, Ev)
    p2 = oracle.relevance(Et * g.uniform(0.1, 9, size=(6, 1)), m, Ev * g.uniform(0.1, 9, size=(40, 1)))
    np.testing.assert_allclose(p, p2, rtol=1e-12, atol=1e-14)
    Et3 = Et.copy()
    Et3[[1, 2, 5]] = g.normal(size=(3, 12)) * 50
    np.testing.assert_allclose(oracle.relevance(Et3, m, Ev), p, rtol=1e-13, atol=1e-15)


def test_relevance_zero_norm_visual_row():
    g = rng(12)
    Et, Ev = g.normal(size=(3, 5)), g.normal(size=(7, 5))
    Ev[4] = 0.0
    _, M, _ = oracle.relevance(Et, _mask(3, [0, 1, 2]), Ev, want_M=True)
    assert np.all(M[:, 4] == 0.0)


# --------------------------------------------------------------------------
# Top-k (Sec. 4.3 top N1, Sec. 4.4 top N2)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(5))
def test_topk_matches_lexsort(seed):
    g = rng(300 + seed)
    n = int(g.integers(1, 400))
    s = g.integers(0, 7, size=n).astype(np.float64) * 0.25  # many ties
    k = int(g.integers(1, n + 1))
    idx = oracle.topk(s, k)
    order = np.lexsort((np.arange(n), -s))  # primary -s, secondary index
    assert idx.tolist() == sorted(order[:k].tolist())
    assert idx.tolist() == brute.topk(s.tolist(), k)


def test_topk_ties_go_to_lowest_index():
    assert oracle.topk([1.0, 1.0, 1.0, 1.0], 2).tolist() == [0, 1]
    assert oracle.topk([0.5, 0.9, 0.9, 0.1], 1).tolist() == [1]
    assert oracle.topk([0.5, 0.9, 0.9, 0.1], 3).tolist() == [0, 1, 2]
    assert oracle.topk([3.0, 1.0, 2.0], 3).tolist() == [0, 1, 2]


# --------------------------------------------------------------------------
# Sec. 4.3 merge (reading: cosine-nearest kept token, uniform mean)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(6))
def test_merge_matches_brute_force(seed):
    g = rng(400 + seed)
    nv, d = int(g.integers(2, 17)), int(g.integers(2, 6))
    Ev = g.normal(size=(nv, d))
    keep = sorted(g.choice(nv, size=int(g.integers(1, nv + 1)), replace=False).tolist())
    a, mg = oracle.merge(Ev, keep)
    ab, mb = brute.merge(Ev.tolist(), keep)
    assert a.tolist() == ab
    np.testing.assert_allclose(mg, mb, rtol=1e-12, atol=1e-14)


def test_merge_invariants_and_closed_form():
    g = rng(13)
    d = 6
    C = g.normal(size=(3, d))
    # rows 0, 2, 5 are the kept centroids; every other row is a positive multiple of one
    Ev = np.stack([C[0], 2.0 * C[0], C[1], 0.5 * C[1], 3.0 * C[1], C[2], 7.0 * C[2]])
    keep = [0, 2, 5]
    a, mg = oracle.merge(Ev, keep)
    assert a.tolist() == [0, 0, 1, 1, 1, 2, 2]  # each kept row is its own centroid
    np.testing.assert_allclose(mg[0], (1 + 2) * C[0] / 2, rtol=1e-13)
    np.testing.assert_allclose(mg[1], (1 + 0.5 + 3) * C[1] / 3, rtol=1e-13)
    np.testing.assert_allclose(mg[2], (1 + 7) * C[2] / 2, rtol=1e-13)
    # ties go to the lower kept position: two identical centroids
    Ev2 = np.stack([C[0], C[0], C[0] * 4.0])
    a2, _ = oracle.merge(Ev2, [0, 1])
    assert a2.tolist() == [0, 1, 0]


def test_merge_scale_invariance_and_counts():
    g = rng(14)
    Ev = g.normal(size=(60, 9))
    keep = sorted(g.choice(60, size=17, replace=False).tolist())
    a, _ = oracle.merge(Ev, keep)
    a2, _ = oracle.merge(Ev * g.uniform(0.2, 5.0, size=(60, 1)), keep)
    assert a.tolist() == a2.tolist()
    assert np.bincount(a, minlength=17).sum() == 60
    assert all(a[k] == i for i, k in enumerate(keep))


# --------------------------------------------------------------------------
# Sec. 4.4: head-aware scores
# --------------------------------------------------------------------------
def _qk(g, L, Hq, Hkv, dh, scale=1.0):
    return g.normal(size=(L, Hq, dh)) * scale, g.normal(size=(L, Hkv, dh)) * scale


@pytest.mark.parametrize("seed", range(6))
def test_head_scores_matches_brute_force(seed):
    g = rng(500 + seed)
    Hkv = int(g.integers(1, 3))
    Hq = Hkv * int(g.integers(1, 4))
    dh = int(g.integers(2, 6))
    nsys, nv, nt = int(g.integers(0, 4)), int(g.integers(1, 17)), int(g.integers(1, 9))
    L = nsys + nv + nt
    Q, K = _qk(g, L, Hq, Hkv, dh, 1.3)
    heads = sorted(g.choice(Hq, size=int(g.integers(1, Hq + 1)), replace=False).tolist())
    rows = list(range(nsys + nv, L))
    v = oracle.head_scores(Q, K, heads, rows, nsys, nv)
    vb = brute.head_scores(Q.tolist(), K.tolist(), heads, rows, nsys, nv)
    np.testing.assert_allclose(v, vb, rtol=1e-12, atol=1e-15)


def test_head_scores_uniform_attention_closed_form():
    # Q = 0: every causal row is uniform, A_{t,k} = 1/(t+1), so
    # v_i = (1/|R|) sum_j 1/(t_j + 1) for every visual column (all precede the text rows).
    # Excluding the query's own key would give 1/t_j instead.
    g = rng(15)
    L, Hq, dh, vs, nv = 30, 4, 8, 3, 12
    Q = np.zeros((L, Hq, dh))
    K = g.normal(size=(L, Hq, dh))
    rows = list(range(vs + nv, L))
    v = oracle.head_scores(Q, K, [1, 3], rows, vs, nv)
    np.testing.assert_allclose(v, np.mean([1.0 / (t + 1) for t in rows]), rtol=1e-13)


def test_head_scores_probability_rows_sum_to_one():
    # with the "visual" range covering every key, each row's mass is 1, so sum_i v_i = 1
    g = rng(16)
    L, Hq, dh = 25, 2, 4
    Q, K = _qk(g, L, Hq, Hq, dh, 2.0)
    v = oracle.head_scores(Q, K, [0, 1], [5, 9, 24], 0, L)
    assert abs(v.sum() - 1.0) < 1e-13


def test_head_scores_scale_closed_form():
    # two keys, row t = 1: logits c/sqrt(dh) (key 0) and 0 (key 1 = 0 vector), so
    # A_{1,0} = 1 / (1 + exp(-c / sqrt(dh))). Dropping 1/sqrt(dh) would use c instead.
    dh, c = 16, 3.0
    Q = np.zeros((2, 1, dh))
    K = np.zeros((2, 1, dh))
    Q[1, 0, 0] = c
    K[0, 0, 0] = 1.0
    v = oracle.head_scores(Q, K, [0], [1], 0, 1)
    np.testing.assert_allclose(v[0], 1.0 / (1.0 + math.exp(-c / math.sqrt(dh))), rtol=1e-14)


def test_head_scores_ignores_unselected_heads():
    g = rng(17)
    L, Hq, dh = 40, 6, 8
    Q, K = _qk(g, L, Hq, Hq, dh)
    heads, rows = [1, 4], list(range(30, 40))
    v = oracle.head_scores(Q, K, heads, rows, 2, 20)
    Q2, K2 = Q.copy(), K.copy()
    for h in (0, 2, 3, 5):
        Q2[:, h] = g.normal(size=(L, dh)) * 10
        K2[:, h] = g.normal(size=(L, dh)) * 10
    np.testing.assert_allclose(oracle.head_scores(Q2, K2, heads, rows, 2, 20), v, rtol=1e-14)
    # permuting the selected list does not matter either
    np.testing.assert_allclose(oracle.head_scores(Q, K, [4, 1], rows, 2, 20), v, rtol=1e-13)


def test_head_scores_all_heads_is_fastv_mean():
    # All Attention Heads (Sec. 4.4, middle layer) equals the plain mean over heads of
    # scipy's causal softmax, sliced to the visual columns and averaged over text rows
    g = rng(18)
    L, Hq, dh, vs, nv = 36, 4, 8, 4, 20
    Q, K = _qk(g, L, Hq, Hq, dh)
    rows = list(range(vs + nv, L))
    v = oracle.head_scores(Q, K, list(range(Hq)), rows, vs, nv)
    logits = np.einsum("thd,khd->htk", Q, K) / math.sqrt(dh)
    logits = np.where(np.tril(np.ones((L, L), bool))[None], logits, -np.inf)
    A = softmax(logits, axis=-1)
    expect = A[:, rows][:, :, vs:vs + nv].mean(axis=(0, 1))
    np.testing.assert_allclose(v, expect, rtol=1e-12)


def test_head_scores_gqa_equals_repeated_kv():
    # grouped-query attention: head h reads kv head h // (Hq/Hkv); same as repeat_kv
    g = rng(19)
    L, Hq, Hkv, dh = 30, 6, 2, 8
    Q, K = _qk(g, L, Hq, Hkv, dh)
    rows = list(range(22, 30))
    heads = [1, 2, 4]
    v = oracle.head_scores(Q, K, heads, rows, 1, 15)
    Krep = np.repeat(K, Hq // Hkv, axis=1)
    np.testing.assert_allclose(oracle.head_scores(Q, Krep, heads, rows, 1, 15), v, rtol=1e-14)
    # the wrong mapping (h % Hkv: 1 -> 1, 4 -> 0 instead of 1 -> 0, 4 -> 1) differs
    Kwrong = np.tile(K, (1, Hq // Hkv, 1))
    assert not np.allclose(oracle.head_scores(Q, Kwrong, heads, rows, 1, 15), v)


def test_head_scores_sink_takes_the_mass():
    # a key aligned with every query and 8x a typical norm soaks up the softmax mass,
    # so the visual columns' scores drop (normalisation over the full causal range)
    g = rng(20)
    L, dh, vs, nv = 40, 16, 3, 25
    u = g.normal(size=dh)
    u /= np.linalg.norm(u)
    Q = g.normal(size=(L, 1, dh)) + 3.0 * u
    K = g.normal(size=(L, 1, dh))
    rows = list(range(vs + nv, L))
    v0 = oracle.head_scores(Q, K, [0], rows, vs, nv)
    K[0, 0] = 8 * math.sqrt(dh) * u
    v1 = oracle.head_scores(Q, K, [0], rows, vs, nv)
    assert v1.sum() < 0.05 * v0.sum()


# --------------------------------------------------------------------------
# Sec. 4.4: head confidence (next row: visual-head identification)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(3))
def test_head_confidence_matches_brute_force(seed):
    g = rng(600 + seed)
    L, Hq, Hkv, dh, vs, nv = 24, 4, 2, 4, 2, 14
    Q, K = _qk(g, L, Hq, Hkv, dh, 1.5)
    rows = [17, 19, 23]
    np.testing.assert_allclose(oracle.head_confidence(Q, K, rows, vs, nv),
                               brute.head_confidence(Q.tolist(), K.tolist(), rows, vs, nv),
                               rtol=1e-11, atol=1e-18)


def test_head_confidence_closed_forms():
    # uniform rows have zero variance
    g = rng(21)
    L, dh = 20, 4
    Q = np.zeros((L, 2, dh))
    K = g.normal(size=(L, 2, dh))
    np.testing.assert_allclose(oracle.head_confidence(Q, K, [15, 19], 2, 10), 0.0, atol=1e-30)
    # two visual columns with probabilities p, q: population variance ((p - q) / 2)^2
    dh, c = 4, 2.0
    Q = np.zeros((2, 1, dh))
    K = np.zeros((2, 1, dh))
    Q[1, 0, 0] = c
    K[0, 0, 0] = 1.0
    p = 1.0 / (1.0 + math.exp(-c / math.sqrt(dh)))
    np.testing.assert_allclose(oracle.head_confidence(Q, K, [1], 0, 2), [((2 * p - 1) / 2) ** 2], rtol=1e-13)


# --------------------------------------------------------------------------
# Compaction
# --------------------------------------------------------------------------
def test_compact_map_and_gather_are_fancy_indexing():
    g = rng(22)
    L, vs, nv = 60, 5, 30
    keep = np.sort(g.choice(nv, size=9, replace=False))
    src = oracle.compact_map(L, vs, nv, keep)
    np.testing.assert_array_equal(src, np.r_[np.arange(vs), vs + keep, np.arange(vs + nv, L)])
    X = g.normal(size=(L, 7, 3)).astype(np.float32)
    np.testing.assert_array_equal(oracle.gather_rows(X, src), X[src])
    assert np.all(np.diff(oracle.gather_rows(np.arange(L, dtype=np.int32), src)) > 0)
    # keep everything: identity
    np.testing.assert_array_equal(oracle.compact_map(L, vs, nv, np.arange(nv)), np.arange(L))


def test_prune_batch_is_the_composition():
    g = rng(23)
    B, Lm, Hq, dh, vs, nv, k = 3, 30, 4, 8, 3, 15, 5
    tl = np.array([12, 9, 7], np.int32)
    sl = vs + nv + tl
    Q, K = g.normal(size=(B, Lm, Hq, dh)), g.normal(size=(B, Lm, Hq, dh))
    Kraw = K.astype(np.float32)
    Vraw = g.normal(size=(B, Lm, Hq, dh)).astype(np.float32)
    hid = g.normal(size=(B, Lm, 10)).astype(np.float32)
    pos = np.broadcast_to(np.arange(Lm, dtype=np.int32), (1, B, Lm)).copy()
    out = oracle.prune_batch(Q, K, [0, 2], np.full(B, vs + nv), tl, sl, vs, nv, k, hid, Kraw, Vraw, pos)
    for b in range(B):
        rows = list(range(vs + nv, vs + nv + tl[b]))
        v = oracle.head_scores(Q[b, :sl[b]], K[b, :sl[b]], [0, 2], rows, vs, nv)
        np.testing.assert_allclose(out["v"][b], v, rtol=1e-14)
        idx = oracle.topk(v, k)
        np.testing.assert_array_equal(out["idx"][b], idx)
        src = oracle.compact_map(int(sl[b]), vs, nv, idx)
        n = len(src)
        assert out["seq_len"][b] == n
        np.testing.assert_array_equal(out["hidden"][b, :n], hid[b][src])
        np.testing.assert_array_equal(out["K"][b, :n], Kraw[b][src])
        np.testing.assert_array_equal(out["V"][b, :n], Vraw[b][src])
        np.testing.assert_array_equal(out["pos"][0, b, :n], src)
