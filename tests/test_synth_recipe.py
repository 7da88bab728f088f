"""The synthetic inputs have the structure the input recipe states (CPU).

The benchmark and the parity tests run on seeded synthetic inputs that stand in
for the paper's benchmarks. These checks hold the generator to its recipe, so a
change to it that removes the structure the method reacts to (near-duplicate
visual tokens, temporal redundancy, a pooled overview tile, text rows at
embedding scale with visual content, attention sinks) fails here.
"""
import math

import numpy as np
import torch

from paper_2608_25332_gb300 import synth

W = synth.BY_NAME


def _unit_rows(E):
    E = np.asarray(E, np.float64)
    return E / np.linalg.norm(E, axis=1, keepdims=True)


def test_workload_table():
    # (B, N_v, D, H_q, H_kv, text rows, H_sel, keep_pre, keep, dtype) of the five workloads
    table = {
        "llava15_7b_f32_b1": (1, 576, 4096, 32, 32, (64, 64), 4, 192, 64, "f32"),
        "llava15_7b_bf16_b16": (16, 576, 4096, 32, 32, (32, 128), 8, 288, 64, "bf16"),
        "llava15_13b_bf16_b32": (32, 576, 5120, 40, 40, (64, 64), 6, 192, 128, "bf16"),
        "llava_next_7b_bf16_b8": (8, 2880, 4096, 32, 32, (96, 96), 8, 960, 320, "bf16"),
        "video_gqa_bf16_b1": (1, 9216, 3584, 28, 4, (128, 128), 4, 2304, 1024, "bf16"),
    }
    assert sorted(table) == sorted(w.name for w in synth.WORKLOADS)
    for name, t in table.items():
        w = W[name]
        assert (w.B, w.N_v, w.D, w.H_q, w.H_kv, tuple(w.n_t), w.H_sel, w.keep_pre, w.keep, w.dtype) == t, name
        assert w.L_max == synth.N_SYS + w.keep_pre + w.n_t[1]


def test_inputs_are_seeded():
    w = W["llava15_7b_bf16_b16"]
    a, b = synth.pre_llm_inputs(w, batch=2), synth.pre_llm_inputs(w, batch=2)
    for k in a:
        torch.testing.assert_close(a[k], b[k], rtol=0, atol=0, equal_nan=True)
    c = synth.pre_llm_inputs(w, batch=2, seed=w.seed + 1)
    assert not torch.equal(torch.nan_to_num(a["emb_v"]), torch.nan_to_num(c["emb_v"]))


def test_planted_near_duplicates():
    w = W["llava15_7b_bf16_b16"]
    U = _unit_rows(synth.visual_embeddings(w, 0))
    C = U @ U.T
    np.fill_diagonal(C, -1.0)
    best = C.max(axis=1)
    dup = best > 0.95
    # 48 disjoint clusters of 3..8 rows: every member has a partner at cos ~0.97
    assert 48 * 3 <= dup.sum() <= 48 * 8
    # every other row is an independent Gaussian: no partner anywhere near
    assert best[~dup].max() < 0.2


def test_video_frames_are_temporally_redundant():
    w = W["video_gqa_bf16_b1"]
    E = synth.visual_embeddings(w, 0)
    per = 576
    for f in range(w.N_v // per - 1):
        a, b = _unit_rows(E[f * per:(f + 1) * per]), _unit_rows(E[(f + 1) * per:(f + 2) * per])
        cos = (a * b).sum(axis=1)
        assert abs(cos.mean() - 0.9) < 0.02, (f, cos.mean())


def test_anyres_seams_and_overview_tile():
    w = W["llava_next_7b_bf16_b8"]
    E = synth.visual_embeddings(w, 0)
    side = 24
    U = _unit_rows(E)

    def tok(tile, r, c):
        return tile * side * side + r * side + c

    # near-duplicates across the seams of adjacent sub-tiles (about half the seam rows)
    seam = [float(U[tok(0, r, side - 1)] @ U[tok(1, r, 0)]) for r in range(side)]
    assert sum(c > 0.95 for c in seam) >= 6
    # the fifth tile follows the 2x2 average pool of the 48 x 48 mosaic of sub-tiles
    mosaic = np.zeros((2 * side, 2 * side, w.D))
    for t in range(4):
        tr, tc = divmod(t, 2)
        mosaic[tr * side:(tr + 1) * side, tc * side:(tc + 1) * side] = \
            E[t * side * side:(t + 1) * side * side].reshape(side, side, w.D)
    pooled = mosaic.reshape(side, 2, side, 2, w.D).mean(axis=(1, 3)).reshape(side * side, w.D)
    cos = (_unit_rows(pooled) * U[4 * side * side:]).sum(axis=1)
    assert np.median(cos) > 0.9


def test_text_rows_at_embedding_scale_with_visual_content():
    w = W["llava15_7b_bf16_b16"]
    Ev = synth.visual_embeddings(w, 0)
    n_t = 80  # of at most 128 rows: the rest are padding
    Et = synth.text_embeddings(w, 0, Ev, n_t)
    assert Et.shape == (128, w.D) and np.isnan(Et[n_t:]).all() and not np.isnan(Et[:n_t]).any()
    norms = np.linalg.norm(Et[:n_t], axis=1)
    assert abs(np.median(norms) / (0.02 * math.sqrt(w.D)) - 1) < 0.1
    # a quarter of the rows carry a visual row's direction (cos ~0.7 with it)
    best = (_unit_rows(Et[:n_t]) @ _unit_rows(Ev).T).max(axis=1)
    assert (best > 0.5).sum() == n_t // 4


def test_in_llm_layout_sinks_and_padding():
    w = W["llava15_7b_bf16_b16"]
    g = synth.in_llm_inputs(w, batch=3)
    tl = g["text_len"].numpy()
    seq = g["seq_len"].numpy()
    assert g["vis_start"] == synth.N_SYS and g["N_v"] == w.keep_pre and g["keep"] == w.keep
    assert np.array_equal(seq, synth.N_SYS + w.keep_pre + tl)
    assert np.array_equal(g["text_start"].numpy(), np.full(3, synth.N_SYS + w.keep_pre))
    heads = g["head_list"].numpy()
    assert len(heads) == w.H_sel and np.all(np.diff(heads) > 0) and heads.min() >= 0 and heads.max() < w.H_q
    K = g["K"].float().numpy()
    typical = math.sqrt(synth.D_HEAD)
    for b in range(3):
        n = np.linalg.norm(K[b, :seq[b]], axis=-1)  # [L, H_kv]
        sinks = np.flatnonzero((n > 4 * typical).all(axis=1))
        # row 0 and one visual row, at eight times a typical key norm
        assert len(sinks) == 2 and sinks[0] == 0 and synth.N_SYS <= sinks[1] < synth.N_SYS + w.keep_pre
        assert abs(n[0].mean() / (8 * typical) - 1) < 0.01
        assert np.isnan(K[b, seq[b]:]).all() and not np.isnan(K[b, :seq[b]]).any()
        assert np.array_equal(g["pos"].numpy()[0, b, :seq[b]], np.arange(seq[b]))


def test_video_position_ids_are_mrope_grid_rows():
    w = W["video_gqa_bf16_b1"]
    assert w.P == 3
    g = synth.in_llm_inputs(w, with_kv=False)
    pos = g["pos"].numpy()[:, 0]
    vs, nv = g["vis_start"], g["N_v"]
    t, h, ww = pos[0, vs:vs + nv] - vs, pos[1, vs:vs + nv] - vs, pos[2, vs:vs + nv] - vs
    assert t.min() >= 0 and t.max() < 16 and h.max() < 24 and ww.max() < 24
    flat = t * 576 + h * 24 + ww  # a sorted subset of the 16 x 24 x 24 grid
    assert np.all(np.diff(flat) > 0)
