"""Seeded synthetic inputs shaped like the paper's workloads.

This module is shared by the CUDA path's tests/benchmark and by the oracle's
tests. It holds none of the pruning method's arithmetic: it only draws random
tensors (numpy PCG64, then one round-to-nearest-even cast to the workload dtype
through torch) and lays them out.

Workloads (sizes follow the models the paper evaluates: LLaVA-1.5-7B/13B,
LLaVA-NeXT-7B anyres with 4 tiles plus a global overview tile of 576 tokens
each, and a Qwen2.5-VL-style GQA video of 16 frames):

  name                    dtype B   N_v  D     Hq/Hkv N_t      Hsel keep_pre keep
  llava15_7b_f32_b1       f32   1   576  4096  32/32  64       4    192      64
  llava15_7b_bf16_b16     bf16  16  576  4096  32/32  U[32,128] 8   288      64
  llava15_13b_bf16_b32    bf16  32  576  5120  40/40  64       6    192      128
  llava_next_7b_bf16_b8   bf16  8   2880 4096  32/32  96       8    960      320
  video_gqa_bf16_b1       bf16  1   9216 3584  28/4   128      4    2304     1024

Pre-LLM inputs (Sec. 4.2-4.3): visual embeddings E_v [B, N_v, D] ~ N(0, 1) with
planted near-duplicate clusters (member = centre + 0.25 * noise, rescaled to the
centre's norm: cosine ~0.97); the anyres workload plants duplicates across the
tile seams and makes the fifth tile a 2x2-average-pooled overview of the four
sub-tiles plus noise; the video workload makes frame f+1 = 0.9 * frame f +
sqrt(0.19) * noise (frame-to-frame cosine ~0.9). Text embeddings E_t
[B, N_t_max, D] ~ N(0, 0.02^2) (embedding-table scale, which keeps the unscaled
text self-similarity softmax smooth); a quarter of the text rows get a visual
cluster direction added at the same norm. Rows past a sample's text length are
NaN, so a kernel that reads them into a result fails loudly.

In-LLM inputs at the pruning layer (Sec. 4.4): the sequence of a sample is
[35 system rows | keep_pre visual rows | N_t text rows]; L_max = 35 + keep_pre +
max N_t. Q [B, L_max, Hq, 128] = N(0, 1) + u_g (u_g a unit direction per key/
value head g, so the queries of a group share a mean direction); K, V
[B, L_max, Hkv, 128] ~ N(0, 1); two sink keys per sample (row 0 and one seeded
visual row) are 8 * sqrt(128) * u_g, eight times a typical key norm and aligned
with the group's mean query direction; hidden [B, L_max, D] ~ N(0, 1); position
ids int32 [P, B, L_max]: P = 1 (0..L-1) for LLaVA, P = 3 (t, h, w) M-RoPE ids
for the video workload, whose visual rows are a seeded sorted subset of the
16 x 24 x 24 grid. Rows past seq_len are NaN (ids -1).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np
import torch

N_SYS = 35
VISUAL_FOCUS = 12.0  # query offset of a planted visual head (a typical query norm is ~11.3)
D_HEAD = 128
SEED_BASE = 20260000


@dataclass(frozen=True)
class Workload:
    name: str
    dtype: str  # "f32" | "bf16"
    B: int
    N_v: int
    D: int
    H_q: int
    H_kv: int
    n_t: tuple  # (min, max) text length, inclusive
    H_sel: int
    keep_pre: int
    keep: int
    layout: str = "image"  # "image" | "anyres" | "video"
    P: int = 1
    index: int = 0

    @property
    def seed(self) -> int:
        return SEED_BASE + self.index

    @property
    def L_max(self) -> int:
        return N_SYS + self.keep_pre + self.n_t[1]

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16


WORKLOADS = [
    Workload("llava15_7b_f32_b1", "f32", 1, 576, 4096, 32, 32, (64, 64), 4, 192, 64, index=0),
    Workload("llava15_7b_bf16_b16", "bf16", 16, 576, 4096, 32, 32, (32, 128), 8, 288, 64, index=1),
    Workload("llava15_13b_bf16_b32", "bf16", 32, 576, 5120, 40, 40, (64, 64), 6, 192, 128, index=2),
    Workload("llava_next_7b_bf16_b8", "bf16", 8, 2880, 4096, 32, 32, (96, 96), 8, 960, 320,
             layout="anyres", index=3),
    Workload("video_gqa_bf16_b1", "bf16", 1, 9216, 3584, 28, 4, (128, 128), 4, 2304, 1024,
             layout="video", P=3, index=4),
]
BY_NAME = {w.name: w for w in WORKLOADS}


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([seed, stream]))


def _cast(a: np.ndarray, dtype) -> torch.Tensor:
    """One round-to-nearest-even cast of an fp32 numpy array to the workload dtype."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dtype)


def _unit(rng, d):
    u = rng.standard_normal(d).astype(np.float32)
    return u / np.linalg.norm(u)


def _plant_duplicate(E, src, dst, rng, noise=0.25):
    """Row dst becomes a near-copy of row src at src's norm (cosine ~0.97)."""
    c = E[src]
    m = c + noise * rng.standard_normal(c.shape[0]).astype(np.float32)
    E[dst] = m * (np.linalg.norm(c) / max(np.linalg.norm(m), 1e-30))


def visual_embeddings(w: Workload, b: int, seed: int | None = None) -> np.ndarray:
    """E_v of sample b as fp32 [N_v, D] (before the dtype cast)."""
    seed = w.seed if seed is None else seed
    rng = _rng(seed, 1000 + b)
    N, D = w.N_v, w.D
    E = rng.standard_normal((N, D), dtype=np.float32)
    if w.layout == "video":
        per = 576
        frames = N // per
        for f in range(1, frames):
            E[f * per:(f + 1) * per] = (0.9 * E[(f - 1) * per:f * per]
                                        + math.sqrt(0.19) * E[f * per:(f + 1) * per])
        return E
    if w.layout == "anyres":
        # four 24x24 sub-tiles laid out 2x2 (rows 0..2303), then a 24x24 overview tile
        side = 24

        def tok(tile, r, c):
            return tile * side * side + r * side + c
        for r in range(side):  # duplicates across the vertical seams (tiles 0|1, 2|3)
            if rng.random() < 0.5:
                _plant_duplicate(E, tok(0, r, side - 1), tok(1, r, 0), rng)
            if rng.random() < 0.5:
                _plant_duplicate(E, tok(2, r, side - 1), tok(3, r, 0), rng)
        for c in range(side):  # and across the horizontal seams (tiles 0/2, 1/3)
            if rng.random() < 0.5:
                _plant_duplicate(E, tok(0, side - 1, c), tok(2, 0, c), rng)
            if rng.random() < 0.5:
                _plant_duplicate(E, tok(1, side - 1, c), tok(3, 0, c), rng)
        # overview tile: 2x2 average pool of the 48x48 mosaic, rescaled, plus noise
        mosaic = np.zeros((2 * side, 2 * side, D), np.float32)
        for t in range(4):
            tr, tc = divmod(t, 2)
            mosaic[tr * side:(tr + 1) * side, tc * side:(tc + 1) * side] = \
                E[t * side * side:(t + 1) * side * side].reshape(side, side, D)
        pooled = mosaic.reshape(side, 2, side, 2, D).mean(axis=(1, 3)).reshape(side * side, D)
        pooled *= 2.0  # the mean of 4 iid N(0,1) has std 1/2
        base = 4 * side * side
        E[base:base + side * side] = pooled + 0.3 * rng.standard_normal(pooled.shape, dtype=np.float32)
        n_clusters = 48
    else:
        n_clusters = 48
    perm = rng.permutation(N)
    o = 0
    for _ in range(n_clusters):
        size = int(rng.integers(3, 9))
        if o + size > N:
            break
        members = perm[o:o + size]
        o += size
        for m in members[1:]:
            _plant_duplicate(E, members[0], m, rng)
    return E


def text_lengths(w: Workload, seed: int | None = None) -> np.ndarray:
    seed = w.seed if seed is None else seed
    lo, hi = w.n_t
    if lo == hi:
        return np.full(w.B, lo, np.int32)
    return _rng(seed, 7).integers(lo, hi + 1, size=w.B).astype(np.int32)


def text_embeddings(w: Workload, b: int, E_v: np.ndarray, n_t: int,
                    seed: int | None = None) -> np.ndarray:
    """E_t of sample b as fp32 [N_t_max, D]; rows >= n_t are NaN."""
    seed = w.seed if seed is None else seed
    rng = _rng(seed, 2000 + b)
    Nm, D = w.n_t[1], w.D
    E = (0.02 * rng.standard_normal((Nm, D), dtype=np.float32))
    n_vis = max(1, n_t // 4)
    rows = rng.choice(n_t, size=n_vis, replace=False)
    for r in rows:
        j = int(rng.integers(0, E_v.shape[0]))
        dirn = E_v[j] / max(np.linalg.norm(E_v[j]), 1e-30)
        E[r] = E[r] + dirn * np.linalg.norm(E[r])
    E[n_t:] = np.nan
    return E


def pre_llm_inputs(w: Workload, device="cpu", seed: int | None = None, batch: int | None = None):
    """Inputs of the pre-LLM pass (Sec. 4.2-4.3) as torch tensors in the workload dtype."""
    B = w.B if batch is None else batch
    tl = text_lengths(w, seed)[:B] if batch is None or batch <= w.B else \
        np.resize(text_lengths(w, seed), B)
    Ev = np.empty((B, w.N_v, w.D), np.float32)
    Et = np.empty((B, w.n_t[1], w.D), np.float32)
    for b in range(B):
        Ev[b] = visual_embeddings(w, b, seed)
        Et[b] = text_embeddings(w, b, Ev[b], int(tl[b]), seed)
    return dict(
        emb_v=_cast(Ev, w.torch_dtype).to(device),
        emb_t=_cast(Et, w.torch_dtype).to(device),
        text_len=torch.from_numpy(tl.astype(np.int32)).to(device),
    )


def in_llm_inputs(w: Workload, device="cpu", seed: int | None = None, batch: int | None = None,
                  with_kv: bool = True, visual_heads: bool = False, focus: float = VISUAL_FOCUS):
    """Inputs of the in-LLM pruning step (Sec. 4.4) at the pruning layer.

    visual_heads: the heads of head_list become planted visual heads - on the
    text rows their queries get `focus` times the unit direction of the summed
    keys of 16 seeded visual rows of the sample (per key/value group), so their
    attention concentrates on those tokens (sharp focus on a few visual tokens,
    the behaviour the paper's head confidence detects). Drawn from a separate
    stream: every other value is the same as without it."""
    seed = w.seed if seed is None else seed
    B = w.B if batch is None else batch
    tl_all = text_lengths(w, seed)
    tl = np.resize(tl_all, B).astype(np.int32)
    Lm, Hq, Hkv, dh, nv = w.L_max, w.H_q, w.H_kv, D_HEAD, w.keep_pre
    group = Hq // Hkv
    rng = _rng(seed, 3000)
    heads = np.sort(rng.choice(Hq, size=w.H_sel, replace=False)).astype(np.int32)
    U = np.stack([_unit(rng, dh) for _ in range(Hkv)])  # [Hkv, dh]
    vis_start = N_SYS
    seq_len = (N_SYS + nv + tl).astype(np.int32)
    text_start = np.full(B, N_SYS + nv, np.int32)
    Q = np.empty((B, Lm, Hq, dh), np.float32)
    K = np.empty((B, Lm, Hkv, dh), np.float32)
    V = np.empty((B, Lm, Hkv, dh), np.float32) if with_kv else None
    H = np.empty((B, Lm, w.D), np.float32)
    pos = np.full((w.P, B, Lm), -1, np.int32)
    for b in range(B):
        r = _rng(seed, 4000 + b)
        Q[b] = r.standard_normal((Lm, Hq, dh), dtype=np.float32)
        Q[b] += np.repeat(U, group, axis=0)[None]
        K[b] = r.standard_normal((Lm, Hkv, dh), dtype=np.float32)
        sink_vis = vis_start + int(r.integers(0, nv))
        for s in (0, sink_vis):
            K[b, s] = 8.0 * math.sqrt(dh) * U
        if with_kv:
            V[b] = r.standard_normal((Lm, Hkv, dh), dtype=np.float32)
        H[b] = r.standard_normal((Lm, w.D), dtype=np.float32)
        L = int(seq_len[b])
        if w.P == 1:
            pos[0, b, :L] = np.arange(L, dtype=np.int32)
        else:
            grid = np.sort(r.choice(16 * 24 * 24, size=nv, replace=False))
            f, rem = np.divmod(grid, 576)
            hh, ww = np.divmod(rem, 24)
            for p in range(3):
                pos[p, b, :vis_start] = np.arange(vis_start)
            pos[0, b, vis_start:vis_start + nv] = vis_start + f
            pos[1, b, vis_start:vis_start + nv] = vis_start + hh
            pos[2, b, vis_start:vis_start + nv] = vis_start + ww
            t0 = vis_start + 24
            for p in range(3):
                pos[p, b, vis_start + nv:L] = t0 + np.arange(L - vis_start - nv)
        if visual_heads:
            rv = _rng(seed, 6000 + b)
            focus_rows = vis_start + rv.choice(nv, size=16, replace=False)
            t0, t1 = int(text_start[b]), int(text_start[b] + tl[b])
            for h in heads:
                g = h // group
                d = K[b, focus_rows, g].sum(axis=0)
                Q[b, t0:t1, h] += focus * d / np.linalg.norm(d)
        for arr in (Q, K, V, H):
            if arr is not None:
                arr[b, L:] = np.nan
    dt = w.torch_dtype
    out = dict(
        Q=_cast(Q, dt).to(device), K=_cast(K, dt).to(device),
        hidden=_cast(H, dt).to(device), pos=torch.from_numpy(pos).to(device),
        head_list=torch.from_numpy(heads).to(device),
        text_start=torch.from_numpy(text_start).to(device),
        text_len=torch.from_numpy(tl).to(device),
        seq_len=torch.from_numpy(seq_len).to(device),
        vis_start=vis_start, N_v=nv, keep=w.keep,
    )
    out["V"] = _cast(V, dt).to(device) if with_kv else None
    return out


def random_scores(B: int, N: int, seed: int, ties: bool = True) -> torch.Tensor:
    """fp32 scores [B, N] for top-k tests; with ties, about a third of the values are
    drawn from a small set so that equal keys straddle the k-th boundary."""
    rng = _rng(seed, 5000)
    s = rng.random((B, N), dtype=np.float32)
    if ties:
        pool = rng.random(5, dtype=np.float32)
        mask = rng.random((B, N)) < 0.33
        s[mask] = pool[rng.integers(0, 5, size=int(mask.sum()))]
    return torch.from_numpy(s)


def schedule_inputs(w: Workload, device="cpu", seed: int | None = None, batch: int | None = None):
    """Inputs of the progressive schedule (Sec. 4.1): the pre-LLM inputs, the
    shallow pruning layer's inputs (keep_pre visual rows, planted visual heads)
    and the middle layer's queries over the sequence the shallow layer leaves
    (L_max - keep_pre + keep rows: 35 system rows, keep visual rows, the text).
    The middle layer's keys, values, hidden states and position ids are the
    shallow layer's compacted outputs, so they are not drawn here. Middle-layer
    queries: N(0, 1) + u_g as at the shallow layer, NaN past the sequence."""
    seed = w.seed if seed is None else seed
    B = w.B if batch is None else batch
    pre = pre_llm_inputs(w, seed=seed, batch=B)
    shallow = in_llm_inputs(w, seed=seed, batch=B, visual_heads=True)
    rng = _rng(seed, 3000)
    rng.choice(w.H_q, size=w.H_sel, replace=False)  # same draws as in_llm_inputs
    U = np.stack([_unit(rng, D_HEAD) for _ in range(w.H_kv)])
    L2 = w.L_max - w.keep_pre + w.keep
    tl = shallow["text_len"].numpy()
    Q = np.empty((B, L2, w.H_q, D_HEAD), np.float32)
    for b in range(B):
        r = _rng(seed, 8000 + b)
        Q[b] = r.standard_normal((L2, w.H_q, D_HEAD), dtype=np.float32)
        Q[b] += np.repeat(U, w.H_q // w.H_kv, axis=0)[None]
        Q[b, N_SYS + w.keep + int(tl[b]):] = np.nan
    middle = dict(Q=_cast(Q, w.torch_dtype).to(device),
                  text_start=torch.full((B,), N_SYS + w.keep, dtype=torch.int32).to(device))
    return dict(pre={k: v.to(device) for k, v in pre.items()},
                shallow={k: (v.to(device) if isinstance(v, torch.Tensor) else v) for k, v in shallow.items()},
                middle=middle)


# The ablation of Sec. 5 (pruning before the LLM disabled) on LLaVA-1.5-7B:
# all 576 visual tokens reach the shallow pruning layer; visual tokens kept
# after the shallow and after the middle layer.
ABLATION_BUDGETS = ((219, 60), (146, 40), (73, 20), (54, 15), (36, 10), (18, 5))


def ablation_workload(n_shallow: int, base: str = "llava15_7b_bf16_b16") -> Workload:
    """The base workload with every visual token at the shallow layer (keep_pre =
    N_v) and n_shallow kept there; same seeds."""
    w = BY_NAME[base]
    return replace(w, name=f"{w.name}_ablation_{n_shallow}", keep_pre=w.N_v, keep=n_shallow)
