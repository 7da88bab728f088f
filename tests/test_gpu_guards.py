"""Guard bytes around every output and the workspace of each call.

compute-sanitizer is closed on this machine, so out-of-range writes are caught
the way a memory checker's red zones would: every output tensor and the
workspace live inside a larger buffer whose bytes before and after them hold a
fixed pattern; after the call the pattern must be intact. Output rows at or
past seq_len_out[b] are pre-filled with another pattern and must be left
untouched, as include/provip.h promises. The shapes are the edge and random
shapes of test_gpu_edges.py (ragged text lengths, text-free samples, GQA,
one kept token, nothing pruned), every head-score form, both dtypes.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_25332_gb300 import provip as P

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
GUARD = 4096      # bytes of red zone on each side (a multiple of the 256-byte workspace alignment)
RED = 0xA5        # red-zone byte
FILL = 0x5A       # pre-fill of the outputs' own bytes


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


class Guarded:
    """A tensor of the given shape and dtype inside a byte buffer with red zones."""

    def __init__(self, shape, dtype):
        n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        self.n = n
        self.buf = torch.full((GUARD + n + GUARD,), RED, dtype=torch.uint8, device=DEV)
        self.buf[GUARD:GUARD + n] = FILL
        self.t = self.buf[GUARD:GUARD + n].view(dtype).view(shape)

    def check(self, what):
        b = self.buf.cpu().numpy()
        lo, hi = b[:GUARD], b[GUARD + self.n:]
        bad = np.flatnonzero(lo != RED).tolist() + [GUARD + self.n + i for i in np.flatnonzero(hi != RED)]
        assert not bad, f"{what}: {len(bad)} red-zone bytes overwritten (first at buffer offset {bad[0]})"


def guarded_ws(nbytes):
    return Guarded((max(int(nbytes), 1),), torch.uint8)


def _rows_untouched(g, seq_len_out, what, row_axis=1):
    """rows >= seq_len_out[b] of an output [B, L_out, ...] (row_axis 1) or
    [P, B, L_out] (row_axis 2) still hold the pre-fill"""
    a = g.t.cpu().contiguous().view(torch.uint8).numpy()
    B = len(seq_len_out)
    for b in range(B):
        n = int(seq_len_out[b])
        tail = a[b, n:] if row_axis == 1 else a[:, b, n * 4:]
        assert np.all(tail == FILL), f"{what}: sample {b} rows >= seq_len_out = {n} were written"


def _in_llm_case(seed, B, nsys, nv, tls, Hq, Hkv, D, dtype):
    rng = np.random.default_rng(seed)
    Ntm = max(max(tls), 1)
    Lm = nsys + nv + Ntm
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    mk = lambda *s: torch.from_numpy(rng.standard_normal(s).astype(np.float32)).to(td)
    tl = np.array(tls, np.int32)
    sl = (nsys + nv + tl).astype(np.int32)
    c = dict(Q=mk(B, Lm, Hq, 128), K=mk(B, Lm, Hkv, 128), V=mk(B, Lm, Hkv, 128), H=mk(B, Lm, D),
             pos=torch.from_numpy(rng.integers(0, 1 << 20, (3, B, Lm)).astype(np.int32)), tl=tl, sl=sl,
             ts=np.full(B, nsys + nv, np.int32), nsys=nsys, nv=nv, Ntm=Ntm)
    for k in ("Q", "K", "V", "H"):
        for b in range(B):
            c[k][b, sl[b]:] = float("nan")  # padding rows: never read
    return c


def _guard_step(step, B, L_out, D, Hkv, has_scores, extra=()):
    """replace a step object's outputs and workspace by guarded ones"""
    dt = step.hidden_out.dtype
    gs = {"hidden_out": Guarded((B, L_out, D), dt), "K_out": Guarded((B, L_out, Hkv, 128), dt),
          "V_out": Guarded((B, L_out, Hkv, 128), dt), "pos_out": Guarded((3, B, L_out), torch.int32),
          "idx": Guarded(tuple(step.idx.shape), torch.int32), "seq_len_out": Guarded((B,), torch.int32),
          "ws": guarded_ws(step.ws.numel())}
    if has_scores:
        gs["scores"] = Guarded(tuple(step.scores.shape), torch.float32)
    for name in extra:
        gs[name] = Guarded(tuple(getattr(step, name).shape), getattr(step, name).dtype)
    for k, g in gs.items():
        setattr(step, k, g.t)
    return gs


SHAPES = [  # (seed, B, nsys, nv, text lengths, Hq, Hkv, D, keep)
    (1, 3, 5, 37, (1, 9, 130), 4, 2, 256, 1),         # one kept token; every row copied by the helper warps
    (2, 3, 5, 37, (1, 9, 130), 4, 2, 256, 37),        # nothing pruned
    (3, 2, 0, 300, (0, 64), 8, 2, 3072, 100),         # no prefix, a text-free sample; 6 KiB hidden rows (bulk)
    (4, 4, 35, 150, (17, 128, 40, 3), 16, 16, 5120, 60),  # 10 KiB hidden rows in two pieces, 4 KiB K/V rows
    (5, 1, 7, 700, (200,), 8, 1, 128, 333),           # two row blocks of text, one key/value head
]


@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("algo", ["ALGO_AUTO", "ALGO_TCGEN05_STREAM", "ALGO_TCGEN05_CLUSTER",
                                  "ALGO_TCGEN05_TWOPASS", "ALGO_SIMT", "SIMT_F32"])
def test_prune_writes_only_its_outputs(shape, algo):
    seed, B, nsys, nv, tls, Hq, Hkv, D, keep = shape
    dtype = "f32" if algo == "SIMT_F32" else "bf16"
    a = P.ALGO_SIMT if algo == "SIMT_F32" else getattr(P, algo)
    c = _in_llm_case(seed, B, nsys, nv, tls, Hq, Hkv, D, dtype)
    g = {k: c[k].to(DEV) for k in ("Q", "K", "V", "H", "pos")}
    ts, tl, sl = (torch.from_numpy(x).to(DEV) for x in (c["ts"], c["tl"], c["sl"]))
    heads = list(range(0, Hq, 2))
    step = P.PruneStep(g["Q"], g["K"], g["V"], g["H"], g["pos"], heads, c["Ntm"], nv, keep, algo=a,
                       want_scores=True)
    L_out = g["Q"].shape[1] - nv + keep
    gs = _guard_step(step, B, L_out, D, Hkv, True)
    out = step(g["Q"], g["K"], g["V"], g["H"], g["pos"], ts, tl, sl, nsys)
    torch.cuda.synchronize()
    what = f"prune {algo} shape {shape}"
    for k, gg in gs.items():
        gg.check(f"{what} {k}")
    slo = out["seq_len"].cpu().numpy()
    assert np.array_equal(slo, c["sl"] - nv + keep), what
    for k in ("hidden_out", "K_out", "V_out"):
        _rows_untouched(gs[k], slo, f"{what} {k}")
    _rows_untouched(gs["pos_out"], slo, f"{what} pos_out", row_axis=2)
    idx = out["idx"].cpu().numpy()
    assert np.all(np.diff(idx, axis=1) > 0) and idx.min() >= 0 and idx.max() < nv, what


@pytest.mark.parametrize("shape", SHAPES[2:])
@pytest.mark.parametrize("algo", ["ALGO_AUTO", "ALGO_TCGEN05_STREAM", "ALGO_TCGEN05_CLUSTER", "ALGO_SIMT"])
def test_visual_heads_prune_writes_only_its_outputs(shape, algo):
    seed, B, nsys, nv, tls, Hq, Hkv, D, keep = shape
    c = _in_llm_case(seed, B, nsys, nv, tls, Hq, Hkv, D, "bf16")
    g = {k: c[k].to(DEV) for k in ("Q", "K", "V", "H", "pos")}
    ts, tl, sl = (torch.from_numpy(x).to(DEV) for x in (c["ts"], c["tl"], c["sl"]))
    n_vis = min(3, Hq)
    step = P.VisualHeadsPruneStep(g["Q"], g["K"], g["V"], g["H"], g["pos"], c["Ntm"], nv, keep, n_vis,
                                  algo=getattr(P, algo))
    L_out = g["Q"].shape[1] - nv + keep
    gs = _guard_step(step, B, L_out, D, Hkv, True, extra=("vis_heads", "conf"))
    out = step(g["Q"], g["K"], g["V"], g["H"], g["pos"], ts, tl, sl, nsys)
    torch.cuda.synchronize()
    what = f"visual heads {algo} shape {shape}"
    for k, gg in gs.items():
        gg.check(f"{what} {k}")
    slo = out["seq_len"].cpu().numpy()
    for k in ("hidden_out", "K_out", "V_out"):
        _rows_untouched(gs[k], slo, f"{what} {k}")
    _rows_untouched(gs["pos_out"], slo, f"{what} pos_out", row_axis=2)


@pytest.mark.parametrize("algo", ["ALGO_AUTO", "ALGO_TCGEN05_STREAM", "ALGO_TCGEN05_CLUSTER",
                                  "ALGO_TCGEN05_TWOPASS", "ALGO_SIMT"])
def test_head_scores_writes_only_its_outputs(algo):
    seed, B, nsys, nv, tls, Hq, Hkv, D, keep = SHAPES[3]
    c = _in_llm_case(seed, B, nsys, nv, tls, Hq, Hkv, D, "bf16")
    Q, K = c["Q"].to(DEV), c["K"].to(DEV)
    ts, tl, sl = (torch.from_numpy(x).to(DEV) for x in (c["ts"], c["tl"], c["sl"]))
    L = P.lib()
    a = getattr(P, algo)
    Lm = Q.shape[1]
    heads = (ctypes.c_int * 2)(0, 3)
    ws = guarded_ws(L.provip_head_scores_workspace_size(B, Lm, 2, c["Ntm"], nv, a, P.BF16))
    sc = Guarded((B, nv), torch.float32)
    rc = L.provip_head_scores(P._ptr(Q), P._ptr(K), B, Lm, Hq, Hkv, 128, heads, 2, P._i32(ts), P._i32(tl), None,
                              c["Ntm"], nsys, nv, P._i32(sl), P.BF16, a, P._ptr(sc.t), P._ptr(ws.t), ws.t.numel(),
                              P._stream(Q.device))
    assert rc == 0, P.lib().provip_last_error()
    torch.cuda.synchronize()
    ws.check(f"head_scores {algo} workspace")
    sc.check(f"head_scores {algo} scores")
    assert torch.isfinite(sc.t).all()


@pytest.mark.parametrize("dtype,B,N_v,D,tls,keep_pre", [
    ("bf16", 3, 37, 64, (1, 5, 17), 1),
    ("bf16", 2, 37, 64, (3, 8), 37),
    ("bf16", 2, 300, 128, (128, 33), 100),
    ("bf16", 2, 200, 136, (129, 2), 50),
    ("bf16", 2, 150, 136, (40, 7), 60),
    ("f32", 2, 37, 64, (1, 9), 10),
])
def test_similarity_reduce_writes_only_its_outputs(dtype, B, N_v, D, tls, keep_pre):
    rng = np.random.default_rng(77)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    Ntm = max(tls)
    ev = torch.from_numpy(rng.standard_normal((B, N_v, D)).astype(np.float32)).to(td).to(DEV)
    et_np = (rng.standard_normal((B, Ntm, D)) * 0.25 / D ** 0.25).astype(np.float32)
    for b, t in enumerate(tls):
        et_np[b, t:] = np.nan
    et = torch.from_numpy(et_np).to(td).to(DEV)
    tl = torch.tensor(tls, dtype=torch.int32, device=DEV)
    gs = {"idx": Guarded((B, keep_pre), torch.int32), "merged": Guarded((B, keep_pre, D), td),
          "p": Guarded((B, N_v), torch.float32), "mask": Guarded((B, Ntm), torch.uint8),
          "assign": Guarded((B, N_v), torch.int32),
          "ws": guarded_ws(P.lib().provip_similarity_reduce_workspace_size(B, N_v, D, Ntm, keep_pre))}
    P.provip_similarity_reduce(ev, et, tl, keep_pre, ws=gs["ws"].t,
                               out={k: gs[k].t for k in ("idx", "merged", "p", "mask", "assign")})
    torch.cuda.synchronize()
    what = f"similarity_reduce {dtype} B={B} N_v={N_v} D={D} tl={tls} keep={keep_pre}"
    for k, g in gs.items():
        g.check(f"{what} {k}")
    m = gs["mask"].t.cpu().numpy()
    for b, t in enumerate(tls):
        assert not m[b, t:].any(), f"{what}: mask written past the text rows"


def test_topk_and_compact_write_only_their_outputs():
    B, N, k = 5, 3000, 700
    scores = torch.rand(B, N, device=DEV)
    idx = Guarded((B, k), torch.int32)
    rc = P.lib().provip_topk(P._ptr(scores), B, N, k, P._ptr(idx.t), P._stream(scores.device))
    assert rc == 0
    torch.cuda.synchronize()
    idx.check("topk idx")
    ref = torch.sort(torch.topk(scores, k, dim=1).indices, dim=1).values.to(torch.int32)
    assert torch.equal(idx.t, ref)
    # compaction of video-shaped rows: 8 KiB hidden rows (bulk copies), 1 KiB K/V rows (helper warps)
    c = _in_llm_case(9, 2, 35, 400, (128, 77), 8, 4, 4096, "bf16")
    g = {kk: c[kk].to(DEV) for kk in ("K", "V", "H", "pos")}
    sl = torch.from_numpy(c["sl"]).to(DEV)
    keep = 150
    kidx = torch.sort(torch.randperm(400, device=DEV)[:keep]).values.to(torch.int32)
    kidx = torch.stack([kidx, kidx])
    L_out = g["H"].shape[1] - 400 + keep
    outs = (Guarded((2, L_out, 4096), torch.bfloat16), Guarded((2, L_out, 4, 128), torch.bfloat16),
            Guarded((2, L_out, 4, 128), torch.bfloat16), Guarded((3, 2, L_out), torch.int32))
    r = P.provip_compact(kidx, g["H"], g["K"], g["V"], g["pos"], sl, 35, 400, out=tuple(o.t for o in outs))
    torch.cuda.synchronize()
    for name, o in zip(("hidden", "K", "V", "pos"), outs):
        o.check(f"compact {name}")
    slo = r["seq_len"].cpu().numpy()
    for name, o in zip(("hidden", "K", "V"), outs[:3]):
        _rows_untouched(o, slo, f"compact {name}")
    _rows_untouched(outs[3], slo, "compact pos", row_axis=2)
