"""Thin Python binding of the C ABI (include/provip.h), same names.

Argument marshalling only: torch tensors give device pointers, the current
torch stream gives the cudaStream_t, and torch allocates the workspace and the
outputs. Every step of the pruning path runs in the CUDA library; there is no
CPU or PyTorch fallback - if ``libprovip.so`` is missing or a call fails, a
``ProvipError`` is raised.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libprovip.so")

OK = 0
ERR_INVALID_ARG = -1
ERR_UNSUPPORTED = -2
ERR_WORKSPACE = -3
ERR_CUDA = -4
ERR_TIMEOUT = -5
DEVSTAT_TIMEOUT, DEVSTAT_BAD_ARG = 1, 2  # bits of the device status word
F32, BF16 = 0, 1
ALGO_AUTO, ALGO_SIMT, ALGO_TCGEN05, ALGO_TCGEN05_TWOPASS = 0, 1, 2, 3
ALGO_TCGEN05_STREAM, ALGO_TCGEN05_CLUSTER = 4, 5
PRUNE_OVERLAP_PREVIOUS = 1
PRUNE_CONCURRENT = 2
PRUNE_HOST_ROWS = 4

_P = ctypes.c_void_p
_I = ctypes.c_int
_Z = ctypes.c_size_t

# name -> (restype, argtypes); mirrors include/provip.h
_SIGS = {
    "provip_status_string": (ctypes.c_char_p, [_I]),
    "provip_last_error": (ctypes.c_char_p, []),
    "provip_version": (_I, []),
    "provip_set_option": (_I, [_I, _I]),
    "provip_device_status": (_I, [_P, _I]),
    "provip_selftest_wait_timeout": (_I, [_P]),
    "provip_crit_text_workspace_size": (_Z, [_I, _I, _I]),
    "provip_crit_text": (_I, [_P, _I, _I, _I, _P, _I, _P, _P, _P, _Z, _P]),
    "provip_relevance_workspace_size": (_Z, [_I, _I, _I, _I]),
    "provip_relevance": (_I, [_P, _I, _I, _I, _P, _P, _I, _P, _I, _P, _P, _Z, _P]),
    "provip_topk": (_I, [_P, _I, _I, _I, _P, _P]),
    "provip_merge_workspace_size": (_Z, [_I, _I, _I, _I]),
    "provip_merge": (_I, [_P, _I, _I, _I, _P, _I, _I, _P, _P, _P, _Z, _P]),
    "provip_similarity_reduce_workspace_size": (_Z, [_I, _I, _I, _I, _I]),
    "provip_similarity_reduce": (_I, [_P, _I, _I, _I, _P, _P, _I, _P, _I, _I, _P, _P, _P, _P, _P, _P, _Z,
                                      _P]),
    "provip_head_scores_workspace_size": (_Z, [_I, _I, _I, _I, _I, _I, _I]),
    "provip_head_scores": (_I, [_P, _P, _I, _I, _I, _I, _I, _P, _I, _P, _P, _P, _I, _I, _I, _P, _I, _I,
                                _P, _P, _Z, _P]),
    "provip_head_scores_noalloc": (_I, [_P, _P, _I, _I, _I, _I, _I, _P, _I, _P, _P, _P, _I, _I, _I, _P, _I,
                                        _I, _P, _P]),
    "provip_compact": (_I, [_P, _I, _I, _I, _P, _I, _P, _P, _I, _I, _P, _I, _P, _I, _I, _I, _P, _P, _P,
                            _P, _P, _P]),
    "provip_topk_compact": (_I, [_P, _I, _I, _I, _P, _I, _P, _P, _I, _I, _P, _I, _P, _I, _I, _I, _P, _P,
                                 _P, _P, _P, _P, _P]),
    "provip_head_topk": (_I, [_P, _P, _I, _I, _I, _I, _I, _P, _I, _P, _P, _P, _I, _I, _I, _P, _I, _I, _I,
                              _P, _P, _P, _Z, _P]),
    "provip_prune_workspace_size": (_Z, [_I, _I, _I, _I, _I, _I, _I]),
    "provip_prune": (_I, [_P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _I, _P, _P, _P, _I, _I, _I, _P, _P,
                          _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _Z, ctypes.c_uint, _P]),
    "provip_visual_heads_workspace_size": (_Z, [_I, _I, _I, _I, _I, _I, _I, _I]),
    "provip_head_confidence": (_I, [_P, _P, _I, _I, _I, _I, _I, _P, _P, _P, _I, _I, _I, _P, _I, _I, _I,
                                    _P, _P, _P, _Z, _P]),
    "provip_prune_visual_heads": (_I, [_P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P, _I, _I, _I, _P,
                                       _P, _I, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _Z,
                                       ctypes.c_uint, _P]),
}


class ProvipError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"{msg} (status {code})")
        self.code = code


_lib = None
_lock = threading.Lock()


def lib():
    """Loads libprovip.so (raises if it has not been built: there is no fallback)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise ProvipError(ERR_UNSUPPORTED, f"CUDA library not built: {LIB_PATH} is missing "
                                  "(run __graft_entry__.build())")
            L = ctypes.CDLL(LIB_PATH)
            for name, (res, args) in _SIGS.items():
                f = getattr(L, name)
                f.restype = res
                f.argtypes = args
            _lib = L
    return _lib


def _check(rc, what):
    if rc != OK:
        L = lib()
        msg = L.provip_last_error().decode() or L.provip_status_string(rc).decode()
        raise ProvipError(rc, f"{what}: {msg}")


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise ProvipError(ERR_UNSUPPORTED, f"unsupported dtype {t.dtype}")


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ProvipError(ERR_INVALID_ARG, "tensor must live on the GPU")
    if not t.is_contiguous():
        raise ProvipError(ERR_INVALID_ARG, "tensor must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _ptr_host_ok(t):
    """a device tensor, or a pinned host tensor (mapped into the device's
    address space) for the arguments PROVIP_PRUNE_HOST_ROWS allows there"""
    if t is not None and not t.is_cuda:
        if not t.is_pinned():
            raise ProvipError(ERR_INVALID_ARG, "a host tensor must be pinned (pin_memory())")
        if not t.is_contiguous():
            raise ProvipError(ERR_INVALID_ARG, "tensor must be contiguous")
        return ctypes.c_void_p(t.data_ptr())
    return _ptr(t)


def _stream(device):
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _i32(t):
    if t is None:
        return None
    if t.dtype != torch.int32:
        raise ProvipError(ERR_INVALID_ARG, "index/length tensors must be int32")
    return _ptr(t)


def _i32_host_ok(t):
    if t is None:
        return None
    if t.dtype != torch.int32:
        raise ProvipError(ERR_INVALID_ARG, "index/length tensors must be int32")
    return _ptr_host_ok(t)


def _u8(t):
    if t is None:
        return None
    if t.dtype != torch.uint8:
        raise ProvipError(ERR_INVALID_ARG, "masks must be uint8")
    return _ptr(t)


def workspace(nbytes: int, device) -> torch.Tensor:
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device)


# ---------------------------------------------------------------------------
# status
# ---------------------------------------------------------------------------
def provip_device_status(clear: bool = True):
    """Synchronises and returns (status code, device status bits)."""
    bits = ctypes.c_uint(0)
    rc = lib().provip_device_status(ctypes.byref(bits), 1 if clear else 0)
    return rc, bits.value


def provip_selftest_wait_timeout(device="cuda:0"):
    """Enqueues the failure-detection self test: a bounded wait that nothing
    completes gives up after 2 s and sets the TIMEOUT bit of the device status
    word (read it with provip_device_status)."""
    _check(lib().provip_selftest_wait_timeout(_stream(torch.device(device))), "provip_selftest_wait_timeout")


def provip_version() -> int:
    return lib().provip_version()


OPT_MERGE_PAIRS = 1


def provip_set_option(option: int, value: int) -> None:
    """Process-wide kernel-choice switch (PROVIP_OPT_*), for calls enqueued after it."""
    _check(lib().provip_set_option(int(option), int(value)), "provip_set_option")


# ---------------------------------------------------------------------------
# pre-LLM pass
# ---------------------------------------------------------------------------
def provip_crit_text(emb_t, text_len, want_r=False, out=None, ws=None):
    """Sec. 4.2: the critical-row mask T [B, N_t_max] (and r when want_r); out: a
    pre-allocated mask to write, ws: a pre-allocated workspace."""
    B, Ntm, D = emb_t.shape
    dev = emb_t.device
    mask = out if out is not None else torch.empty((B, Ntm), dtype=torch.uint8, device=dev)
    r = torch.empty((B, Ntm), dtype=torch.float32, device=dev) if want_r else None
    L = lib()
    need = L.provip_crit_text_workspace_size(B, Ntm, D)
    if ws is None or ws.numel() < need:
        ws = workspace(need, dev)
    rc = L.provip_crit_text(_ptr(emb_t), B, Ntm, D, _i32(text_len), _dtype_code(emb_t), _u8(mask),
                            _ptr(r), _ptr(ws), ws.numel(), _stream(dev))
    _check(rc, "provip_crit_text")
    return (mask, r) if want_r else mask


def provip_relevance(emb_v, emb_t, text_len, crit_mask):
    B, Nv, D = emb_v.shape
    Ntm = emb_t.shape[1]
    dev = emb_v.device
    p = torch.empty((B, Nv), dtype=torch.float32, device=dev)
    L = lib()
    ws = workspace(L.provip_relevance_workspace_size(B, Nv, D, Ntm), dev)
    rc = L.provip_relevance(_ptr(emb_v), B, Nv, D, _ptr(emb_t), _i32(text_len), Ntm, _u8(crit_mask),
                            _dtype_code(emb_v), _ptr(p), _ptr(ws), ws.numel(), _stream(dev))
    _check(rc, "provip_relevance")
    return p


def provip_topk(scores, k):
    B, N = scores.shape
    idx = torch.empty((B, k), dtype=torch.int32, device=scores.device)
    rc = lib().provip_topk(_ptr(scores), B, N, k, _ptr(idx), _stream(scores.device))
    _check(rc, "provip_topk")
    return idx


def provip_merge(emb_v, keep_idx, want_merged=True):
    B, Nv, D = emb_v.shape
    keep = keep_idx.shape[1]
    dev = emb_v.device
    assign = torch.empty((B, Nv), dtype=torch.int32, device=dev)
    merged = torch.empty((B, keep, D), dtype=emb_v.dtype, device=dev) if want_merged else None
    L = lib()
    ws = workspace(L.provip_merge_workspace_size(B, Nv, D, keep), dev)
    rc = L.provip_merge(_ptr(emb_v), B, Nv, D, _i32(keep_idx), keep, _dtype_code(emb_v), _ptr(assign),
                        _ptr(merged), _ptr(ws), ws.numel(), _stream(dev))
    _check(rc, "provip_merge")
    return assign, merged


def provip_similarity_reduce(emb_v, emb_t, text_len, keep_pre, crit_mask=None, want_merged=True,
                             ws=None, out=None, want_assign=False):
    """Sec. 4.2-4.3 end to end. Returns dict(idx, merged, p, mask, assign); out:
    the same dict of pre-allocated outputs to write instead (assign optional:
    the merge's nearest-centroid positions [B, N_v], with want_assign or given
    in out)."""
    B, Nv, D = emb_v.shape
    Ntm = emb_t.shape[1]
    dev = emb_v.device
    if out is not None:
        idx, merged, p, mask = out["idx"], out.get("merged"), out["p"], out["mask"]
        assign = out.get("assign")
    else:
        idx = torch.empty((B, keep_pre), dtype=torch.int32, device=dev)
        merged = torch.empty((B, keep_pre, D), dtype=emb_v.dtype, device=dev) if want_merged else None
        p = torch.empty((B, Nv), dtype=torch.float32, device=dev)
        mask = torch.empty((B, Ntm), dtype=torch.uint8, device=dev)
        assign = torch.empty((B, Nv), dtype=torch.int32, device=dev) if (want_assign and want_merged) else None
    L = lib()
    need = L.provip_similarity_reduce_workspace_size(B, Nv, D, Ntm, keep_pre)
    if ws is None or ws.numel() < need:
        ws = workspace(need, dev)
    rc = L.provip_similarity_reduce(_ptr(emb_v), B, Nv, D, _ptr(emb_t), _i32(text_len), Ntm,
                                    _u8(crit_mask), keep_pre, _dtype_code(emb_v), _ptr(idx),
                                    _ptr(merged), _i32(assign), _ptr(p), _ptr(mask), _ptr(ws),
                                    ws.numel(), _stream(dev))
    _check(rc, "provip_similarity_reduce")
    return dict(idx=idx, merged=merged, p=p, mask=mask, assign=assign)


# ---------------------------------------------------------------------------
# in-LLM pass
# ---------------------------------------------------------------------------
def _heads_arg(head_list, H_q):
    """head_list is read on the host (a list, a CPU tensor, or a device tensor copied once);
    None means every head (a NULL list with H_sel = H_q)."""
    if head_list is None:
        return None, int(H_q)
    hl = [int(h) for h in (head_list.tolist() if hasattr(head_list, "tolist") else head_list)]
    arr = (ctypes.c_int * len(hl))(*hl)
    return arr, len(hl)


def provip_head_scores(Q, K, head_list, text_start, text_len, seq_len, vis_start, N_v,
                       row_mask=None, algo=ALGO_AUTO, N_t_max=None, ws=None):
    B, Lm, Hq, dh = Q.shape
    Hkv = K.shape[2]
    dev = Q.device
    heads, hs = _heads_arg(head_list, Hq)
    Ntm = int(N_t_max if N_t_max is not None else (row_mask.shape[1] if row_mask is not None
                                                   else int(text_len.max().item())))
    scores = torch.empty((B, N_v), dtype=torch.float32, device=dev)
    L = lib()
    dt = _dtype_code(Q)
    need = L.provip_head_scores_workspace_size(B, Lm, hs, Ntm, N_v, algo, dt)
    if ws is None or ws.numel() < need:
        ws = workspace(need, dev)
    rc = L.provip_head_scores(_ptr(Q), _ptr(K), B, Lm, Hq, Hkv, dh, heads, hs, _i32(text_start),
                              _i32(text_len), _u8(row_mask), Ntm, vis_start, N_v, _i32(seq_len), dt,
                              algo, _ptr(scores), _ptr(ws), ws.numel(), _stream(dev))
    _check(rc, "provip_head_scores")
    return scores


def _outs(hidden, K, V, pos, B, L_out, device=None):
    dev = hidden.device if device is None else device
    ho = torch.empty((B, L_out) + tuple(hidden.shape[2:]), dtype=hidden.dtype, device=dev)
    ko = torch.empty((B, L_out) + tuple(K.shape[2:]), dtype=K.dtype, device=dev) if K is not None else None
    vo = torch.empty((B, L_out) + tuple(V.shape[2:]), dtype=V.dtype, device=dev) if V is not None else None
    po = torch.full((pos.shape[0], B, L_out), -1, dtype=torch.int32, device=dev) if pos is not None else None
    return ho, ko, vo, po


def provip_compact(idx, hidden, K, V, pos, seq_len, vis_start, N_v, out=None):
    """hidden, K, V, pos and the outputs may be device tensors or pinned host
    tensors (the library detects host memory); idx and seq_len live on the
    device, and the outputs default to device tensors."""
    B, Lm, D = hidden.shape
    keep = idx.shape[1]
    Hkv, dh = (K.shape[2], K.shape[3]) if K is not None else (0, 0)
    P = pos.shape[0] if pos is not None else 0
    ho, ko, vo, po = out if out is not None else _outs(hidden, K, V, pos, B, Lm - N_v + keep, idx.device)
    slo = torch.empty(B, dtype=torch.int32, device=idx.device)
    rc = lib().provip_compact(_i32(idx), B, N_v, keep, _ptr_host_ok(hidden), D, _ptr_host_ok(K), _ptr_host_ok(V),
                              Hkv, dh, _i32_host_ok(pos), P, _i32(seq_len), Lm, vis_start, _dtype_code(hidden),
                              _ptr_host_ok(ho), _ptr_host_ok(ko), _ptr_host_ok(vo), _i32_host_ok(po), _i32(slo),
                              _stream(idx.device))
    _check(rc, "provip_compact")
    return dict(hidden=ho, K=ko, V=vo, pos=po, seq_len=slo)


def provip_topk_compact(scores, keep, hidden, K, V, pos, seq_len, vis_start):
    B, Lm, D = hidden.shape
    N_v = scores.shape[1]
    Hkv, dh = (K.shape[2], K.shape[3]) if K is not None else (0, 0)
    P = pos.shape[0] if pos is not None else 0
    ho, ko, vo, po = _outs(hidden, K, V, pos, B, Lm - N_v + keep)
    idx = torch.empty((B, keep), dtype=torch.int32, device=hidden.device)
    slo = torch.empty(B, dtype=torch.int32, device=hidden.device)
    rc = lib().provip_topk_compact(_ptr(scores), B, N_v, keep, _ptr(hidden), D, _ptr(K), _ptr(V), Hkv,
                                   dh, _i32(pos), P, _i32(seq_len), Lm, vis_start,
                                   _dtype_code(hidden), _ptr(ho), _ptr(ko), _ptr(vo), _i32(po),
                                   _ptr(idx), _i32(slo), _stream(hidden.device))
    _check(rc, "provip_topk_compact")
    return dict(hidden=ho, K=ko, V=vo, pos=po, idx=idx, seq_len=slo)


class PruneStep:
    """Pre-allocated outputs + workspace for repeated provip_prune calls (one shape)."""

    def __init__(self, Q, K, V, hidden, pos, head_list, N_t_max, N_v, keep, algo=ALGO_AUTO,
                 want_scores=True, flags=0, ws=None, device=None, host_rows=False):
        """Q, K, V, hidden, pos give the shapes and dtypes (meta tensors are fine
        with device=...). host_rows: the compacted outputs are pinned host
        tensors, and hidden, V and pos may be pinned host tensors too
        (PROVIP_PRUNE_HOST_ROWS)."""
        B, Lm, Hq, dh = Q.shape
        self.shape = (B, Lm, Hq, K.shape[2], dh, hidden.shape[2])
        self.heads, self.H_sel = _heads_arg(head_list, Q.shape[2])
        self.N_t_max, self.N_v, self.keep, self.algo = int(N_t_max), int(N_v), int(keep), algo
        self.flags = int(flags) | (PRUNE_HOST_ROWS if host_rows else 0)
        dev = Q.device if device is None else torch.device(device)
        self.dtype = _dtype_code(Q)
        L_out = Lm - N_v + keep
        self.hidden_out, self.K_out, self.V_out, self.pos_out = _outs(hidden, K, V, pos, B, L_out, dev)
        if host_rows:
            self.hidden_out, self.K_out, self.V_out, self.pos_out = (
                None if t is None else torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
                for t in (self.hidden_out, self.K_out, self.V_out, self.pos_out))
        self.idx = torch.empty((B, keep), dtype=torch.int32, device=dev)
        self.seq_len_out = torch.empty(B, dtype=torch.int32, device=dev)
        self.scores = torch.empty((B, N_v), dtype=torch.float32, device=dev) if want_scores else None
        need = lib().provip_prune_workspace_size(B, Lm, self.H_sel, self.N_t_max, N_v, algo, self.dtype)
        self.ws = ws if ws is not None and ws.numel() >= need else workspace(need, dev)

    def __call__(self, Q, K, V, hidden, pos, text_start, text_len, seq_len, vis_start,
                 row_mask=None, stream=None):
        B, Lm, Hq, Hkv, dh, D = self.shape
        P = pos.shape[0] if pos is not None else 0
        st = ctypes.c_void_p(stream.cuda_stream) if stream is not None else _stream(Q.device)
        hp = _ptr_host_ok if self.flags & PRUNE_HOST_ROWS else _ptr
        rc = lib().provip_prune(_ptr(Q), _ptr(K), hp(V), hp(hidden), B, Lm, Hq, Hkv, dh, D,
                                self.heads, self.H_sel, _i32(text_start), _i32(text_len),
                                _u8(row_mask), self.N_t_max, vis_start, self.N_v, _i32(seq_len),
                                _i32_host_ok(pos) if hp is _ptr_host_ok else _i32(pos), P, self.keep,
                                self.dtype, self.algo, hp(self.hidden_out), hp(self.K_out),
                                hp(self.V_out),
                                _i32_host_ok(self.pos_out) if hp is _ptr_host_ok else _i32(self.pos_out),
                                _ptr(self.idx), _i32(self.seq_len_out), _ptr(self.scores),
                                _ptr(self.ws), self.ws.numel(), self.flags, st)
        _check(rc, "provip_prune")
        return dict(hidden=self.hidden_out, K=self.K_out, V=self.V_out, pos=self.pos_out,
                    idx=self.idx, seq_len=self.seq_len_out, scores=self.scores)


def provip_prune(Q, K, V, hidden, pos, head_list, text_start, text_len, seq_len, vis_start, N_v,
                 keep, row_mask=None, algo=ALGO_AUTO, N_t_max=None):
    Ntm = int(N_t_max if N_t_max is not None else int(text_len.max().item()))
    step = PruneStep(Q, K, V, hidden, pos, head_list, Ntm, N_v, keep, algo)
    return step(Q, K, V, hidden, pos, text_start, text_len, seq_len, vis_start, row_mask)


def provip_head_topk(Q, K, head_list, text_start, text_len, seq_len, vis_start, N_v, keep,
                     row_mask=None, algo=ALGO_AUTO, N_t_max=None, ws=None, want_scores=True):
    B, Lm, Hq, dh = Q.shape
    Hkv = K.shape[2]
    dev = Q.device
    heads, hs = _heads_arg(head_list, Hq)
    Ntm = int(N_t_max if N_t_max is not None else int(text_len.max().item()))
    idx = torch.empty((B, keep), dtype=torch.int32, device=dev)
    scores = torch.empty((B, N_v), dtype=torch.float32, device=dev) if want_scores else None
    L = lib()
    dt = _dtype_code(Q)
    need = L.provip_head_scores_workspace_size(B, Lm, hs, Ntm, N_v, algo, dt)
    if ws is None or ws.numel() < need:
        ws = workspace(need, dev)
    rc = L.provip_head_topk(_ptr(Q), _ptr(K), B, Lm, Hq, Hkv, dh, heads, hs, _i32(text_start),
                            _i32(text_len), _u8(row_mask), Ntm, vis_start, N_v, _i32(seq_len), keep, dt,
                            algo, _ptr(idx), _ptr(scores), _ptr(ws), ws.numel(), _stream(dev))
    _check(rc, "provip_head_topk")
    return idx, scores


def provip_head_scores_noalloc(Q, K, head_list, text_start, text_len, seq_len, vis_start, N_v,
                               row_mask=None, algo=ALGO_AUTO, N_t_max=None):
    """provip_head_scores without a workspace: the scratch is the library's own
    static device array (for hosts that cannot allocate device memory; shapes
    needing more than PROVIP_NOALLOC_SCRATCH_BYTES are rejected)."""
    B, Lm, Hq, dh = Q.shape
    Hkv = K.shape[2]
    dev = Q.device
    heads, hs = _heads_arg(head_list, Hq)
    Ntm = int(N_t_max if N_t_max is not None else int(text_len.max().item()))
    scores = torch.empty((B, N_v), dtype=torch.float32, device=dev)
    rc = lib().provip_head_scores_noalloc(_ptr(Q), _ptr(K), B, Lm, Hq, Hkv, dh, heads, hs, _i32(text_start),
                                          _i32(text_len), _u8(row_mask), Ntm, vis_start, N_v, _i32(seq_len),
                                          _dtype_code(Q), algo, _ptr(scores), _stream(dev))
    _check(rc, "provip_head_scores_noalloc")
    return scores


# ---------------------------------------------------------------------------
# visual-head identification (Sec. 4.4)
# ---------------------------------------------------------------------------
def provip_head_confidence(Q, K, text_start, text_len, seq_len, vis_start, N_v, N_vis,
                           crit_mask=None, algo=ALGO_AUTO, N_t_max=None, ws=None, want_conf=True):
    """Head confidence C [B, H_q] over the critical rows and the N_vis visual heads
    [B, N_vis] (ascending) of every sample. Returns (vis_heads, conf or None)."""
    B, Lm, Hq, dh = Q.shape
    Hkv = K.shape[2]
    dev = Q.device
    Ntm = int(N_t_max if N_t_max is not None else (crit_mask.shape[1] if crit_mask is not None
                                                   else int(text_len.max().item())))
    vis = torch.empty((B, N_vis), dtype=torch.int32, device=dev)
    conf = torch.empty((B, Hq), dtype=torch.float32, device=dev) if want_conf else None
    L = lib()
    dt = _dtype_code(Q)
    need = L.provip_visual_heads_workspace_size(B, Lm, Hq, Ntm, N_v, N_vis, algo, dt)
    if ws is None or ws.numel() < need:
        ws = workspace(need, dev)
    rc = L.provip_head_confidence(_ptr(Q), _ptr(K), B, Lm, Hq, Hkv, dh, _i32(text_start),
                                  _i32(text_len), _u8(crit_mask), Ntm, vis_start, N_v, _i32(seq_len),
                                  N_vis, dt, algo, _ptr(conf), _ptr(vis), _ptr(ws), ws.numel(),
                                  _stream(dev))
    _check(rc, "provip_head_confidence")
    return vis, conf


class VisualHeadsPruneStep:
    """Pre-allocated outputs + workspace for repeated provip_prune_visual_heads calls."""

    def __init__(self, Q, K, V, hidden, pos, N_t_max, N_v, keep, N_vis, algo=ALGO_AUTO,
                 want_scores=True, want_conf=True, flags=0, ws=None, device=None):
        """Q, K, V, hidden, pos give the shapes and dtypes (meta tensors are fine
        with device=...)."""
        B, Lm, Hq, dh = Q.shape
        self.shape = (B, Lm, Hq, K.shape[2], dh, hidden.shape[2])
        self.N_t_max, self.N_v, self.keep, self.N_vis, self.algo = int(N_t_max), int(N_v), int(keep), int(N_vis), algo
        self.flags = int(flags)
        dev = Q.device if device is None else torch.device(device)
        self.dtype = _dtype_code(Q)
        L_out = Lm - N_v + keep
        self.hidden_out, self.K_out, self.V_out, self.pos_out = _outs(hidden, K, V, pos, B, L_out, dev)
        self.idx = torch.empty((B, keep), dtype=torch.int32, device=dev)
        self.seq_len_out = torch.empty(B, dtype=torch.int32, device=dev)
        self.scores = torch.empty((B, N_v), dtype=torch.float32, device=dev) if want_scores else None
        self.vis_heads = torch.empty((B, self.N_vis), dtype=torch.int32, device=dev)
        self.conf = torch.empty((B, Hq), dtype=torch.float32, device=dev) if want_conf else None
        need = lib().provip_visual_heads_workspace_size(B, Lm, Hq, self.N_t_max, N_v, self.N_vis, algo,
                                                        self.dtype)
        self.ws = ws if ws is not None and ws.numel() >= need else workspace(need, dev)

    def __call__(self, Q, K, V, hidden, pos, text_start, text_len, seq_len, vis_start,
                 crit_mask=None, stream=None):
        B, Lm, Hq, Hkv, dh, D = self.shape
        P = pos.shape[0] if pos is not None else 0
        st = ctypes.c_void_p(stream.cuda_stream) if stream is not None else _stream(Q.device)
        rc = lib().provip_prune_visual_heads(
            _ptr(Q), _ptr(K), _ptr(V), _ptr(hidden), B, Lm, Hq, Hkv, dh, D, _i32(text_start),
            _i32(text_len), _u8(crit_mask), self.N_t_max, vis_start, self.N_v, _i32(seq_len),
            _i32(pos), P, self.N_vis, self.keep, self.dtype, self.algo, _ptr(self.hidden_out),
            _ptr(self.K_out), _ptr(self.V_out), _i32(self.pos_out), _ptr(self.idx),
            _i32(self.seq_len_out), _ptr(self.scores), _ptr(self.vis_heads), _ptr(self.conf),
            _ptr(self.ws), self.ws.numel(), self.flags, st)
        _check(rc, "provip_prune_visual_heads")
        return dict(hidden=self.hidden_out, K=self.K_out, V=self.V_out, pos=self.pos_out,
                    idx=self.idx, seq_len=self.seq_len_out, scores=self.scores,
                    vis_heads=self.vis_heads, conf=self.conf)


def provip_prune_visual_heads(Q, K, V, hidden, pos, text_start, text_len, seq_len, vis_start, N_v,
                              keep, N_vis, crit_mask=None, algo=ALGO_AUTO, N_t_max=None):
    Ntm = int(N_t_max if N_t_max is not None else (crit_mask.shape[1] if crit_mask is not None
                                                   else int(text_len.max().item())))
    step = VisualHeadsPruneStep(Q, K, V, hidden, pos, Ntm, N_v, keep, N_vis, algo)
    return step(Q, K, V, hidden, pos, text_start, text_len, seq_len, vis_start, crit_mask)
