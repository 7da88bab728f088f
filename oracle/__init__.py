"""ProViP oracle: plain fp64 CPU restatement of the pruning path (test infrastructure).

TEST INFRASTRUCTURE ONLY. The tests, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` are the only
callers. The CUDA library never imports, links or executes anything here, and
nothing here imports the CUDA library.

The arithmetic lives in ``provip_oracle.c`` (double precision, plain loops, one
function per equation group of the paper, Sec. 4.2-4.4); this module compiles it
with gcc and wraps it with ctypes + numpy. ``oracle.brute`` holds pure-Python
brute-force versions for tiny inputs, used to pin the C code.

Parity status per function:
  crit_text, relevance, topk, head_scores, head_confidence, compact_map:
      pinned (closed forms, invariants, library routines, brute force; see the
      ``tests/test_oracle_*.py`` files).
  merge: the paper defers the aggregation rule to ApET and does not state it.
      The reading implemented (cosine-nearest kept token, uniform mean) is pinned
      by brute force and invariants only: "parity unpinned" by the paper.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "provip_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libprovip_oracle.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile the oracle shared library with gcc (-O2, OpenMP). Returns its path."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-std=c99", "-o", tmp, _SRC, "-lm"]
        )
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_P = ctypes.c_void_p
_I = ctypes.c_int
_Z = ctypes.c_size_t


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB_PATH)
            L.po_crit_text.argtypes = [_P, _I, _I, _P, _P]
            L.po_relevance.argtypes = [_P, _P, _I, _P, _I, _I, _P, _P, _P]
            L.po_topk.argtypes = [_P, _I, _I, _P]
            L.po_merge.argtypes = [_P, _I, _I, _P, _I, _P, _P]
            L.po_head_scores.argtypes = [_P, _P, _I, _I, _I, _I, _P, _I, _P, _I, _I, _I, _P]
            L.po_head_confidence.argtypes = [_P, _P, _I, _I, _I, _I, _P, _I, _I, _I, _P]
            L.po_compact_map.argtypes = [_I, _I, _I, _P, _I, _P]
            L.po_gather_rows.argtypes = [_P, _Z, _P, _I, _P]
            L.po_gather_rows.restype = None
            L.po_prune_batch.argtypes = (
                [_I, _I, _P, _P, _P, _I, _I, _I, _P, _I, _P, _P, _I, _I, _I, _P, _Z, _P, _P, _Z, _P, _I]
                + [_P, _P, _P, _P, _P, _P, _P, _I]
            )
            L.po_max_threads.argtypes = []
            _lib = L
    return _lib


def _f64(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _i32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def _check(rc, what):
    if rc != 0:
        raise ValueError(f"oracle {what} failed with code {rc}")


def crit_text(E_t):
    """Sec. 4.2: returns (r [n], mask [n] uint8) for one sample's text rows E_t [n, d]."""
    E = _f64(E_t)
    n, d = E.shape
    r = np.zeros(n, np.float64)
    m = np.zeros(n, np.uint8)
    _check(lib().po_crit_text(_ptr(E), n, d, _ptr(r), _ptr(m)), "crit_text")
    return r, m


def relevance(E_t, mask, E_v, want_M=False):
    """Sec. 4.3: p [nv] (and optionally M [|T|, nv], mu [|T|]) for one sample."""
    Et, Ev = _f64(E_t), _f64(E_v)
    mk = np.ascontiguousarray(np.asarray(mask, dtype=np.uint8))
    nt, d = Et.shape
    nv = Ev.shape[0]
    nT = int((mk != 0).sum())
    p = np.zeros(nv, np.float64)
    M = np.zeros((max(nT, 1), nv), np.float64) if want_M else None
    mu = np.zeros(max(nT, 1), np.float64) if want_M else None
    rc = lib().po_relevance(_ptr(Et), _ptr(mk), nt, _ptr(Ev), nv, d, _ptr(p),
                            _ptr(M) if want_M else None, _ptr(mu) if want_M else None)
    _check(rc, "relevance")
    return (p, M[:nT], mu[:nT]) if want_M else p


def topk(scores, k):
    """Top-k indices (ties to the lower index), ascending."""
    s = _f64(scores)
    idx = np.zeros(k, np.int32)
    _check(lib().po_topk(_ptr(s), s.shape[0], k, _ptr(idx)), "topk")
    return idx


def merge(E_v, keep):
    """Sec. 4.3 merge reading: returns (assign [nv] positions in keep, merged [n1, d])."""
    Ev = _f64(E_v)
    kp = _i32(keep)
    nv, d = Ev.shape
    assign = np.zeros(nv, np.int32)
    merged = np.zeros((kp.shape[0], d), np.float64)
    _check(lib().po_merge(_ptr(Ev), nv, d, _ptr(kp), kp.shape[0], _ptr(assign), _ptr(merged)), "merge")
    return assign, merged


def head_scores(Q, K, heads, rows, vis_start, nv):
    """Sec. 4.4: v [nv] for one sample. Q [L, Hq, dh], K [L, Hkv, dh]."""
    Qd, Kd = _f64(Q), _f64(K)
    L, Hq, dh = Qd.shape
    Hkv = Kd.shape[1]
    hl, rw = _i32(heads), _i32(rows)
    v = np.zeros(nv, np.float64)
    rc = lib().po_head_scores(_ptr(Qd), _ptr(Kd), L, Hq, Hkv, dh, _ptr(hl), hl.shape[0],
                              _ptr(rw), rw.shape[0], vis_start, nv, _ptr(v))
    _check(rc, "head_scores")
    return v


def head_confidence(Q, K, rows, vis_start, nv):
    """Sec. 4.4: C [Hq] head confidence over the given (critical) rows."""
    Qd, Kd = _f64(Q), _f64(K)
    L, Hq, dh = Qd.shape
    Hkv = Kd.shape[1]
    rw = _i32(rows)
    C = np.zeros(Hq, np.float64)
    rc = lib().po_head_confidence(_ptr(Qd), _ptr(Kd), L, Hq, Hkv, dh, _ptr(rw), rw.shape[0],
                                  vis_start, nv, _ptr(C))
    _check(rc, "head_confidence")
    return C


def compact_map(seq_len, vis_start, nv, keep):
    """Source rows of the compacted sequence, in order."""
    kp = _i32(keep)
    src = np.zeros(seq_len, np.int32)
    n = lib().po_compact_map(seq_len, vis_start, nv, _ptr(kp), kp.shape[0], _ptr(src))
    if n < 0:
        raise ValueError("oracle compact_map: invalid arguments")
    return src[:n]


def gather_rows(src, rows):
    """Byte-exact row gather of a C-contiguous 2-D (or higher) array along axis 0."""
    a = np.ascontiguousarray(src)
    rw = _i32(rows)
    out = np.empty((rw.shape[0],) + a.shape[1:], a.dtype)
    row_bytes = a[0].nbytes if a.shape[0] else 0
    lib().po_gather_rows(_ptr(a), row_bytes, _ptr(rw), rw.shape[0], _ptr(out))
    return out


def prune_batch(Q, K, heads, text_start, text_len, seq_len, vis_start, nv, k,
                hidden, Kraw, Vraw, pos, threads=0):
    """Sec. 4.4 end to end for a batch (the timed CPU baseline).

    Q, K: fp64 [B, Lmax, H, dh]; hidden, Kraw, Vraw: raw arrays [B, Lmax, ...]
    (any dtype, copied byte-exactly); pos int32 [P, B, Lmax].
    Returns dict(v, idx, hidden, K, V, pos, seq_len).
    """
    Qd, Kd = _f64(Q), _f64(K)
    B, Lmax, Hq, dh = Qd.shape
    Hkv = Kd.shape[2]
    hl = _i32(heads)
    ts, tl, sl = _i32(text_start), _i32(text_len), _i32(seq_len)
    hid = np.ascontiguousarray(hidden)
    Kr = np.ascontiguousarray(Kraw) if Kraw is not None else None
    Vr = np.ascontiguousarray(Vraw) if Vraw is not None else None
    ps = _i32(pos)
    P = ps.shape[0]
    Lout = Lmax - nv + k
    v = np.zeros((B, nv), np.float64)
    idx = np.zeros((B, k), np.int32)
    hid_o = np.zeros((B, Lout) + hid.shape[2:], hid.dtype)
    K_o = np.zeros((B, Lout) + Kr.shape[2:], Kr.dtype) if Kr is not None else None
    V_o = np.zeros((B, Lout) + Vr.shape[2:], Vr.dtype) if Vr is not None else None
    pos_o = np.zeros((P, B, Lout), np.int32)
    slo = np.zeros(B, np.int32)
    hid_rb = hid[0, 0].nbytes
    kv_rb = Kr[0, 0].nbytes if Kr is not None else 0
    rc = lib().po_prune_batch(
        B, Lmax, _ptr(sl), _ptr(Qd), _ptr(Kd), Hq, Hkv, dh, _ptr(hl), hl.shape[0], _ptr(ts),
        _ptr(tl), vis_start, nv, k, _ptr(hid), hid_rb,
        _ptr(Kr) if Kr is not None else None, _ptr(Vr) if Vr is not None else None, kv_rb,
        _ptr(ps), P, _ptr(v), _ptr(idx), _ptr(hid_o),
        _ptr(K_o) if K_o is not None else None, _ptr(V_o) if V_o is not None else None,
        _ptr(pos_o), _ptr(slo), int(threads))
    _check(rc, "prune_batch")
    return dict(v=v, idx=idx, hidden=hid_o, K=K_o, V=V_o, pos=pos_o, seq_len=slo)


def max_threads() -> int:
    return int(lib().po_max_threads())
