"""fp64 CPU oracle for SPIRe speculation-round attention (test infrastructure).

This package is the slow, obviously correct reference the CUDA library is
checked against.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it.
It shares no code with ``paper_2504_06419_gb300`` and never imports it.

The arithmetic lives in ``spire_oracle.c`` (plain C, double precision, a
pthread pool over independent (sequence, query head) units).  This module
compiles it with gcc on first use and wraps it with ctypes.  Inputs are numpy
arrays; bf16 tensors are passed as their raw 16-bit patterns (``uint16``).

Functions (each follows the passage cited in ``spire_oracle.c``):
  verify(...)          verification attention of the k+1 block tokens
                       (Section 2: t_verify; Fig. 1 and Table 1 captions)
  draft_ring(...)      sink + sliding-window attention over the bounded cache
                       (Section 3.1, Section 3.3)
  draft_logical(...)   the same mask over a full-length logical memory
  ring_pack(...)       place logical memory entries into the bounded cache
  draft_slot(p, ...)   slot of logical position p
  feedback_mix(...)    per-layer feedback memory vectors (Section 3.3)
  feedback_append(...) memory vector -> K/V projection -> bounded-cache slot
  round_bf16(v)        nearest-even bf16 bits of a double
  verify_tokens(...)   modified rejection sampling of a round's draft tokens
  magicdec(...)        StreamingLLM draft attention over the target's paged cache
                       with positions inside the reduced cache
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "spire_oracle.c")
_LIB = os.path.join(_HERE, "libspire_oracle.so")
_lock = threading.Lock()
_lib = None

_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_F64 = ctypes.c_double


def build(force: bool = False, src: str = _SRC, out: str = _LIB) -> str:
    """Compile the oracle shared library with gcc (plain C11, -O2, pthreads)."""
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    tmp = out + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-pthread",
           "-fno-fast-math", "-ffp-contract=off", "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def _declare(lib):
    lib.oracle_verify.restype = _I64
    lib.oracle_verify.argtypes = [_P, _P, _P, _P, _P, _I32, _I32, _I32, _I32, _I32,
                                  _I32, _I32, _I32, _F64, _P, _P, _I32]
    lib.oracle_draft_ring.restype = _I64
    lib.oracle_draft_ring.argtypes = [_P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32,
                                      _F64, _P, _P, _I32]
    lib.oracle_draft_logical.restype = _I64
    lib.oracle_draft_logical.argtypes = [_P, _P, _P, _P, _I32, _I32, _I32, _I32, _I64,
                                         _I32, _I32, _F64, _P, _P, _I32]
    lib.oracle_ring_pack.restype = _I64
    lib.oracle_ring_pack.argtypes = [_P, _P, _P, _I32, _I32, _I32, _I64, _I32, _I32, _P]
    lib.oracle_draft_slot.restype = _I64
    lib.oracle_draft_slot.argtypes = [_I64, _I32, _I32]
    lib.oracle_round_bf16.restype = ctypes.c_uint16
    lib.oracle_round_bf16.argtypes = [_F64]
    lib.oracle_feedback_mix.restype = _I64
    lib.oracle_feedback_mix.argtypes = [_P, _P, _I32, _I32, _I32, _I32, _P]
    lib.oracle_magicdec.restype = _I64
    lib.oracle_magicdec.argtypes = [_P, _P, _P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _I32,
                                    _I32, _I32, _F64, _F64, _P]
    lib.oracle_verify_tokens.restype = _I64
    lib.oracle_verify_tokens.argtypes = [_P, _P, _P, _P, _P, _I32, _I32, _I32, _P, _P]
    lib.oracle_feedback_append.restype = _I64
    lib.oracle_feedback_append.argtypes = [_P, _P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32,
                                           _I32, _I32, _F64, _P]
    return lib


def load(path: str | None = None):
    """Load (building first if needed) the oracle library; returns a ctypes CDLL."""
    global _lib
    if path is not None:
        return _declare(ctypes.CDLL(path))
    with _lock:
        if _lib is None:
            _lib = _declare(ctypes.CDLL(build()))
    return _lib


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


def _u16(a) -> np.ndarray:
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError("bf16 inputs must be passed as uint16 bit patterns, got %s" % a.dtype)
    return a


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


def _ptr(a) -> int:
    return a.ctypes.data if a is not None else None


def _mask(unit_mask, n):
    if unit_mask is None:
        return None
    m = np.ascontiguousarray(unit_mask, dtype=np.uint8).reshape(-1)
    if m.size != n:
        raise ValueError("unit_mask must have B*Hq entries")
    return m


def verify(q, k_cache, v_cache, block_table, ctx_lens, k, scale=1.0,
           unit_mask=None, threads=None, lib=None):
    """Verification attention, fp64.

    q [B, k+1, Hq, D], k_cache / v_cache [num_pages, Hkv, page_size, D] (uint16
    bf16 bits), block_table int32 [B, max_pages], ctx_lens int32 [B].
    Returns (out float64 [B, k+1, Hq, D], n_bad_sequences).
    """
    lib = lib or load()
    q, kc, vc = _u16(q), _u16(k_cache), _u16(v_cache)
    bt, cl = _i32(block_table), _i32(ctx_lens)
    B, rows, Hq, D = q.shape
    if rows != k + 1:
        raise ValueError("q must have k+1 rows")
    num_pages, Hkv, page_size, D2 = kc.shape
    if D2 != D or vc.shape != kc.shape:
        raise ValueError("cache shape mismatch")
    max_pages = bt.shape[1] if bt.ndim == 2 else 0
    out = np.zeros((B, rows, Hq, D), dtype=np.float64)
    m = _mask(unit_mask, B * Hq)
    n_bad = lib.oracle_verify(_ptr(q), _ptr(kc), _ptr(vc), _ptr(bt), _ptr(cl), B, k, Hq,
                              Hkv, D, page_size, max_pages, num_pages, float(scale),
                              _ptr(m), _ptr(out), threads or default_threads())
    if n_bad < 0:
        raise ValueError("oracle_verify rejected its arguments")
    return out, int(n_bad)


def draft_ring(q, kv, ctx_lens, n_sink, window, scale=1.0, unit_mask=None,
               threads=None, lib=None):
    """Draft sink+window attention over the bounded cache kv [B, 2, Hkv, S, D]."""
    lib = lib or load()
    q, kv, cl = _u16(q), _u16(kv), _i32(ctx_lens)
    B, Hq, D = q.shape
    _, two, Hkv, S, D2 = kv.shape
    if two != 2 or D2 != D or S != n_sink + window:
        raise ValueError("kv must be [B, 2, Hkv, n_sink + window, D]")
    out = np.zeros((B, Hq, D), dtype=np.float64)
    m = _mask(unit_mask, B * Hq)
    n_bad = lib.oracle_draft_ring(_ptr(q), _ptr(kv), _ptr(cl), B, Hq, Hkv, D, n_sink,
                                  window, float(scale), _ptr(m), _ptr(out),
                                  threads or default_threads())
    if n_bad < 0:
        raise ValueError("oracle_draft_ring rejected its arguments")
    return out, int(n_bad)


def draft_logical(q, k_log, v_log, ctx_lens, n_sink, window, scale=1.0,
                  unit_mask=None, threads=None, lib=None):
    """Draft attention over a full logical memory k_log / v_log [B, Hkv, T, D]."""
    lib = lib or load()
    q, kl, vl, cl = _u16(q), _u16(k_log), _u16(v_log), _i32(ctx_lens)
    B, Hq, D = q.shape
    _, Hkv, T, D2 = kl.shape
    if D2 != D or vl.shape != kl.shape:
        raise ValueError("logical cache shape mismatch")
    out = np.zeros((B, Hq, D), dtype=np.float64)
    m = _mask(unit_mask, B * Hq)
    n_bad = lib.oracle_draft_logical(_ptr(q), _ptr(kl), _ptr(vl), _ptr(cl), B, Hq, Hkv, D,
                                     T, n_sink, window, float(scale), _ptr(m), _ptr(out),
                                     threads or default_threads())
    if n_bad < 0:
        raise ValueError("oracle_draft_logical rejected its arguments")
    return out, int(n_bad)


def ring_pack(k_log, v_log, ctx_lens, n_sink, window, kv_out=None, lib=None):
    """Pack logical memory entries into a bounded cache; returns kv [B,2,Hkv,S,D]."""
    lib = lib or load()
    kl, vl, cl = _u16(k_log), _u16(v_log), _i32(ctx_lens)
    B, Hkv, T, D = kl.shape
    S = n_sink + window
    if kv_out is None:
        kv_out = np.zeros((B, 2, Hkv, S, D), dtype=np.uint16)
    if lib.oracle_ring_pack(_ptr(kl), _ptr(vl), _ptr(cl), B, Hkv, D, T, n_sink, window,
                            _ptr(kv_out)) != 0:
        raise ValueError("oracle_ring_pack rejected its arguments")
    return kv_out


def draft_slot(p, n_sink, window, lib=None):
    lib = lib or load()
    return int(lib.oracle_draft_slot(int(p), int(n_sink), int(window)))


def round_bf16(v, lib=None):
    """Nearest-even bf16 bit pattern of the double v."""
    lib = lib or load()
    return int(lib.oracle_round_bf16(float(v)))


def feedback_mix(x, w, lib=None):
    """Memory vectors m [n_dl, B, d_model] (float64) from activations
    x [n_act, B, d_model] (bf16 bits) and mixing weights w [n_dl, n_act]."""
    lib = lib or load()
    x = _u16(x)
    w = np.ascontiguousarray(w, dtype=np.float64)
    n_act, B, d_model = x.shape
    n_dl, n_act2 = w.shape
    if n_act2 != n_act:
        raise ValueError("w must be [n_dl, n_act]")
    m = np.zeros((n_dl, B, d_model), dtype=np.float64)
    if lib.oracle_feedback_mix(_ptr(x), _ptr(w), n_act, n_dl, B, d_model, _ptr(m)) != 0:
        raise ValueError("oracle_feedback_mix rejected its arguments")
    return m


def feedback_append(x, w, w_kv, pos, kv, n_sink, window, rope_theta=0.0, lib=None):
    """Append one memory entry per sequence and draft layer to the bounded
    caches kv [n_dl, B, 2, Hkv, S, D] (bf16 bits, updated in place).

    x [n_act, B, d_model] bf16 bits; w [n_dl, n_act]; w_kv [n_dl, 2*Hkv*D,
    d_model] bf16 bits; pos int32 [B].  Returns the number of sequences with
    a negative position (left unwritten)."""
    lib = lib or load()
    x, wkv, ps = _u16(x), _u16(w_kv), _i32(pos)
    w = np.ascontiguousarray(w, dtype=np.float64)
    if not (isinstance(kv, np.ndarray) and kv.dtype == np.uint16 and kv.flags.c_contiguous):
        raise TypeError("kv must be a C-contiguous uint16 array (updated in place)")
    n_act, B, d_model = x.shape
    n_dl, two, Hkv, S, D = kv.shape[0], kv.shape[2], kv.shape[3], kv.shape[4], kv.shape[5]
    if (kv.shape[1] != B or two != 2 or S != n_sink + window or w.shape != (n_dl, n_act)
            or wkv.shape != (n_dl, 2 * Hkv * D, d_model) or ps.shape != (B,)):
        raise ValueError("feedback_append: shape mismatch")
    n_bad = lib.oracle_feedback_append(_ptr(x), _ptr(w), _ptr(wkv), _ptr(ps), n_act, n_dl, B,
                                       d_model, Hkv, D, n_sink, window, float(rope_theta),
                                       _ptr(kv))
    if n_bad < 0:
        raise ValueError("oracle_feedback_append rejected its arguments")
    return int(n_bad)


def verify_tokens(p, q, x, u, e, lib=None):
    """Token verification of one round per sequence.

    p float32 [B, k+1, V], q float32 [B, k, V], x int32 [B, k], u float32 [B, k],
    e float32 [B, V].  Returns (out int32 [B, k+1], n_accepted int32 [B], n_bad)."""
    lib = lib or load()
    p = np.ascontiguousarray(p, dtype=np.float32)
    q = np.ascontiguousarray(q, dtype=np.float32)
    x = _i32(x)
    u = np.ascontiguousarray(u, dtype=np.float32)
    e = np.ascontiguousarray(e, dtype=np.float32)
    B, kp1, V = p.shape
    k = kp1 - 1
    if q.shape != (B, k, V) or x.shape != (B, k) or u.shape != (B, k) or e.shape != (B, V):
        raise ValueError("verify_tokens: shape mismatch")
    out = np.zeros((B, kp1), dtype=np.int32)
    n_acc = np.zeros(B, dtype=np.int32)
    n_bad = lib.oracle_verify_tokens(_ptr(p), _ptr(q), _ptr(x), _ptr(u), _ptr(e), B, k, V,
                                     _ptr(out), _ptr(n_acc))
    if n_bad < 0:
        raise ValueError("oracle_verify_tokens rejected its arguments")
    return out, n_acc, int(n_bad)


def magicdec(q, k_cache, v_cache, block_table, ctx_lens, n_sink, window, rope_theta,
             scale=1.0, lib=None):
    """MagicDec draft attention: q bf16 bits [B, Hq, D] (not rotated), the
    target's paged caches [num_pages, Hkv, page_size, D] (keys rotated by their
    original positions), block_table [B, max_pages], ctx_lens [B].
    Returns (out float64 [B, Hq, D], n_bad)."""
    lib = lib or load()
    q, kc, vc = _u16(q), _u16(k_cache), _u16(v_cache)
    bt, cl = _i32(block_table), _i32(ctx_lens)
    B, Hq, D = q.shape
    num_pages, Hkv, page_size, D2 = kc.shape
    if D2 != D or vc.shape != kc.shape:
        raise ValueError("cache shape mismatch")
    out = np.zeros((B, Hq, D), dtype=np.float64)
    n_bad = lib.oracle_magicdec(_ptr(q), _ptr(kc), _ptr(vc), _ptr(bt), _ptr(cl), B, Hq, Hkv, D,
                                page_size, bt.shape[1], num_pages, int(n_sink), int(window),
                                float(rope_theta), float(scale), _ptr(out))
    if n_bad < 0:
        raise ValueError("oracle_magicdec rejected its arguments")
    return out, int(n_bad)
