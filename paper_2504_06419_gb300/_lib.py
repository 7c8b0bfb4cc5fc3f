"""ctypes binding of libspire (include/spire.h): the same names and arguments,
marshalling only.  Every step of the attention runs in the library's CUDA
kernels; there is no Python or CPU fallback.  If libspire.so has not been
built, importing this module raises.

Tensor arguments may be torch tensors (their data_ptr() is passed) or plain
integers holding device addresses.  `stream` may be a torch.cuda.Stream, an
integer cudaStream_t, or None (the current torch stream of the tensors'
device).
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libspire.so")

SPIRE_OK = 0
SPIRE_ERR_INVALID_ARG = 1
SPIRE_ERR_UNSUPPORTED = 2
SPIRE_ERR_WORKSPACE = 3
SPIRE_ERR_CUDA = 4

SPIRE_DEVERR_CTX_LEN = 1
SPIRE_DEVERR_PAGE_ID = 2
SPIRE_DEVERR_TIMEOUT = 4
SPIRE_DEVERR_VALUE = 8

SPIRE_MAX_ROWS_PER_KV_HEAD = 128

EXPORTED = (
    "spire_verify_workspace_bytes",
    "spire_verify_attention",
    "spire_verify_attention_noalloc",
    "spire_draft_workspace_bytes",
    "spire_draft_sparse_attention",
    "spire_feedback_append_workspace_bytes",
    "spire_feedback_append",
    "spire_magicdec_workspace_bytes",
    "spire_magicdec_attention",
    "spire_verify_tokens_workspace_bytes",
    "spire_verify_tokens",
    "spire_draft_slot",
    "spire_get_device_error",
    "spire_get_cta_times",
    "spire_stream_read",
    "spire_test_stall_next_call",
    "spire_test_draft_slots",
    "spire_status_string",
)


class spire_attn_desc(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32),
        ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32),
        ("num_pages", ctypes.c_int32),
        ("softmax_scale", ctypes.c_float),
    ]


class spire_append_desc(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32),
        ("num_act", ctypes.c_int32),
        ("num_draft_layers", ctypes.c_int32),
        ("d_model", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("n_sink", ctypes.c_int32),
        ("window", ctypes.c_int32),
        ("rope_theta", ctypes.c_float),
    ]


class SpireError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__("%s failed: %s" % (what, status_string(status)))


def _load(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(
            "libspire.so is not built (%s); run `python paper_2504_06419_gb300/build.py`" % path)
    lib = ctypes.CDLL(path)
    P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    D = ctypes.POINTER(spire_attn_desc)
    lib.spire_verify_workspace_bytes.restype = SZ
    lib.spire_verify_workspace_bytes.argtypes = [D, I32]
    lib.spire_verify_attention.restype = ctypes.c_int
    lib.spire_verify_attention.argtypes = [P, P, P, P, P, I32, D, P, P, SZ, P]
    lib.spire_verify_attention_noalloc.restype = ctypes.c_int
    lib.spire_verify_attention_noalloc.argtypes = [P, P, P, P, P, I32, D, P, P]
    lib.spire_draft_workspace_bytes.restype = SZ
    lib.spire_draft_workspace_bytes.argtypes = [D, I32, I32]
    lib.spire_draft_sparse_attention.restype = ctypes.c_int
    lib.spire_draft_sparse_attention.argtypes = [P, P, P, I32, I32, D, P, P, SZ, P]
    A = ctypes.POINTER(spire_append_desc)
    lib.spire_feedback_append_workspace_bytes.restype = SZ
    lib.spire_feedback_append_workspace_bytes.argtypes = [A]
    lib.spire_feedback_append.restype = ctypes.c_int
    lib.spire_feedback_append.argtypes = [P, P, P, P, A, P, P, SZ, P]
    lib.spire_magicdec_workspace_bytes.restype = SZ
    lib.spire_magicdec_workspace_bytes.argtypes = [D, I32, I32]
    lib.spire_magicdec_attention.restype = ctypes.c_int
    lib.spire_magicdec_attention.argtypes = [P, P, P, P, P, I32, I32, ctypes.c_float, D, P, P, SZ,
                                             P]
    lib.spire_verify_tokens_workspace_bytes.restype = SZ
    lib.spire_verify_tokens_workspace_bytes.argtypes = [I32, I32, I32]
    lib.spire_verify_tokens.restype = ctypes.c_int
    lib.spire_verify_tokens.argtypes = [P, P, P, P, P, I32, I32, I32, P, P, P, SZ, P]
    lib.spire_draft_slot.restype = I64
    lib.spire_draft_slot.argtypes = [I64, I32, I32]
    lib.spire_get_device_error.restype = ctypes.c_int
    lib.spire_get_device_error.argtypes = [P, ctypes.POINTER(I32), P]
    lib.spire_get_cta_times.restype = ctypes.c_int
    lib.spire_get_cta_times.argtypes = [P, SZ, ctypes.POINTER(ctypes.c_uint64), I32,
                                        ctypes.POINTER(I32), P]
    lib.spire_stream_read.restype = ctypes.c_int
    lib.spire_stream_read.argtypes = [P, SZ, P]
    lib.spire_test_stall_next_call.restype = ctypes.c_int
    lib.spire_test_stall_next_call.argtypes = [I32]
    lib.spire_test_draft_slots.restype = ctypes.c_int
    lib.spire_test_draft_slots.argtypes = [P, ctypes.c_int64, I32, I32, P]
    lib.spire_status_string.restype = ctypes.c_char_p
    lib.spire_status_string.argtypes = [ctypes.c_int]
    return lib


LIB = _load()


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _desc_ref(desc):
    return ctypes.byref(desc) if desc is not None else None


def _stream(stream, like=None):
    if stream is None:
        import torch
        dev = like.device if like is not None and hasattr(like, "device") else None
        if dev is not None and dev.type == "cuda":
            return torch.cuda.current_stream(dev).cuda_stream
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_desc(batch, num_q_heads, num_kv_heads, head_dim, page_size=64, max_pages_per_seq=0,
              num_pages=0, softmax_scale=1.0) -> spire_attn_desc:
    return spire_attn_desc(int(batch), int(num_q_heads), int(num_kv_heads), int(head_dim),
                           int(page_size), int(max_pages_per_seq), int(num_pages),
                           float(softmax_scale))


def spire_verify_workspace_bytes(desc: spire_attn_desc, k: int) -> int:
    return int(LIB.spire_verify_workspace_bytes(_desc_ref(desc), int(k)))


def spire_draft_workspace_bytes(desc: spire_attn_desc, n_sink: int, window: int) -> int:
    return int(LIB.spire_draft_workspace_bytes(_desc_ref(desc), int(n_sink), int(window)))


def spire_verify_attention(q, k_cache, v_cache, block_table, ctx_lens, k, desc, out, workspace,
                           ws_bytes, stream=None) -> int:
    return int(LIB.spire_verify_attention(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(ctx_lens), int(k),
        _desc_ref(desc), _ptr(out), _ptr(workspace), int(ws_bytes), _stream(stream, q)))


def spire_verify_attention_noalloc(q, k_cache, v_cache, block_table, ctx_lens, k, desc, out,
                                   stream=None) -> int:
    """Verification attention with the library's own fixed scratch (no
    workspace argument, nothing allocated); see include/spire.h."""
    return int(LIB.spire_verify_attention_noalloc(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(ctx_lens), int(k),
        _desc_ref(desc), _ptr(out), _stream(stream, q)))


def spire_draft_sparse_attention(q, kv, ctx_lens, n_sink, window, desc, out, workspace, ws_bytes,
                                 stream=None) -> int:
    return int(LIB.spire_draft_sparse_attention(
        _ptr(q), _ptr(kv), _ptr(ctx_lens), int(n_sink), int(window), _desc_ref(desc),
        _ptr(out), _ptr(workspace), int(ws_bytes), _stream(stream, q)))


def make_append_desc(batch, num_act, num_draft_layers, d_model, num_kv_heads, head_dim, n_sink,
                     window, rope_theta=0.0) -> spire_append_desc:
    return spire_append_desc(int(batch), int(num_act), int(num_draft_layers), int(d_model),
                             int(num_kv_heads), int(head_dim), int(n_sink), int(window),
                             float(rope_theta))


def spire_feedback_append_workspace_bytes(desc: spire_append_desc) -> int:
    return int(LIB.spire_feedback_append_workspace_bytes(_desc_ref(desc)))


def spire_feedback_append(x, mix_w, w_kv, pos, desc, kv, workspace, ws_bytes, stream=None) -> int:
    return int(LIB.spire_feedback_append(
        _ptr(x), _ptr(mix_w), _ptr(w_kv), _ptr(pos), _desc_ref(desc), _ptr(kv), _ptr(workspace),
        int(ws_bytes), _stream(stream, x)))


def spire_magicdec_workspace_bytes(desc: spire_attn_desc, n_sink: int, window: int) -> int:
    return int(LIB.spire_magicdec_workspace_bytes(_desc_ref(desc), int(n_sink), int(window)))


def spire_magicdec_attention(q, k_cache, v_cache, block_table, ctx_lens, n_sink, window,
                             rope_theta, desc, out, workspace, ws_bytes, stream=None) -> int:
    return int(LIB.spire_magicdec_attention(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(ctx_lens), int(n_sink),
        int(window), float(rope_theta), _desc_ref(desc), _ptr(out), _ptr(workspace),
        int(ws_bytes), _stream(stream, q)))


def spire_verify_tokens_workspace_bytes(batch: int, k: int, vocab: int) -> int:
    return int(LIB.spire_verify_tokens_workspace_bytes(int(batch), int(k), int(vocab)))


def spire_verify_tokens(p, q, draft_tokens, u, e, batch, k, vocab, out_tokens, n_accepted,
                        workspace, ws_bytes, stream=None) -> int:
    return int(LIB.spire_verify_tokens(
        _ptr(p), _ptr(q), _ptr(draft_tokens), _ptr(u), _ptr(e), int(batch), int(k), int(vocab),
        _ptr(out_tokens), _ptr(n_accepted), _ptr(workspace), int(ws_bytes), _stream(stream, p)))


def spire_draft_slot(pos: int, n_sink: int, window: int) -> int:
    return int(LIB.spire_draft_slot(int(pos), int(n_sink), int(window)))


def spire_get_device_error(workspace, stream=None) -> int:
    code = ctypes.c_int32(0)
    st = LIB.spire_get_device_error(_ptr(workspace), ctypes.byref(code),
                                    _stream(stream, workspace))
    if st != SPIRE_OK:
        raise SpireError(st, "spire_get_device_error")
    return int(code.value)


def spire_get_cta_times(workspace, ws_bytes, max_ctas=1024, stream=None):
    """Per-CTA (start_ns, end_ns) of the last verify / draft call on `workspace`."""
    buf = (ctypes.c_uint64 * (2 * max_ctas))()
    n = ctypes.c_int32(0)
    st = LIB.spire_get_cta_times(_ptr(workspace), int(ws_bytes), buf, int(max_ctas),
                                 ctypes.byref(n), _stream(stream, workspace))
    if st != SPIRE_OK:
        raise SpireError(st, "spire_get_cta_times")
    m = min(n.value, max_ctas)
    return [(int(buf[2 * i]), int(buf[2 * i + 1])) for i in range(m)]


def spire_stream_read(src, nbytes, stream=None) -> int:
    """One launch that only reads nbytes at src (the floor of a call that
    moves that many bytes); see include/spire.h."""
    return int(LIB.spire_stream_read(_ptr(src), int(nbytes), _stream(stream, src)))


def spire_test_draft_slots(out, n, n_sink, window, stream=None) -> int:
    """Test hook: the device evaluation of the slot helper for p = 0..n-1
    into out (int64); see include/spire.h."""
    return int(LIB.spire_test_draft_slots(_ptr(out), int(n), int(n_sink), int(window),
                                          _stream(stream, out)))


def spire_test_stall_next_call(pair) -> int:
    """Test hook: the next attention call on this thread stalls `pair` (its
    waits run out); see include/spire.h."""
    return int(LIB.spire_test_stall_next_call(int(pair)))


def status_string(status: int) -> str:
    return LIB.spire_status_string(int(status)).decode()


spire_status_string = status_string
