"""libspire: GB300-native attention of one SPIRe speculation round.

SPIRe (Neelam et al., arXiv 2504.06419) is a draft model for speculative
decoding at large batch and long context, where each round is k draft passes
plus one verification pass over k+1 tokens (Section 2) and the dominant cost
is streaming KV caches (Section 3.1).  This package wraps the CUDA library
libspire (include/spire.h):

  spire_verify_attention         verification attention over paged, ragged
                                 bf16 KV with GQA, causal within the block
  spire_draft_sparse_attention   draft sink + sliding-window attention over a
                                 bounded feedback-memory cache (Section 3.3)
  spire_feedback_append          the draft step's cache update: per-layer
                                 memory vector, K/V projection, bounded-cache
                                 slot (Section 3.3)
  spire_magicdec_attention       the MagicDec baseline's draft attention over
                                 the target's own cache (Section 3.1 footnote)
  spire_verify_tokens            token verification: modified rejection
                                 sampling of the round's drafts (Section 1)

The functions below allocate outputs and workspaces with PyTorch and call the
C ABI; all computation runs in the library's kernels.
"""
from __future__ import annotations

import torch

from . import _lib
from ._lib import (SpireError, make_append_desc, make_desc, spire_draft_slot,
                   spire_draft_sparse_attention, spire_draft_workspace_bytes,
                   spire_feedback_append, spire_feedback_append_workspace_bytes,
                   spire_get_cta_times, spire_get_device_error, spire_magicdec_attention,
                   spire_stream_read, spire_test_draft_slots, spire_test_stall_next_call,
                   spire_magicdec_workspace_bytes, spire_status_string, spire_verify_attention,
                   spire_verify_attention_noalloc, spire_verify_tokens,
                   spire_verify_tokens_workspace_bytes, spire_verify_workspace_bytes)

__all__ = [
    "SpireError", "make_desc", "make_append_desc", "spire_verify_attention",
    "spire_verify_attention_noalloc", "spire_draft_sparse_attention", "spire_feedback_append",
    "spire_feedback_append_workspace_bytes", "feedback_append", "spire_verify_tokens",
    "spire_verify_tokens_workspace_bytes", "verify_tokens", "spire_magicdec_attention",
    "spire_magicdec_workspace_bytes", "magicdec_attention",
    "spire_verify_workspace_bytes", "spire_draft_workspace_bytes", "spire_draft_slot",
    "spire_get_device_error", "spire_get_cta_times", "spire_stream_read", "spire_test_draft_slots",
    "spire_test_stall_next_call", "spire_status_string",
    "verify_attention",
    "draft_attention",
    "verify_desc", "draft_desc",
]


def verify_desc(q, k_cache, block_table, softmax_scale=1.0):
    B, _, Hq, D = q.shape
    return make_desc(B, Hq, k_cache.shape[1], D, k_cache.shape[2], block_table.shape[1],
                     k_cache.shape[0], softmax_scale)


def draft_desc(q, kv, softmax_scale=1.0):
    B, Hq, D = q.shape
    return make_desc(B, Hq, kv.shape[2], D, 64, 0, 0, softmax_scale)


def verify_attention(q, k_cache, v_cache, block_table, ctx_lens, k, softmax_scale=1.0,
                     out=None, workspace=None, stream=None):
    """Verification attention; returns out fp32 [B, k+1, Hq, D]."""
    desc = verify_desc(q, k_cache, block_table, softmax_scale)
    ws_bytes = spire_verify_workspace_bytes(desc, k)
    if out is None:
        out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
    if workspace is None:
        workspace = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=q.device)
    st = spire_verify_attention(q, k_cache, v_cache, block_table, ctx_lens, k, desc, out,
                                workspace, workspace.numel(), stream)
    if st != 0:
        raise SpireError(st, "spire_verify_attention")
    return out


def draft_attention(q, kv, ctx_lens, n_sink, window, softmax_scale=1.0, out=None,
                    workspace=None, stream=None):
    """Draft sink + window attention; returns out fp32 [B, Hq, D]."""
    desc = draft_desc(q, kv, softmax_scale)
    ws_bytes = spire_draft_workspace_bytes(desc, n_sink, window)
    if out is None:
        out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
    if workspace is None:
        workspace = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=q.device)
    st = spire_draft_sparse_attention(q, kv, ctx_lens, n_sink, window, desc, out, workspace,
                                      workspace.numel(), stream)
    if st != 0:
        raise SpireError(st, "spire_draft_sparse_attention")
    return out


def feedback_append(x, mix_w, w_kv, pos, kv, n_sink, window, rope_theta=0.0, workspace=None,
                    stream=None):
    """Write one feedback-memory entry per sequence into every draft layer's
    bounded cache kv [n_dl, B, 2, Hkv, n_sink + window, D] (bf16, in place).

    x [n_act, B, d_model] bf16, mix_w [n_dl, n_act] fp32, w_kv [n_dl, 2*Hkv*D,
    d_model] bf16, pos [B] int32 (device).  Returns kv."""
    n_act, B, d_model = x.shape
    n_dl, Hkv, D = kv.shape[0], kv.shape[3], kv.shape[5]
    desc = make_append_desc(B, n_act, n_dl, d_model, Hkv, D, n_sink, window, rope_theta)
    ws_bytes = spire_feedback_append_workspace_bytes(desc)
    if ws_bytes == 0:
        raise SpireError(1, "spire_feedback_append_workspace_bytes")
    if workspace is None:
        workspace = torch.empty(ws_bytes, dtype=torch.uint8, device=x.device)
    st = spire_feedback_append(x, mix_w, w_kv, pos, desc, kv, workspace, workspace.numel(),
                               stream)
    if st != 0:
        raise SpireError(st, "spire_feedback_append")
    return kv


def verify_tokens(p, q, draft_tokens, u, e, workspace=None, stream=None):
    """Token verification of one round per sequence (modified rejection
    sampling).  p fp32 [B, k+1, V], q fp32 [B, k, V], draft_tokens int32 [B, k],
    u fp32 [B, k], e fp32 [B, V] (Exp(1) variates), all on the GPU.
    Returns (out_tokens int32 [B, k+1], n_accepted int32 [B])."""
    B, kp1, V = p.shape
    k = kp1 - 1
    ws_bytes = spire_verify_tokens_workspace_bytes(B, k, V)
    if ws_bytes == 0:
        raise SpireError(1, "spire_verify_tokens_workspace_bytes")
    if workspace is None:
        workspace = torch.empty(ws_bytes, dtype=torch.uint8, device=p.device)
    out = torch.empty((B, kp1), dtype=torch.int32, device=p.device)
    n_acc = torch.empty((B,), dtype=torch.int32, device=p.device)
    st = spire_verify_tokens(p, q if k > 0 else None, draft_tokens if k > 0 else None,
                             u if k > 0 else None, e, B, k, V, out, n_acc, workspace,
                             workspace.numel(), stream)
    if st != 0:
        raise SpireError(st, "spire_verify_tokens")
    return out, n_acc


def magicdec_attention(q, k_cache, v_cache, block_table, ctx_lens, n_sink, window, rope_theta,
                       softmax_scale=1.0, out=None, workspace=None, stream=None):
    """MagicDec draft attention over the target's paged cache; q bf16
    [B, Hq, D] (not rotated).  Returns out fp32 [B, Hq, D]."""
    B, Hq, D = q.shape
    desc = make_desc(B, Hq, k_cache.shape[1], D, k_cache.shape[2], block_table.shape[1],
                     k_cache.shape[0], softmax_scale)
    ws_bytes = spire_magicdec_workspace_bytes(desc, n_sink, window)
    if out is None:
        out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
    if workspace is None:
        workspace = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=q.device)
    st = spire_magicdec_attention(q, k_cache, v_cache, block_table, ctx_lens, n_sink, window,
                                  rope_theta, desc, out, workspace, workspace.numel(), stream)
    if st != 0:
        raise SpireError(st, "spire_magicdec_attention")
    return out
