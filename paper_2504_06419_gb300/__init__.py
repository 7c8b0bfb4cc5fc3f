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

The functions below allocate outputs and workspaces with PyTorch and call the
C ABI; all computation runs in the library's kernels.
"""
from __future__ import annotations

import torch

from . import _lib
from ._lib import (SpireError, make_desc, spire_draft_slot, spire_draft_sparse_attention,
                   spire_draft_workspace_bytes, spire_get_device_error, spire_status_string,
                   spire_verify_attention, spire_verify_attention_noalloc,
                   spire_verify_workspace_bytes)

__all__ = [
    "SpireError", "make_desc", "spire_verify_attention", "spire_verify_attention_noalloc",
    "spire_draft_sparse_attention",
    "spire_verify_workspace_bytes", "spire_draft_workspace_bytes", "spire_draft_slot",
    "spire_get_device_error", "spire_status_string", "verify_attention", "draft_attention",
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
