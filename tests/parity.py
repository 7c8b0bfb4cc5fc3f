"""Helpers shared by the GPU parity tests: run the CUDA path through the C ABI,
run the oracle on the very same inputs, and compare.

Tolerance (per call, over the whole compared output): max |gpu - oracle| <= 1e-2
and ||gpu - oracle||_2 / ||oracle||_2 <= 1e-3.  Also per output row (one
(sequence, block row, query head) vector of head_dim values): the row's
relative L2 error <= 1e-3, so that a wrong row of a long sequence, whose
outputs are small (|o| ~ 1/sqrt(L) for flat logits), cannot hide behind the
larger outputs of short sequences in the whole-tensor norm.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import workloads as wl

MAX_ABS = 1e-2
REL_L2 = 1e-3
# Per-row bound where an attention operand is itself computed and rounded to
# bf16 before the attention (MagicDec's keys and query turned to cache
# positions; a draft step over entries the feedback append just wrote).  The
# kernel computes such a value in fp32 and the oracle in fp64, so a value that
# lies next to a bf16 rounding boundary can round to the neighbouring bf16
# number on one side: one element moves by one bf16 unit (2^-8 of it), one
# score by up to |q_d| 2^-8 |k_d| (about 1e-2 for the largest N(0,1) entries),
# and a row that a few keys dominate by up to about that much, relatively.
# Such rows are held to 1e-2; the whole-tensor gates above stay as they are.
ROW_REL_REROUNDED = 1e-2


def errors(got: np.ndarray, ref: np.ndarray):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape
    if got.size == 0:
        return 0.0, 0.0
    diff = got - ref
    rel = float(np.linalg.norm(diff) / max(np.linalg.norm(ref), 1e-300))
    return rel, float(np.abs(diff).max())


def row_errors(got: np.ndarray, ref: np.ndarray):
    """Relative L2 error of every row (the last axis) and the worst row.
    Returns (rel per row, index tuple of the worst row, its rel).  A row whose
    reference is exactly zero counts its absolute L2 error instead."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape
    if got.size == 0:
        return np.zeros(got.shape[:-1]), (), 0.0
    num = np.linalg.norm(got - ref, axis=-1)
    den = np.linalg.norm(ref, axis=-1)
    rel = np.where(den > 0, num / np.where(den > 0, den, 1.0), num)
    worst = np.unravel_index(int(np.argmax(rel)), rel.shape)
    return rel, tuple(int(i) for i in worst), float(rel[worst])


def assert_close(got, ref, what="", row_rel=REL_L2):
    """Whole-tensor gates (rel L2 <= 1e-3, max abs <= 1e-2) and the per-row
    gate row_rel (1e-3; ROW_REL_REROUNDED where operands were re-rounded)."""
    assert np.all(np.isfinite(got)), "%s: non-finite GPU output" % what
    rel, mx = errors(got, ref)
    assert rel <= REL_L2 and mx <= MAX_ABS, "%s: rel_l2=%.3g max_abs=%.3g" % (what, rel, mx)
    _, worst, wrel = row_errors(got, ref)
    assert wrel <= row_rel, "%s: row %s has rel_l2=%.3g (whole tensor %.3g)" % (
        what, worst, wrel, rel)
    return rel, mx


def gpu_verify(spire, vi: wl.VerifyInputs):
    out = spire.verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens, vi.k,
                                 softmax_scale=vi.scale)
    torch.cuda.synchronize()
    return out


def gpu_draft(spire, di: wl.DraftInputs):
    out = spire.draft_attention(di.q, di.kv, di.ctx_lens, di.n_sink, di.window,
                                softmax_scale=di.scale)
    torch.cuda.synchronize()
    return out


def oracle_verify(vi: wl.VerifyInputs, unit_mask=None):
    ref, n_bad = oracle.verify(wl.bf16_bits(vi.q), wl.bf16_bits(vi.k_cache),
                               wl.bf16_bits(vi.v_cache), vi.block_table.cpu().numpy(),
                               vi.ctx_lens.cpu().numpy(), vi.k, scale=vi.scale,
                               unit_mask=unit_mask)
    return ref, n_bad


def oracle_draft(di: wl.DraftInputs, unit_mask=None):
    return oracle.draft_ring(wl.bf16_bits(di.q), wl.bf16_bits(di.kv), di.ctx_lens.cpu().numpy(),
                             di.n_sink, di.window, scale=di.scale, unit_mask=unit_mask)


def compact_verify(vi: wl.VerifyInputs, seqs) -> wl.VerifyInputs:
    """The inputs of a subset of sequences, with only their pages (gathered on
    the device) -- lets the oracle check a few sequences of a huge cache."""
    seqs = torch.as_tensor(list(seqs), dtype=torch.long, device=vi.q.device)
    L = vi.ctx_lens[seqs].long()
    pages = (L + 63) // 64
    mp = int(pages.max())
    bt = torch.full((len(seqs), mp), -1, dtype=torch.int32, device=vi.q.device)
    src = []
    off = 0
    for j in range(len(seqs)):
        p = int(pages[j])
        src.append(vi.block_table[seqs[j], :p].long())
        bt[j, :p] = torch.arange(off, off + p, dtype=torch.int32, device=vi.q.device)
        off += p
    src = torch.cat(src)
    return wl.VerifyInputs(q=vi.q[seqs].contiguous(), k_cache=vi.k_cache[src].contiguous(),
                           v_cache=vi.v_cache[src].contiguous(), block_table=bt,
                           ctx_lens=vi.ctx_lens[seqs].contiguous(), k=vi.k, scale=vi.scale)
