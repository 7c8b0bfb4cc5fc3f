"""Helpers shared by the GPU parity tests: run the CUDA path through the C ABI,
run the oracle on the very same inputs, and compare.

Tolerance (per call, over the whole compared output): max |gpu - oracle| <= 1e-2
and ||gpu - oracle||_2 / ||oracle||_2 <= 1e-3.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import workloads as wl

MAX_ABS = 1e-2
REL_L2 = 1e-3


def errors(got: np.ndarray, ref: np.ndarray):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape
    if got.size == 0:
        return 0.0, 0.0
    diff = got - ref
    rel = float(np.linalg.norm(diff) / max(np.linalg.norm(ref), 1e-300))
    return rel, float(np.abs(diff).max())


def assert_close(got, ref, what=""):
    assert np.all(np.isfinite(got)), "%s: non-finite GPU output" % what
    rel, mx = errors(got, ref)
    assert rel <= REL_L2 and mx <= MAX_ABS, "%s: rel_l2=%.3g max_abs=%.3g" % (what, rel, mx)
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
