"""Full-size parity on the benchmark workloads.

Each call runs at full size in the same launch configuration the benchmark
times.  The oracle then recomputes every sequence of the batch (the 26 GB
large-batch verify cache 32 sequences at a time, each group's pages gathered
on the device first); every head and block row must match within max-abs
1e-2 and relative L2 1e-3, over the tensor and row by row.
"""
import pytest
import torch

import parity
import workloads as wl

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def spire():
    import paper_2504_06419_gb300 as m
    return m


@pytest.mark.parametrize("name", ["tiny", "uniform8k", "ragged", "big"])
def test_verify_full_config(spire, name):
    cfg = wl.CONFIGS[name]
    L = wl.sample_ctx_lens(cfg)
    vi = wl.make_verify(L, cfg.k, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim,
                        seed=cfg.seed, device=DEV, shuffle=cfg.paged_shuffle)
    desc = spire.verify_desc(vi.q, vi.k_cache, vi.block_table)
    ws = torch.empty(spire.spire_verify_workspace_bytes(desc, cfg.k), dtype=torch.uint8,
                     device=DEV)
    out = spire.verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens,
                                 cfg.k, workspace=ws)
    assert spire.spire_get_device_error(ws) == 0
    del ws
    if name == "big":           # the whole batch, 32 sequences at a time
        for g0 in range(0, len(L), 32):
            seqs = list(range(g0, min(len(L), g0 + 32)))
            sub = parity.compact_verify(vi, seqs)
            got = out[g0:g0 + len(seqs)].cpu().numpy()
            ref, n_bad = parity.oracle_verify(sub)
            assert n_bad == 0
            parity.assert_close(got, ref, "verify big (sequences %d..%d)" % (seqs[0], seqs[-1]))
            del sub
    else:                       # the whole batch at once
        ref, n_bad = parity.oracle_verify(vi)
        assert n_bad == 0
        parity.assert_close(out.cpu().numpy(), ref, "verify %s (all %d sequences)" % (name, len(L)))
    del vi, out
    torch.cuda.empty_cache()


DRAFT_RUNS = [("tiny", None), ("uniform8k", None), ("ragged", None), ("big", None),
              ("draft_sweep", 256), ("draft_sweep", 1024), ("draft_sweep", 4096)]


@pytest.mark.parametrize("name,window", DRAFT_RUNS, ids=["%s-%s" % r for r in DRAFT_RUNS])
def test_draft_full_config(spire, name, window):
    cfg = wl.CONFIGS[name]
    w = window or cfg.window
    L = wl.sample_ctx_lens(cfg)
    for j in (0, cfg.k - 1):
        t = wl.draft_ctx_for_step(L, cfg.k, j)
        di = wl.make_draft(t, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim, cfg.n_sink, w,
                           seed=cfg.seed + 17 * (j + 1), device=DEV)
        out = parity.gpu_draft(spire, di)
        ref, n_bad = parity.oracle_draft(di)       # every sequence of the batch
        assert n_bad == 0
        parity.assert_close(out.cpu().numpy(), ref, "draft %s w=%d step %d (all %d sequences)"
                            % (name, w, j, len(t)))
        del di, out
    torch.cuda.empty_cache()


def test_magicdec_full_config(spire):
    """The MagicDec draft step as the benchmark runs it: sink 1 + window 64
    over the uniform 8K target cache (B = 64, 32/8 heads, D = 128, shuffled
    pages), keys and query turned to cache positions (theta 1e4); the oracle
    recomputes every sequence."""
    import oracle
    cfg = wl.CONFIGS["uniform8k"]
    L = wl.sample_ctx_lens(cfg)
    vi = wl.make_verify(L, cfg.k, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim,
                        seed=cfg.seed, device=DEV, shuffle=cfg.paged_shuffle)
    t = wl.draft_ctx_for_step(L, cfg.k, 0)
    q = vi.q[:, 0].contiguous()
    ctx = torch.as_tensor(t, dtype=torch.int32, device=DEV)
    out = spire.magicdec_attention(q, vi.k_cache, vi.v_cache, vi.block_table, ctx, 1, 64, 1e4)
    torch.cuda.synchronize()
    ref, n_bad = oracle.magicdec(wl.bf16_bits(q), wl.bf16_bits(vi.k_cache),
                                 wl.bf16_bits(vi.v_cache), vi.block_table.cpu().numpy(),
                                 ctx.cpu().numpy(), 1, 64, 1e4)
    assert n_bad == 0
    parity.assert_close(out.cpu().numpy(), ref, "magicdec uniform8k (all %d sequences)" % len(t),
                        row_rel=parity.ROW_REL_REROUNDED)
    del vi, out
    torch.cuda.empty_cache()
