"""spire_magicdec_attention on the GPU against the fp64 oracle, within the
attention tolerance (max |gpu - oracle| <= 1e-2, relative L2 <= 1e-3)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from parity import ROW_REL_REROUNDED, assert_close

pytestmark = pytest.mark.gpu


def _run(L, Hq, Hkv, D, n_sink, window, theta, seed, edit=None):
    import paper_2504_06419_gb300 as spire
    vi = wl.make_verify(L, 0, Hq, Hkv, D, seed=seed, device="cuda", poison=True)
    q = vi.q[:, 0].contiguous()
    bt, ctx = vi.block_table, vi.ctx_lens
    if edit is not None:
        bt, ctx = edit(bt.clone(), ctx.clone())
    desc = spire.make_desc(len(L), Hq, Hkv, D, 64, bt.shape[1], vi.k_cache.shape[0])
    ws = torch.empty(spire.spire_magicdec_workspace_bytes(desc, n_sink, window),
                     dtype=torch.uint8, device="cuda")
    out = spire.magicdec_attention(q, vi.k_cache, vi.v_cache, bt, ctx, n_sink, window, theta,
                                   workspace=ws)
    err = spire.spire_get_device_error(ws)
    ref, n_bad = oracle.magicdec(wl.bf16_bits(q), wl.bf16_bits(vi.k_cache),
                                 wl.bf16_bits(vi.v_cache), bt.cpu().numpy(), ctx.cpu().numpy(),
                                 n_sink, window, theta)
    return out.cpu().double().numpy(), ref, err, n_bad


CASES = [
    # lengths, Hq, Hkv, D, n_sink, window, theta
    ("paper_sink1_win64", [1, 3, 65, 200, 1000], 4, 1, 64, 1, 64, 10000.0),
    ("gqa_d128", [8192] * 8, 32, 8, 128, 1, 64, 500000.0),
    ("ragged_sink4_win128", [5, 63, 64, 129, 5000, 70000], 8, 2, 128, 4, 128, 10000.0),
    ("window_covers_context", [10, 100, 200], 4, 2, 64, 4, 256, 10000.0),
    ("no_rotation", [300, 301, 302], 8, 8, 64, 2, 30, 0.0),
    ("g8_d128", [4000, 77, 9000], 64, 8, 128, 1, 64, 10000.0),
    ("g3_two_chunks", [500, 1500, 90], 6, 2, 128, 2, 100, 10000.0),
    # 64 query heads per KV head: the draft attention runs on the tcgen05 kernel
    ("g64_tcgen05", [100, 3000, 40], 64, 1, 64, 1, 64, 10000.0),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_magicdec_matches_oracle(case):
    _, L, Hq, Hkv, D, n_sink, window, theta = case
    got, ref, err, n_bad = _run(np.array(L), Hq, Hkv, D, n_sink, window, theta, seed=len(L) + D)
    assert n_bad == 0 and err == 0
    assert_close(got, ref, "magicdec", row_rel=ROW_REL_REROUNDED)


def test_magicdec_invalid_sequences_are_nan():
    def edit(bt, ctx):
        ctx[0] = 0                       # no entry visible
        ctx[1] = bt.shape[1] * 64 + 5    # beyond the block table
        bt[2, 0] = -3                    # a sink page outside the cache
        return bt, ctx
    L = np.array([100, 100, 100, 100])
    got, ref, err, n_bad = _run(L, 4, 1, 64, 1, 16, 10000.0, seed=3, edit=edit)
    assert n_bad == 3 and err == 1       # SPIRE_DEVERR_CTX_LEN
    assert np.all(np.isnan(got[:3])) and np.all(np.isfinite(got[3]))
    assert_close(got[3:], ref[3:], "magicdec valid row", row_rel=ROW_REL_REROUNDED)
