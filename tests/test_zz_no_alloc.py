"""spire_verify_attention_noalloc: the entry point for callers that cannot
allocate device memory when they call us (a serving engine whose free GPU
memory all went to its KV-cache pool, or a plugin host that only passes
input and output pointers).  Its scratch is a fixed 32 MiB array inside the
library.  This file is collected last so that a failure here leaves every
other test already run."""
import pytest
import torch

import parity
import workloads as wl

pytestmark = pytest.mark.gpu
DEV = "cuda"


def test_noalloc_matches_workspace_entry_point_and_oracle_on_two_calls():
    import paper_2504_06419_gb300 as spire
    L, k = [700, 64, 129, 2000, 5], 4
    vi = wl.make_verify(L, k, 32, 8, 128, seed=77, device=DEV, poison=True, spare_pages=2)
    ref_ws = parity.gpu_verify(spire, vi).cpu().numpy()
    ref, n_bad = parity.oracle_verify(vi)
    assert n_bad == 0
    desc = spire.verify_desc(vi.q, vi.k_cache, vi.block_table)
    for call in range(2):   # the shared scratch keeps the last call's contents
        out = torch.full(vi.q.shape, float("nan"), dtype=torch.float32, device=DEV)
        st = spire.spire_verify_attention_noalloc(vi.q, vi.k_cache, vi.v_cache, vi.block_table,
                                                  vi.ctx_lens, k, desc, out)
        assert st == 0, spire.spire_status_string(st)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        rel, mx = parity.errors(got, ref_ws)
        assert rel <= parity.REL_L2 and mx <= parity.MAX_ABS, (call, rel, mx)
        parity.assert_close(got, ref, "noalloc call %d against the oracle" % call)


def test_noalloc_rejects_shapes_beyond_its_scratch():
    import paper_2504_06419_gb300 as spire
    # 64 query heads on one KV head, k = 1: 128 rows per KV head need ~68 MB
    desc = spire.make_desc(4, 64, 1, 128, 64, 4, 16)
    assert spire.spire_verify_workspace_bytes(desc, 1) > (32 << 20)
    dummy = torch.zeros(16, dtype=torch.float32, device=DEV)
    st = spire.spire_verify_attention_noalloc(dummy, dummy, dummy, dummy, dummy, 1, desc, dummy)
    assert st == 3   # SPIRE_ERR_WORKSPACE


def test_noalloc_reports_other_cases_as_the_workspace_entry_point():
    """Beyond-scratch shapes that the workspace entry point itself answers
    without a workspace get its status, not SPIRE_ERR_WORKSPACE."""
    import paper_2504_06419_gb300 as spire
    dummy = torch.zeros(16, dtype=torch.float32, device=DEV)
    empty = spire.make_desc(0, 64, 1, 128, 64, 4, 16)          # B = 0, 128 rows per KV head
    assert spire.spire_verify_workspace_bytes(empty, 1) > (32 << 20)
    assert spire.spire_verify_attention_noalloc(None, None, None, None, None, 1, empty,
                                                None) == 0
    page32 = spire.make_desc(4, 64, 1, 128, 32, 4, 16)         # page size 32: unsupported
    assert spire.spire_verify_attention_noalloc(dummy, dummy, dummy, dummy, dummy, 1, page32,
                                                dummy) == 2
