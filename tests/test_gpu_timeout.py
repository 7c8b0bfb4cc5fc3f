"""The failure path of the attention kernels' bounded waits, run on purpose
without faulting or hanging the GPU: spire_test_stall_next_call makes the
producer of the CTA that reaches one pair issue no loads from it on (no copy
of it is ever in flight), so the consumers' bounded waits for that pair run
out (2 s).  The call must return, the device error word
must report SPIRE_DEVERR_TIMEOUT, and the next normal call on the same
workspace must be correct (the context stays usable, tensor memory was
freed)."""
import pytest
import torch

import parity
import workloads as wl

pytestmark = pytest.mark.gpu
DEV = "cuda"
TIMEOUT = 4   # SPIRE_DEVERR_TIMEOUT


@pytest.mark.parametrize("kind", ["verify_tc", "verify_onecopy72", "verify_onecopy96", "draft"])
def test_waits_run_out_then_the_next_call_is_correct(kind):
    import paper_2504_06419_gb300 as spire
    if kind == "draft":
        inp = wl.make_draft([900, 40, 600, 1500], 32, 8, 128, 16, 512, seed=91, device=DEV)
        desc = spire.draft_desc(inp.q, inp.kv)
        ws = torch.empty(spire.spire_draft_workspace_bytes(desc, 16, 512), dtype=torch.uint8,
                         device=DEV)

        def call():
            out = torch.empty(inp.q.shape, dtype=torch.float32, device=DEV)
            st = spire.spire_draft_sparse_attention(inp.q, inp.kv, inp.ctx_lens, 16, 512, desc,
                                                    out, ws, ws.numel())
            assert st == 0
            return out
        ref, n_bad = parity.oracle_draft(inp)
    else:
        # 20 rows per KV head (four query copies), 72 and 96 (one copy)
        hq, hkv, k = {"verify_tc": (32, 8, 4), "verify_onecopy72": (64, 8, 8),
                      "verify_onecopy96": (64, 8, 11)}[kind]
        inp = wl.make_verify([3000, 700, 64 * 9 + 5, 2500], k, hq, hkv, 128, seed=92, device=DEV)
        desc = spire.verify_desc(inp.q, inp.k_cache, inp.block_table)
        ws = torch.empty(spire.spire_verify_workspace_bytes(desc, k), dtype=torch.uint8,
                         device=DEV)

        def call():
            out = torch.empty(inp.q.shape, dtype=torch.float32, device=DEV)
            st = spire.spire_verify_attention(inp.q, inp.k_cache, inp.v_cache, inp.block_table,
                                              inp.ctx_lens, k, desc, out, ws, ws.numel())
            assert st == 0
            return out
        ref, n_bad = parity.oracle_verify(inp)
    assert n_bad == 0
    # pair 9 = (sequence 1, KV head 1): the stall leaves its CTA's waits to run out
    assert spire.spire_test_stall_next_call(9) == 0
    call()
    torch.cuda.synchronize()
    assert spire.spire_get_device_error(ws) & TIMEOUT
    # the hook applied to that one call only: the next call on the same workspace
    # is complete and correct
    got = call()
    torch.cuda.synchronize()
    assert spire.spire_get_device_error(ws) == 0
    parity.assert_close(got.cpu().numpy(), ref, "%s after a timed-out call" % kind)
