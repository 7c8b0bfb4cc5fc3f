"""The slot helper the feedback append uses to place a new memory entry in the
bounded draft cache (Section 3.1: sinks kept, a sliding window over the rest),
evaluated on the device through spire_test_draft_slots, against the oracle's
independent slot function position by position."""
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("n_sink, window, n", [(4, 64, 10 ** 6), (16, 512, 10 ** 6),
                                               (0, 1, 10 ** 5), (1, 64, 10 ** 5),
                                               (7, 13, 10 ** 5), (32, 2048, 10 ** 5)])
def test_device_slot_matches_oracle(n_sink, window, n):
    import paper_2504_06419_gb300 as spire
    out = torch.full((n,), -7, dtype=torch.int64, device="cuda")
    assert spire.spire_test_draft_slots(out, n, n_sink, window) == 0
    got = out.cpu().tolist()
    lib = oracle.load()
    bad = [p for p in range(n) if got[p] != oracle.draft_slot(p, n_sink, window, lib=lib)]
    assert not bad, "first mismatch at p = %d" % bad[0]
