"""spire_verify_tokens on the GPU against the oracle.

Both sides take every decision in binary32 (the product u * q, the residual
p - q, the quotient w / E) on the same inputs, so the emitted tokens and the
accepted counts must be identical, integer for integer.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl

pytestmark = pytest.mark.gpu


def _compare(ti, expect_err=0):
    import paper_2504_06419_gb300 as spire
    B, kp1, V = ti.p.shape
    ws = torch.empty(spire.spire_verify_tokens_workspace_bytes(B, kp1 - 1, V),
                     dtype=torch.uint8, device="cuda")
    out, n_acc = spire.verify_tokens(ti.p, ti.q, ti.x, ti.u, ti.e, workspace=ws)
    err = spire.spire_get_device_error(ws)
    ro, rn, n_bad = oracle.verify_tokens(ti.p.cpu().numpy(), ti.q.cpu().numpy(),
                                         ti.x.cpu().numpy(), ti.u.cpu().numpy(),
                                         ti.e.cpu().numpy())
    assert np.array_equal(n_acc.cpu().numpy(), rn)
    assert np.array_equal(out.cpu().numpy(), ro)
    assert (err != 0) == (n_bad != 0) and (err & ~expect_err) == 0, (err, n_bad)
    return out.cpu().numpy(), rn


CASES = [
    # batch, k, vocab
    (1, 0, 7),            # plain sampling, scalar loads
    (3, 1, 1001),         # scalar loads (V % 4 != 0), one chunk
    (64, 4, 32000),       # bulk copies: 8 units of 4096 per sequence, a 3328-entry tail
    (17, 8, 8193),        # scalar loads, a chunk of one entry
    (2, 0, 4096),         # plain sampling on the bulk-copy path: one unit, no q row
    (5, 3, 100),          # one unit of 100 entries (a 400-byte copy)
    (64, 4, 128256),      # a Llama 3 sized vocabulary
]


@pytest.mark.parametrize("case", CASES, ids=["b%d_k%d_v%d" % c for c in CASES])
def test_tokens_match_oracle(case):
    B, k, V = case
    ti = wl.make_tokens(B, k, V, seed=B * 31 + k * 7 + V, device="cuda")
    out, n_acc = _compare(ti)
    if k > 0 and B >= 16:
        # a realistic mix: some rounds stop early, some accept drafts
        assert 0 < n_acc.mean() < k


def test_tokens_identical_models_accept_everything():
    ti = wl.make_tokens(32, 4, 4096, seed=5, device="cuda")
    ti.q = ti.p[:, :4].contiguous()
    out, n_acc = _compare(ti)
    assert np.all(n_acc == 4)


def test_tokens_disjoint_draft_rejects_at_once():
    """A draft distribution with no mass where the target has it: the first
    draft is always rejected and the residual is the target row itself."""
    ti = wl.make_tokens(8, 3, 64, seed=6, device="cuda")
    p = torch.zeros_like(ti.p)
    p[..., :32] = 1.0 / 32
    q = torch.zeros_like(ti.q)
    q[..., 32:] = 1.0 / 32
    ti.p, ti.q = p, q
    ti.x = torch.full_like(ti.x, 40)
    out, n_acc = _compare(ti)
    assert np.all(n_acc == 0) and np.all(out[:, 0] < 32)


def test_tokens_invalid_inputs_are_reported():
    ti = wl.make_tokens(4, 2, 1024, seed=7, device="cuda")
    ti.x[1, 0] = 5000          # out of range: rejected at once
    ti.e[2, :] = 0.0           # no valid E: no draw
    ti.e[3, 10] = -1.0         # one skipped E
    _compare(ti, expect_err=1 | 8)


def test_tokens_repeatable():
    import paper_2504_06419_gb300 as spire
    ti = wl.make_tokens(16, 4, 50000, seed=8, device="cuda")
    a = spire.verify_tokens(ti.p, ti.q, ti.x, ti.u, ti.e)[0].cpu()
    b = spire.verify_tokens(ti.p, ti.q, ti.x, ti.u, ti.e)[0].cpu()
    assert torch.equal(a, b)
