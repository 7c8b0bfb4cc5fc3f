"""spire_feedback_append on the GPU against the fp64 oracle.

Tolerance, from the arithmetic: the kernel multiplies the weights by each
bf16 activation x_l (exact products, fp32 accumulation on the tensor cores,
split over d_model and the splits added in fp32), then mixes the n_act
accumulators with a = softmax(w) in fp32.  Before rounding an output
y = sum_l a_l sum_c W_c x_lc is then off by a few 2^-24 * sqrt(d_model) of
A = sum_l a_l sum_c |W_c| |x_lc| (the rotation mixes the two outputs of a
pair, so for keys A is the pair's sum); A >= sum_c |W_c| |m_c|.  The stored
bf16 entry must be within one bf16 unit of the oracle's exactly rounded value
plus delta * A, delta = 2^-14 (the worst-case chain of d_model = 4096 fp32
additions gives 2^-12 * A, the typical one 2^-18 * A); near a cancellation
(|y| much smaller than A) that can be more than one unit.  At least 98 % of
the entries must be identical, and every slot the call must not write stays
bit-identical.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl

pytestmark = pytest.mark.gpu


def _ulps(a, b):
    def ordered(x):
        x = x.astype(np.int32)
        return np.where(x & 0x8000, -(x & 0x7FFF), x)
    return np.abs(ordered(a) - ordered(b))


DELTA = 2.0 ** -14


def _bits_f64(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _bf16_unit(v):
    """Spacing of bf16 values at |v| (8 significant bits; subnormal floor)."""
    a = np.abs(v)
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    return np.where(a > 0, np.maximum(2.0 ** (e - 7), 2.0 ** -133), 2.0 ** -133)


def _magnitudes(ai, theta, Hkv, D):
    """A = sum_l a_l |W| |x_l| per (layer, sequence, output row), pair-summed
    for rotated keys."""
    w = ai.mix_w.cpu().double().numpy()
    a = np.exp(w - w.max(axis=1, keepdims=True))
    a /= a.sum(axis=1, keepdims=True)                    # [n_dl, n_act]
    X = np.abs(_bits_f64(wl.bf16_bits(ai.x)))            # [n_act, B, C]
    W = np.abs(_bits_f64(wl.bf16_bits(ai.w_kv)))         # [n_dl, F, C]
    A = np.einsum("il,ifc,lbc->ibf", a, W, X)            # [n_dl, B, F]
    n_dl, B, F = A.shape
    A = A.reshape(n_dl, B, 2, Hkv, D)
    if theta > 0:
        k = A[:, :, 0]
        pair = k[..., :D // 2] + k[..., D // 2:]
        A[:, :, 0] = np.concatenate([pair, pair], axis=-1)
    return A


def _run(pos, n_act, n_dl, d_model, Hkv, D, n_sink, window, theta, seed):
    import paper_2504_06419_gb300 as spire
    ai = wl.make_append(pos, n_act, n_dl, d_model, Hkv, D, n_sink, window, seed=seed,
                        device="cuda")
    kv0 = wl.bf16_bits(ai.kv)
    kv = ai.kv.clone()
    desc = spire.make_append_desc(len(pos), n_act, n_dl, d_model, Hkv, D, n_sink, window, theta)
    ws = torch.empty(spire.spire_feedback_append_workspace_bytes(desc), dtype=torch.uint8,
                     device="cuda")
    st = spire.spire_feedback_append(ai.x, ai.mix_w, ai.w_kv, ai.pos, desc, kv, ws, ws.numel())
    assert st == 0, spire.spire_status_string(st)
    err = spire.spire_get_device_error(ws)
    got = wl.bf16_bits(kv)
    want = kv0.copy()
    n_bad = oracle.feedback_append(wl.bf16_bits(ai.x), ai.mix_w.cpu().double().numpy(),
                                   wl.bf16_bits(ai.w_kv), np.asarray(pos, dtype=np.int32), want,
                                   n_sink, window, rope_theta=theta)
    return got, want, kv0, err, n_bad, _magnitudes(ai, theta, Hkv, D)


def _check(got, want, kv0, pos, n_sink, window, A):
    written = np.zeros(got.shape, dtype=bool)
    for b, p in enumerate(pos):
        if p >= 0:
            written[:, b, :, :, oracle.draft_slot(int(p), n_sink, window)] = True
    assert np.array_equal(got[~written], kv0[~written]), "a slot the call must not write changed"
    g, w = _bits_f64(got[written]), _bits_f64(want[written])
    # A per written entry: [n_dl, B, 2, Hkv, D] broadcast over the written slot
    slots = np.moveaxis(written, 4, -1)                      # [n_dl, B, 2, Hkv, D, S]
    a = np.repeat(A[..., None], got.shape[4], axis=-1)[slots]
    bound = _bf16_unit(w) + DELTA * a
    err = np.abs(g - w)
    assert np.all(err <= bound), "worst excess %.3g over the bound" % (err - bound).max()
    u = _ulps(got[written], want[written])
    assert (u == 0).mean() >= 0.98, "only %.4f identical" % (u == 0).mean()
    return u


CASES = [
    # pos, n_act, n_dl, d_model, Hkv, D, n_sink, window, rope_theta
    ("tiny", [0, 1, 9], 2, 1, 64, 1, 64, 2, 5, 0.0),
    ("rope_d128", [0, 3, 4, 20, 100003], 3, 2, 256, 2, 128, 4, 16, 10000.0),
    ("ragged_b37_d64", list(range(0, 370, 10)), 4, 3, 512, 4, 64, 1, 64, 500000.0),
    ("two_token_blocks", list(range(300)), 3, 1, 256, 2, 128, 16, 48, 0.0),
    ("no_sink_ring", [5, 6, 7, 8, 70000, 1 << 30], 1, 1, 128, 1, 128, 0, 8, 10000.0),
    ("draft_2x4096", list(range(7000, 7064)), 3, 2, 4096, 8, 128, 16, 512, 10000.0),
    # 16 activations: 16 tokens per block, one MMA of N = 256
    ("sixteen_activations", list(range(3, 60, 3)), 16, 2, 128, 2, 64, 2, 30, 10000.0),
    # 5 K splits (clusters of 5) over 48-token blocks: 9 or 10 tokens per rank
    ("five_splits_uneven", list(range(0, 504, 7)), 5, 1, 320, 3, 64, 4, 20, 500000.0),
    # 20 row tiles: clusters of 7 asked for, fewer if the GPU cannot hold 20 of them
    ("twenty_tiles", [11, 12, 13, 14, 15, 16, 17, 18], 3, 1, 512, 10, 128, 8, 8, 10000.0),
    # one token, one K block: a single CTA without a split
    ("one_token_one_block", [4], 2, 1, 64, 1, 128, 2, 6, 10000.0),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_append_matches_oracle(case):
    _, pos, n_act, n_dl, d_model, Hkv, D, n_sink, window, theta = case
    got, want, kv0, err, n_bad, A = _run(pos, n_act, n_dl, d_model, Hkv, D, n_sink, window, theta,
                                         seed=len(pos) + d_model)
    assert err == 0 and n_bad == 0
    _check(got, want, kv0, pos, n_sink, window, A)


def test_append_negative_position_is_reported_and_skipped():
    pos = [-1, 2, -5, 7]
    got, want, kv0, err, n_bad, A = _run(pos, 2, 2, 128, 2, 64, 1, 4, 10000.0, seed=9)
    assert n_bad == 2
    assert err == 1          # SPIRE_DEVERR_CTX_LEN
    assert np.array_equal(got[:, 0], kv0[:, 0]) and np.array_equal(got[:, 2], kv0[:, 2])
    _check(got, want, kv0, pos, 1, 4, A)


def test_append_large_grid_shares_one_error_word():
    """16 layers x 4 row-tile pairs x 9 token blocks: more than 512 CTAs, so
    they share one error word (cleared by its own launch); a negative
    position is still reported and skipped."""
    pos = list(range(720))
    pos[500] = -3
    got, want, kv0, err, n_bad, A = _run(pos, 3, 16, 64, 4, 128, 4, 60, 10000.0, seed=77)
    assert n_bad == 1 and err == 1
    assert np.array_equal(got[:, 500], kv0[:, 500])
    _check(got, want, kv0, pos, 4, 60, A)


def test_append_is_deterministic():
    a = _run(list(range(40)), 3, 2, 1024, 4, 128, 4, 28, 10000.0, seed=5)[0]
    b = _run(list(range(40)), 3, 2, 1024, 4, 128, 4, 28, 10000.0, seed=5)[0]
    assert np.array_equal(a, b)


def test_append_then_draft_attention():
    """One draft step end to end: append entry t of every sequence, then
    attend with t + 1 visible entries (the new entry included); compared with
    the oracle's append followed by its draft attention."""
    import paper_2504_06419_gb300 as spire
    from parity import ROW_REL_REROUNDED, assert_close
    t = np.array([0, 5, 20, 47, 300], dtype=np.int32)
    n_sink, window, Hq, Hkv, D = 4, 16, 8, 2, 128
    ai = wl.make_append(t, 3, 1, 256, Hkv, D, n_sink, window, seed=31, device="cuda")
    want_kv = wl.bf16_bits(ai.kv)
    oracle.feedback_append(wl.bf16_bits(ai.x), ai.mix_w.cpu().double().numpy(),
                           wl.bf16_bits(ai.w_kv), t, want_kv, n_sink, window, rope_theta=10000.0)
    spire.feedback_append(ai.x, ai.mix_w, ai.w_kv, ai.pos, ai.kv, n_sink, window, 10000.0)
    q = wl.make_draft(t + 1, Hq, Hkv, D, n_sink, window, seed=32, device="cuda").q
    ctx = torch.from_numpy(t + 1).cuda()
    out = spire.draft_attention(q, ai.kv[0], ctx, n_sink, window)
    # the oracle attends over its own appended cache
    ref, n_bad = oracle.draft_ring(wl.bf16_bits(q), want_kv[0], t + 1, n_sink, window)
    assert n_bad == 0
    assert_close(out.cpu().double().numpy(), ref, "append + draft", row_rel=ROW_REL_REROUNDED)
