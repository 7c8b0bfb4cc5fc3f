"""Pins of the fp64 oracle against facts the paper's definitions and plain
mathematics fix -- not against the oracle itself.

Every pin takes the ctypes handle of an oracle build, so the same pins run on
the real oracle (test_oracle_pins.py) and on deliberately broken copies of it
(test_oracle_mutants.py), which shows each plausible mistake trips a pin.

What fixes each expected value:
  * closed forms: with q = 0 every visible key has the same weight, so the
    output is the exact arithmetic mean of the visible values; if value j
    encodes its own logical position, that mean is a closed-form function of
    the visible set (verify: positions 0..L-k+i-1; draft: sinks plus window);
  * a two-key softmax is the logistic function;
  * a library routine: torch's fp64 scaled_dot_product_attention with an
    explicit boolean mask;
  * invariants the definitions imply: constant V, one dominant logit,
    row i == decoding at length L-k+i, window >= t == full attention,
    causality, page-permutation invariance, ring packing == logical mask.
"""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
import workloads

PAGE = 64


def _f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Exact for values representable in bf16 (small integers, powers of 2)."""
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
    rt = t.to(torch.float32).numpy()
    assert np.array_equal(rt, np.asarray(x, dtype=np.float32)), "value not exact in bf16"
    return t.view(torch.int16).numpy().view(np.uint16)


def _bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _paged_from_logical(Kl, Vl, L, rng, page=PAGE):
    """Scatter logical per-sequence K/V [B, Hkv, T, D] (bits) into a shuffled
    paged cache; returns (k_cache, v_cache, block_table)."""
    B, Hkv, T, D = Kl.shape
    pages = [(int(l) + page - 1) // page for l in L]
    n = sum(pages)
    order = rng.permutation(n)
    bt = np.full((B, max(pages)), -1, dtype=np.int32)
    kc = np.zeros((n, Hkv, page, D), dtype=np.uint16)
    vc = np.zeros_like(kc)
    off = 0
    for b in range(B):
        for p in range(pages[b]):
            phys = order[off + p]
            bt[b, p] = phys
            lo, hi = p * page, min((p + 1) * page, int(L[b]))
            kc[phys, :, :hi - lo] = Kl[b, :, lo:hi]
            vc[phys, :, :hi - lo] = Vl[b, :, lo:hi]
        off += pages[b]
    return kc, vc, bt


# --------------------------------------------------------------------------
# verify pins
# --------------------------------------------------------------------------
def pin_verify_uniform_logits_closed_form(lib):
    """q = 0: row i of sequence b, head h returns the mean of the values at
    logical positions 0..L-k+i-1.  Value j carries (j, kv-head index, 1, 0)."""
    rng = np.random.default_rng(11)
    k, Hq, Hkv, D = 3, 6, 3, 4
    G = Hq // Hkv
    L = np.array([4, 64, 65, 130, 200], dtype=np.int32)
    B, T = len(L), int(L.max())
    Kl = _f32_to_bf16_bits(rng.integers(-3, 4, size=(B, Hkv, T, D)).astype(np.float32))
    vals = np.zeros((B, Hkv, T, D), dtype=np.float32)
    vals[..., 0] = np.arange(T)[None, None, :]
    vals[..., 1] = np.arange(Hkv)[None, :, None]
    vals[..., 2] = 1.0
    Vl = _f32_to_bf16_bits(vals)
    kc, vc, bt = _paged_from_logical(Kl, Vl, L, rng)
    q = np.zeros((B, k + 1, Hq, D), dtype=np.uint16)
    out, n_bad = oracle.verify(q, kc, vc, bt, L, k, lib=lib)
    assert n_bad == 0
    for b in range(B):
        for i in range(k + 1):
            n = int(L[b]) - k + i
            for h in range(Hq):
                exp = np.array([(n - 1) / 2.0, h // G, 1.0, 0.0])
                np.testing.assert_allclose(out[b, i, h], exp, rtol=0, atol=1e-12)


def pin_verify_two_key_logistic(lib):
    """Two visible keys with scores a*scale and 0: weights are the logistic
    function of a*scale."""
    D = 2
    for a, scale in [(1.0, 1.0), (2.0, 0.5), (-3.0, 1.0)]:
        q = _f32_to_bf16_bits(np.array([[[[a, 0.0]]]], dtype=np.float32))
        keys = np.array([[1.0, 0.0], [0.0, 1.0]], dtype=np.float32)
        vals = np.array([[2.0, -1.0], [0.5, 4.0]], dtype=np.float32)
        kc = np.zeros((1, 1, PAGE, D), dtype=np.uint16)
        vc = np.zeros_like(kc)
        kc[0, 0, :2] = _f32_to_bf16_bits(keys)
        vc[0, 0, :2] = _f32_to_bf16_bits(vals)
        bt = np.zeros((1, 1), dtype=np.int32)
        out, _ = oracle.verify(q, kc, vc, bt, np.array([2], np.int32), 0, scale=scale, lib=lib)
        w0 = 1.0 / (1.0 + math.exp(-a * scale))
        exp = w0 * vals[0].astype(np.float64) + (1.0 - w0) * vals[1].astype(np.float64)
        np.testing.assert_allclose(out[0, 0, 0], exp, rtol=1e-14, atol=1e-14)


def pin_verify_constant_v(lib):
    """V identically c returns c for every row."""
    rng = np.random.default_rng(12)
    vi = workloads.make_verify([9, 70, 129], 2, 4, 2, 8, seed=5, device="cpu")
    c = 0.8125
    vc = workloads.bf16_bits(torch.full_like(vi.v_cache, c))
    out, _ = oracle.verify(workloads.bf16_bits(vi.q), workloads.bf16_bits(vi.k_cache), vc,
                           vi.block_table.numpy(), vi.ctx_lens.numpy(), vi.k, lib=lib)
    np.testing.assert_allclose(out, c, rtol=0, atol=1e-15)
    del rng


def pin_verify_one_hot_logit(lib):
    """One key whose score exceeds all others by >= 60 yields its value (the
    others carry weight < e^-60)."""
    D, L = 4, 50
    q = _f32_to_bf16_bits(np.array([[[[16.0, 0, 0, 0]]]], dtype=np.float32))
    keys = np.zeros((L, D), np.float32)
    keys[:, 1] = 1.0
    keys[17, 0] = 4.0        # score 64 vs 0
    rng = np.random.default_rng(13)
    vals = rng.integers(-8, 9, size=(L, D)).astype(np.float32)
    kc = np.zeros((1, 1, PAGE, D), np.uint16)
    vc = np.zeros_like(kc)
    kc[0, 0, :L] = _f32_to_bf16_bits(keys)
    vc[0, 0, :L] = _f32_to_bf16_bits(vals)
    out, _ = oracle.verify(q, kc, vc, np.zeros((1, 1), np.int32), np.array([L], np.int32), 0,
                           lib=lib)
    np.testing.assert_allclose(out[0, 0, 0], vals[17], rtol=0, atol=1e-20 + 64 * math.exp(-60))


def pin_verify_matches_sdpa(lib):
    """torch fp64 scaled_dot_product_attention with an explicit causal-block
    mask and GQA head expansion, on random data."""
    for (L, k, Hq, Hkv, D, scale, seed) in [([7, 64, 100], 2, 4, 2, 16, 1.0, 1),
                                              ([5, 128], 4, 3, 1, 8, 0.37, 2),
                                              ([1, 66], 0, 2, 2, 32, 1.0, 3)]:
        vi = workloads.make_verify(L, k, Hq, Hkv, D, seed=seed, device="cpu", shuffle=True)
        qb, kb, vb = (workloads.bf16_bits(t) for t in (vi.q, vi.k_cache, vi.v_cache))
        out, n_bad = oracle.verify(qb, kb, vb, vi.block_table.numpy(), vi.ctx_lens.numpy(), k,
                                   scale=scale, lib=lib)
        assert n_bad == 0
        G = Hq // Hkv
        for b, Lb in enumerate(L):
            pages = vi.block_table[b, :(Lb + PAGE - 1) // PAGE].long()
            K = vi.k_cache[pages].permute(1, 0, 2, 3).reshape(Hkv, -1, D)[:, :Lb].double()
            V = vi.v_cache[pages].permute(1, 0, 2, 3).reshape(Hkv, -1, D)[:, :Lb].double()
            K = K.repeat_interleave(G, dim=0)
            V = V.repeat_interleave(G, dim=0)
            Q = vi.q[b].permute(1, 0, 2).double()               # [Hq, k+1, D]
            rows = torch.arange(k + 1)[:, None]
            cols = torch.arange(Lb)[None, :]
            mask = cols < (Lb - k + rows)
            ref = torch.nn.functional.scaled_dot_product_attention(
                Q, K, V, attn_mask=mask, scale=scale)            # [Hq, k+1, D]
            np.testing.assert_allclose(out[b], ref.permute(1, 0, 2).numpy(), rtol=1e-12,
                                       atol=1e-12)


def pin_verify_row_equals_decode(lib):
    """Block row i equals single-query decoding (k = 0) at length L-k+i."""
    L, k = [70, 131], 4
    vi = workloads.make_verify(L, k, 4, 2, 16, seed=21, device="cpu")
    qb, kb, vb = (workloads.bf16_bits(t) for t in (vi.q, vi.k_cache, vi.v_cache))
    bt = vi.block_table.numpy()
    out, _ = oracle.verify(qb, kb, vb, bt, np.array(L, np.int32), k, lib=lib)
    for i in range(k + 1):
        Li = np.array([l - k + i for l in L], np.int32)
        dec, _ = oracle.verify(np.ascontiguousarray(qb[:, i:i + 1]), kb, vb, bt, Li, 0, lib=lib)
        np.testing.assert_allclose(out[:, i], dec[:, 0], rtol=1e-15, atol=1e-15)


def pin_verify_causality(lib):
    """Changing the K/V of block token at position L-k+i changes row i and
    leaves rows < i bit-identical."""
    L, k = [100], 4
    vi = workloads.make_verify(L, k, 2, 1, 8, seed=31, device="cpu", shuffle=False)
    qb, kb, vb = (workloads.bf16_bits(t) for t in (vi.q, vi.k_cache, vi.v_cache))
    bt = vi.block_table.numpy()
    base, _ = oracle.verify(qb, kb, vb, bt, np.array(L, np.int32), k, lib=lib)
    for i in range(1, k + 1):
        j = L[0] - k + i - 1          # first key visible to row i but not row i-1
        kb2, vb2 = kb.copy(), vb.copy()
        page, slot = bt[0, j // PAGE], j % PAGE
        kb2[page, :, slot] = _f32_to_bf16_bits(np.full(8, 2.0, np.float32))
        vb2[page, :, slot] = _f32_to_bf16_bits(np.full(8, 64.0, np.float32))
        out, _ = oracle.verify(qb, kb2, vb2, bt, np.array(L, np.int32), k, lib=lib)
        assert np.array_equal(out[:, :i], base[:, :i])
        assert not np.allclose(out[:, i], base[:, i])


def pin_verify_page_permutation(lib):
    """Permuting physical pages (and the block table with them) gives
    bit-identical results."""
    L, k = [130, 64, 3], 1
    vi = workloads.make_verify(L, k, 4, 2, 8, seed=41, device="cpu", shuffle=False)
    qb, kb, vb = (workloads.bf16_bits(t) for t in (vi.q, vi.k_cache, vi.v_cache))
    bt = vi.block_table.numpy()
    base, _ = oracle.verify(qb, kb, vb, bt, np.array(L, np.int32), k, lib=lib)
    perm = np.random.default_rng(3).permutation(kb.shape[0])
    inv = np.argsort(perm)
    bt2 = np.where(bt >= 0, inv[np.maximum(bt, 0)], -1).astype(np.int32)
    out, _ = oracle.verify(qb, kb[perm], vb[perm], bt2, np.array(L, np.int32), k, lib=lib)
    assert np.array_equal(out, base)


def pin_verify_invalid_lengths(lib):
    """Sequences with L < k+1, L beyond the table, or a page id outside the
    cache yield NaN rows and are counted; valid ones are untouched."""
    vi = workloads.make_verify([64, 64, 64, 64], 2, 2, 1, 8, seed=51, device="cpu")
    qb, kb, vb = (workloads.bf16_bits(t) for t in (vi.q, vi.k_cache, vi.v_cache))
    bt = vi.block_table.numpy().copy()
    L = np.array([64, 2, 65, 64], np.int32)
    bt[3, 0] = kb.shape[0]
    out, n_bad = oracle.verify(qb, kb, vb, bt, L, 2, lib=lib)
    assert n_bad == 3
    assert np.all(np.isfinite(out[0])) and np.all(np.isnan(out[1:]))


# --------------------------------------------------------------------------
# draft pins
# --------------------------------------------------------------------------
def _draft_positions_closed_form(t, n_sink, window):
    """Mean logical position over V(t), in closed form."""
    S = n_sink + window
    if t <= S:
        return (t - 1) / 2.0
    s = min(n_sink, t)
    sink_sum = s * (s - 1) / 2.0
    lo = t - window
    win_sum = window * (lo + t - 1) / 2.0
    return (sink_sum + win_sum) / (s + window)


def pin_draft_uniform_logits_closed_form(lib):
    """q = 0: the draft output is the mean over the visible set V(t); value at
    logical position p carries p, so the mean is a closed form in t, n_sink
    and window.  Runs on the logical form and on the packed ring."""
    D, Hkv, Hq = 4, 2, 4
    for (n_sink, window) in [(4, 8), (0, 5), (1, 64), (3, 1)]:
        S = n_sink + window
        ts = np.array([1, 2, n_sink + 1, S - 1 if S > 1 else 1, S, S + 1, 2 * S + 3, 200],
                      dtype=np.int32)
        ts = np.maximum(ts, 1)
        B, T = len(ts), int(ts.max())
        vals = np.zeros((B, Hkv, T, D), np.float32)
        vals[..., 0] = np.arange(T)[None, None, :]
        vals[..., 1] = np.arange(Hkv)[None, :, None]
        vals[..., 3] = 1.0
        Vl = _f32_to_bf16_bits(vals)
        Kl = _f32_to_bf16_bits(np.ones((B, Hkv, T, D), np.float32))
        q = np.zeros((B, Hq, D), np.uint16)
        lo, nb = oracle.draft_logical(q, Kl, Vl, ts, n_sink, window, lib=lib)
        ring = oracle.ring_pack(Kl, Vl, ts, n_sink, window, lib=lib)
        ro, nb2 = oracle.draft_ring(q, ring, ts, n_sink, window, lib=lib)
        assert nb == 0 and nb2 == 0
        for b, t in enumerate(ts):
            for h in range(Hq):
                exp = np.array([_draft_positions_closed_form(int(t), n_sink, window),
                                h // (Hq // Hkv), 0.0, 1.0])
                np.testing.assert_allclose(lo[b, h], exp, rtol=0, atol=1e-12)
                np.testing.assert_allclose(ro[b, h], exp, rtol=0, atol=1e-12)


def pin_draft_matches_sdpa(lib):
    """Logical form vs torch fp64 SDPA with the sink + window mask written as
    a boolean mask over positions 0..T-1."""
    rng = np.random.default_rng(61)
    B, Hq, Hkv, D, T = 3, 4, 2, 16, 90
    for (n_sink, window) in [(4, 16), (0, 7), (2, 100)]:
        ts = np.array([1, 37, 90], np.int32)
        Kf = rng.standard_normal((B, Hkv, T, D)).astype(np.float32)
        Vf = rng.standard_normal((B, Hkv, T, D)).astype(np.float32)
        Qf = (rng.standard_normal((B, Hq, D)) / 4).astype(np.float32)
        Kb, Vb, Qb = (torch.from_numpy(x).to(torch.bfloat16) for x in (Kf, Vf, Qf))
        bits = lambda t: t.view(torch.int16).numpy().view(np.uint16)
        out, _ = oracle.draft_logical(bits(Qb), bits(Kb), bits(Vb), ts, n_sink, window, lib=lib)
        G = Hq // Hkv
        for b, t in enumerate(ts):
            pos = torch.arange(T)
            mask = (pos < t) & ((pos < n_sink) | (pos >= t - window))
            K = Kb[b].double().repeat_interleave(G, 0)
            V = Vb[b].double().repeat_interleave(G, 0)
            Q = Qb[b].double()[:, None, :]
            ref = torch.nn.functional.scaled_dot_product_attention(
                Q, K, V, attn_mask=mask[None, None, :].expand(Hq, 1, T), scale=1.0)
            np.testing.assert_allclose(out[b], ref[:, 0].numpy(), rtol=1e-12, atol=1e-12)


def pin_draft_ring_equals_logical(lib):
    """Packing a logical memory into the bounded cache and attending over the
    ring equals attending over the logical memory with the mask, bit for bit."""
    rng = np.random.default_rng(71)
    B, Hq, Hkv, D = 4, 4, 1, 8
    for (n_sink, window) in [(4, 16), (0, 9), (16, 1)]:
        ts = np.array([3, 20, 21, 95], np.int32)
        T = int(ts.max())
        f = lambda *s: torch.from_numpy(rng.standard_normal(s).astype(np.float32)).to(torch.bfloat16)
        bits = lambda t: t.view(torch.int16).numpy().view(np.uint16)
        Kl, Vl, Q = bits(f(B, Hkv, T, D)), bits(f(B, Hkv, T, D)), bits(f(B, Hq, D))
        lo, _ = oracle.draft_logical(Q, Kl, Vl, ts, n_sink, window, lib=lib)
        ring = oracle.ring_pack(Kl, Vl, ts, n_sink, window, lib=lib)
        ro, _ = oracle.draft_ring(Q, ring, ts, n_sink, window, lib=lib)
        assert np.array_equal(lo, ro)


def pin_draft_window_covers_context(lib):
    """window >= t: the draft output equals full attention over all t entries,
    i.e. the verification oracle at k = 0 over a contiguous cache."""
    rng = np.random.default_rng(81)
    B, Hq, Hkv, D = 3, 4, 2, 16
    n_sink, window = 2, 200
    ts = np.array([1, 64, 150], np.int32)
    S = n_sink + window
    kv = torch.from_numpy(rng.standard_normal((B, 2, Hkv, S, D)).astype(np.float32)).to(torch.bfloat16)
    q = torch.from_numpy((rng.standard_normal((B, Hq, D)) / 4).astype(np.float32)).to(torch.bfloat16)
    bits = lambda t: t.contiguous().view(torch.int16).numpy().view(np.uint16)
    dr, _ = oracle.draft_ring(bits(q), bits(kv), ts, n_sink, window, lib=lib)
    pages = (S + PAGE - 1) // PAGE
    kc = torch.zeros((B * pages, Hkv, PAGE, D), dtype=torch.bfloat16)
    vc = torch.zeros_like(kc)
    for b in range(B):
        for p in range(pages):
            lo, hi = p * PAGE, min(S, (p + 1) * PAGE)
            kc[b * pages + p, :, :hi - lo] = kv[b, 0, :, lo:hi]
            vc[b * pages + p, :, :hi - lo] = kv[b, 1, :, lo:hi]
    bt = np.arange(B * pages, dtype=np.int32).reshape(B, pages)
    full, _ = oracle.verify(bits(q[:, None]), bits(kc), bits(vc), bt, ts, 0, lib=lib)
    np.testing.assert_allclose(dr, full[:, 0], rtol=1e-15, atol=1e-15)


def pin_draft_slot_is_bijective(lib):
    """For every t >= S the visible positions fill each of the S slots exactly
    once; sinks keep their own slot; entries p and p+window share a slot."""
    for (n_sink, window) in [(0, 1), (1, 64), (16, 512), (4, 7)]:
        S = n_sink + window
        for t in [S, S + 1, 3 * S + 5]:
            vis = [p for p in range(t) if p < n_sink or p >= t - window]
            slots = sorted(oracle.draft_slot(p, n_sink, window, lib=lib) for p in vis)
            assert slots == list(range(S))
        for p in range(n_sink):
            assert oracle.draft_slot(p, n_sink, window, lib=lib) == p
        for p in range(n_sink, n_sink + 3 * window):
            assert oracle.draft_slot(p, n_sink, window, lib=lib) == \
                oracle.draft_slot(p + window, n_sink, window, lib=lib)
            assert oracle.draft_slot(p, n_sink, window, lib=lib) >= n_sink


def pin_draft_invalid_t(lib):
    """t = 0 (no memory entry yet) yields NaN and is counted."""
    di = workloads.make_draft([0, 5], 2, 1, 8, 1, 4, seed=3, device="cpu")
    out, n_bad = oracle.draft_ring(workloads.bf16_bits(di.q), workloads.bf16_bits(di.kv),
                                   di.ctx_lens.numpy(), 1, 4, lib=lib)
    assert n_bad == 1 and np.all(np.isnan(out[0])) and np.all(np.isfinite(out[1]))




# --------------------------------------------------------------------------
# feedback-memory append pins
# --------------------------------------------------------------------------
def _rand_bf16_bits(rng, shape, scale=1.0):
    t = torch.from_numpy((rng.standard_normal(shape) * scale).astype(np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _torch_round_bf16_bits(v: np.ndarray) -> np.ndarray:
    """float64 -> float32 -> bf16 (torch, nearest even); double rounding, so
    it may differ from single rounding by one unit in rare near-tie cases."""
    t = torch.from_numpy(np.ascontiguousarray(v, dtype=np.float64).astype(np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _bf16_ulps(a_bits: np.ndarray, b_bits: np.ndarray) -> np.ndarray:
    """Distance in bf16 units between two bit arrays (same-sign values)."""
    def ordered(x):
        x = x.astype(np.int32)
        return np.where(x & 0x8000, -(x & 0x7FFF), x)
    return np.abs(ordered(a_bits) - ordered(b_bits))


def pin_round_bf16_ties_and_library(lib):
    """Nearest-even bf16 rounding: exact ties go to the even neighbour,
    subnormals and overflow follow IEEE rules, and random float32 values
    round as torch's float32 -> bf16 conversion does."""
    ties = {1.0 + 2.0 ** -8: 0x3F80, 1.0 + 3 * 2.0 ** -8: 0x3F82,
            -(1.0 + 2.0 ** -8): 0xBF80, 2.5 * 2.0 ** -133: 0x0002,
            3.5 * 2.0 ** -133: 0x0004, 0.5 * 2.0 ** -133: 0x0000,
            (2 - 2.0 ** -8) * 2.0 ** 127: 0x7F80, 3.0e38: 0x7F62, 0.0: 0x0000}
    for v, want in ties.items():
        assert oracle.round_bf16(v, lib=lib) == want, (v, hex(oracle.round_bf16(v, lib=lib)))
    assert oracle.round_bf16(float("nan"), lib=lib) & 0x7FC0 == 0x7FC0
    rng = np.random.default_rng(21)
    vals = np.concatenate([rng.standard_normal(4000) * 10.0 ** rng.integers(-30, 30, 4000),
                           rng.standard_normal(500) * 1e-39]).astype(np.float32)
    got = np.array([oracle.round_bf16(float(v), lib=lib) for v in vals], dtype=np.uint16)
    assert np.array_equal(got, _torch_round_bf16_bits(vals.astype(np.float64)))


def pin_feedback_mix_one_hot_and_mean(lib):
    """w one-hot (one weight 0, the others -1000) gives m = x^l exactly;
    equal weights give the plain mean over the n_layer + 1 activations."""
    rng = np.random.default_rng(22)
    n_act, B, d_model = 3, 5, 64
    x = _rand_bf16_bits(rng, (n_act, B, d_model))
    xf = _bits_to_f64(x)
    w = np.full((n_act + 1, n_act), -1000.0)
    for i in range(n_act):
        w[i, i] = 0.0
    w[n_act] = 0.37
    m = oracle.feedback_mix(x, w, lib=lib)
    for i in range(n_act):
        assert np.array_equal(m[i], xf[i])
    np.testing.assert_allclose(m[n_act], xf.mean(axis=0), rtol=1e-14, atol=1e-15)


def pin_feedback_mix_two_layer_logistic(lib):
    """Two activations with weights (a, 0): m = s x^0 + (1 - s) x^1 with
    s = 1 / (1 + e^-a), the logistic function; shifting both weights by a
    constant changes nothing."""
    rng = np.random.default_rng(23)
    x = _rand_bf16_bits(rng, (2, 3, 64))
    xf = _bits_to_f64(x)
    for a in (-3.0, 0.0, 0.7, 5.0):
        s = 1.0 / (1.0 + math.exp(-a))
        m = oracle.feedback_mix(x, np.array([[a, 0.0], [a + 11.0, 11.0]]), lib=lib)
        want = s * xf[0] + (1.0 - s) * xf[1]
        np.testing.assert_allclose(m[0], want, rtol=1e-13, atol=1e-15)
        np.testing.assert_allclose(m[1], want, rtol=1e-13, atol=1e-15)


def _append_case(rng, B, Hkv, D, d_model, n_act, n_dl, n_sink, window):
    S = n_sink + window
    x = _rand_bf16_bits(rng, (n_act, B, d_model))
    w = rng.standard_normal((n_dl, n_act))
    kv = _rand_bf16_bits(rng, (n_dl, B, 2, Hkv, S, D))
    return x, w, kv


def pin_feedback_append_selection_projection(lib):
    """With a one-hot mix and a 0/1 selection matrix as the projection, the
    appended K/V rows are the selected activation entries, bit for bit, in
    slot(p) of each layer's cache; every other slot is untouched."""
    rng = np.random.default_rng(24)
    B, Hkv, D, n_act, n_dl, n_sink, window = 3, 2, 8, 2, 2, 2, 5
    F = 2 * Hkv * D
    d_model = F
    x, _, kv0 = _append_case(rng, B, Hkv, D, d_model, n_act, n_dl, n_sink, window)
    w = np.array([[0.0, -1000.0], [-1000.0, 0.0]])
    perms = [rng.permutation(F) for _ in range(n_dl)]
    wkv = np.zeros((n_dl, F, d_model), dtype=np.float32)
    for i in range(n_dl):
        wkv[i, np.arange(F), perms[i]] = 1.0
    wkv = _f32_to_bf16_bits(wkv)
    pos = np.array([0, 6, 40], dtype=np.int32)
    kv = kv0.copy()
    assert oracle.feedback_append(x, w, wkv, pos, kv, n_sink, window, lib=lib) == 0
    want = kv0.copy()
    for i in range(n_dl):
        for b in range(B):
            s = oracle.draft_slot(int(pos[b]), n_sink, window, lib=lib)
            y = x[i, b, perms[i]]
            want[i, b, 0, :, s] = y[:Hkv * D].reshape(Hkv, D)
            want[i, b, 1, :, s] = y[Hkv * D:].reshape(Hkv, D)
    assert np.array_equal(kv, want)


def pin_feedback_append_matches_matmul(lib):
    """Random activations, mixing weights and projections against a float64
    numpy einsum of the same definition, rounded by torch: every entry within
    one bf16 unit, nearly all identical (torch rounds twice: via float32)."""
    rng = np.random.default_rng(25)
    B, Hkv, D, d_model, n_act, n_dl, n_sink, window = 4, 2, 16, 96, 3, 2, 3, 6
    x, w, kv0 = _append_case(rng, B, Hkv, D, d_model, n_act, n_dl, n_sink, window)
    wkv = _rand_bf16_bits(rng, (n_dl, 2 * Hkv * D, d_model), scale=0.1)
    pos = np.array([1, 9, 2, 30], dtype=np.int32)
    kv = kv0.copy()
    oracle.feedback_append(x, w, wkv, pos, kv, n_sink, window, lib=lib)
    a = np.exp(w - w.max(axis=1, keepdims=True))
    a /= a.sum(axis=1, keepdims=True)
    m = np.einsum("il,lbc->ibc", a, _bits_to_f64(x))
    y = np.einsum("ifc,ibc->ibf", _bits_to_f64(wkv), m)
    want = _torch_round_bf16_bits(y)
    got = np.zeros_like(want)
    for i in range(n_dl):
        for b in range(B):
            s = oracle.draft_slot(int(pos[b]), n_sink, window, lib=lib)
            got[i, b] = kv[i, b, :, :, s].reshape(-1)
    ulps = _bf16_ulps(got, want)
    assert ulps.max() <= 1 and (ulps == 0).mean() >= 0.99


def pin_feedback_append_rotary_complex_form(lib):
    """rope_theta > 0 turns each key pair (k[d], k[d + D/2]) by the angle
    p * theta^(-2d/D): the complex number k[d] + i k[d + D/2] times
    e^(i angle).  Values are not rotated, position 0 is the identity, and
    the first and middle frequencies are 1 and theta^-1/2."""
    rng = np.random.default_rng(26)
    B, Hkv, D, n_act, n_dl, n_sink, window = 4, 2, 16, 1, 1, 1, 8
    F = 2 * Hkv * D
    theta = 10000.0
    x, _, kv0 = _append_case(rng, B, Hkv, D, F, n_act, n_dl, n_sink, window)
    w = np.zeros((1, 1))
    wkv = _f32_to_bf16_bits(np.eye(F, dtype=np.float32)[None])
    pos = np.array([0, 1, 77, 100003], dtype=np.int32)
    kv = kv0.copy()
    oracle.feedback_append(x, w, wkv, pos, kv, n_sink, window, rope_theta=theta, lib=lib)
    xf = _bits_to_f64(x[0])
    for b in range(B):
        s = oracle.draft_slot(int(pos[b]), n_sink, window, lib=lib)
        kf = xf[b, :Hkv * D].reshape(Hkv, D)
        assert np.array_equal(kv[0, b, 1, :, s].reshape(-1), x[0, b, Hkv * D:])
        if pos[b] == 0:
            assert np.array_equal(kv[0, b, 0, :, s].reshape(-1), x[0, b, :Hkv * D])
        freq = theta ** (-2.0 * np.arange(D // 2) / D)
        assert freq[0] == 1.0 and abs(freq[D // 4] - theta ** -0.5) < 1e-15
        z = (kf[:, :D // 2] + 1j * kf[:, D // 2:]) * np.exp(1j * float(pos[b]) * freq)[None]
        want = _torch_round_bf16_bits(np.concatenate([z.real, z.imag], axis=1))
        got = kv[0, b, 0, :, s]
        ulps = _bf16_ulps(got, want)
        assert ulps.max() <= 1 and (ulps == 0).mean() >= 0.9


def pin_feedback_append_negative_position(lib):
    """A negative position is counted and writes nothing."""
    rng = np.random.default_rng(27)
    x, w, kv0 = _append_case(rng, 2, 1, 8, 16, 2, 1, 1, 4)
    wkv = _rand_bf16_bits(rng, (1, 16, 16))
    kv = kv0.copy()
    n_bad = oracle.feedback_append(x, w, wkv, np.array([-1, 3], dtype=np.int32), kv, 1, 4,
                                   lib=lib)
    assert n_bad == 1 and np.array_equal(kv[:, 0], kv0[:, 0])
    assert not np.array_equal(kv[:, 1], kv0[:, 1])


# --------------------------------------------------------------------------
# token verification (modified rejection sampling) pins
# --------------------------------------------------------------------------
def pin_tokens_hand_example(lib):
    """Two sequences worked by hand (V = 4, k = 2).
    Sequence 0: draft 3 is accepted (0.9 * 0.25 < 0.4), draft 1 rejected
    (0.5 * 0.6 >= 0.1); residual max(0, p2 - q2) = (0.4, 0, 0, 0.2) with
    E = (1, .5, .5, .3) scores 0.4 and 0.667: token 3.  Sequence 1: both drafts
    accepted; bonus from p3 = (0, .7, .3, 0) with E = (1, 2, .25, 1): scores
    0.35 and 1.2, token 2."""
    p = np.array([[[0.1, 0.2, 0.3, 0.4], [0.5, 0.1, 0.1, 0.3], [0.0, 0.7, 0.3, 0.0]],
                  [[0.1, 0.2, 0.3, 0.4], [0.5, 0.1, 0.1, 0.3], [0.0, 0.7, 0.3, 0.0]]],
                 dtype=np.float32)
    q = np.array([[[0.25, 0.25, 0.25, 0.25], [0.1, 0.6, 0.2, 0.1]],
                  [[0.25, 0.25, 0.25, 0.25], [0.4, 0.1, 0.4, 0.1]]], dtype=np.float32)
    x = np.array([[3, 1], [2, 0]], dtype=np.int32)
    u = np.array([[0.9, 0.5], [0.5, 0.9]], dtype=np.float32)
    e = np.array([[1.0, 0.5, 0.5, 0.3], [1.0, 2.0, 0.25, 1.0]], dtype=np.float32)
    out, n_acc, n_bad = oracle.verify_tokens(p, q, x, u, e, lib=lib)
    assert n_bad == 0
    assert out.tolist() == [[3, 3, -1], [2, 0, 2]] and n_acc.tolist() == [1, 2]


def _round_samples(rng, n, p_rows, q_rows):
    """n independent rounds with fixed distributions: drafts drawn from q_i,
    uniforms and Exp(1) variates from numpy."""
    kp1, V = p_rows.shape
    k = kp1 - 1
    qd = q_rows.astype(np.float64)
    x = np.stack([rng.choice(V, size=n, p=qd[i] / qd[i].sum()) for i in range(k)],
                 axis=1).astype(np.int32)
    u = rng.random((n, k), dtype=np.float32)
    e = rng.exponential(size=(n, V)).astype(np.float32)
    p = np.broadcast_to(p_rows, (n, kp1, V))
    q = np.broadcast_to(q_rows, (n, k, V))
    return p, q, x, u, e


def _chi2_ok(counts, probs):
    from scipy.stats import chisquare
    keep = probs > 0
    assert counts[~keep].sum() == 0, "a token of probability 0 was emitted"
    return chisquare(counts[keep], counts[keep].sum() * probs[keep] / probs[keep].sum()).pvalue


def pin_tokens_emitted_tokens_follow_the_target(lib):
    """The scheme's guarantee (Section 1): the first emitted token is a sample
    of p_1, and, where the first draft was accepted, the second of p_2 (the
    synthetic distributions do not depend on the prefix)."""
    rng = np.random.default_rng(41)
    V, k, n = 6, 3, 120000
    p_rows = rng.dirichlet(np.ones(V), size=k + 1).astype(np.float32)
    q_rows = rng.dirichlet(np.ones(V), size=k).astype(np.float32)
    p, q, x, u, e = _round_samples(rng, n, p_rows, q_rows)
    out, n_acc, _ = oracle.verify_tokens(p, q, x, u, e, lib=lib)
    c0 = np.bincount(out[:, 0], minlength=V)
    assert _chi2_ok(c0, p_rows[0].astype(np.float64)) > 1e-4
    sel = n_acc >= 1
    c1 = np.bincount(out[sel, 1], minlength=V)
    assert _chi2_ok(c1, p_rows[1].astype(np.float64)) > 1e-4


def pin_tokens_acceptance_rate_is_alpha(lib):
    """A draft drawn from q is accepted with probability
    alpha = sum_v min(p_v, q_v), the expected acceptance probability
    (Section 3.4)."""
    rng = np.random.default_rng(42)
    V, k, n = 8, 1, 200000
    p_rows = rng.dirichlet(np.ones(V), size=k + 1).astype(np.float32)
    q_rows = rng.dirichlet(np.ones(V), size=k).astype(np.float32)
    p, q, x, u, e = _round_samples(rng, n, p_rows, q_rows)
    _, n_acc, _ = oracle.verify_tokens(p, q, x, u, e, lib=lib)
    alpha = np.minimum(p_rows[0].astype(np.float64), q_rows[0]).sum()
    rate = (n_acc == 1).mean()
    assert abs(rate - alpha) < 5 * math.sqrt(alpha * (1 - alpha) / n)


def pin_tokens_identical_models_accept_all(lib):
    """p_i = q_i: every draft is accepted (u < 1) and the bonus token is a
    sample of p_{k+1}."""
    rng = np.random.default_rng(43)
    V, k, n = 5, 2, 100000
    rows = rng.dirichlet(np.ones(V), size=k + 1).astype(np.float32)
    p, q, x, u, e = _round_samples(rng, n, rows, rows[:k])
    out, n_acc, _ = oracle.verify_tokens(p, q, x, u, e, lib=lib)
    assert np.all(n_acc == k) and np.array_equal(out[:, :k], x)
    assert _chi2_ok(np.bincount(out[:, k], minlength=V), rows[k].astype(np.float64)) > 1e-4


def pin_tokens_invalid_inputs(lib):
    """A draft token outside [0, V) counts as rejected; an Exp value that is
    not > 0 is skipped; both are counted."""
    p = np.full((2, 2, 3), 1.0 / 3, dtype=np.float32)
    q = np.full((2, 1, 3), 1.0 / 3, dtype=np.float32)
    x = np.array([[7], [1]], dtype=np.int32)
    u = np.zeros((2, 1), dtype=np.float32)
    e = np.array([[1.0, 1.0, 1.0], [0.0, 2.0, 1.0]], dtype=np.float32)
    out, n_acc, n_bad = oracle.verify_tokens(p, q, x, u, e, lib=lib)
    assert n_bad == 2
    assert n_acc.tolist() == [0, 1]
    # sequence 0: residual of p = q is empty, so the draw falls back to p (ties: token 0)
    assert out[0].tolist() == [0, -1]
    # sequence 1: bonus from p_2 with E_0 skipped: scores (1/3)/2 and (1/3)/1 -> token 2
    assert out[1].tolist() == [1, 2]


# --------------------------------------------------------------------------
# MagicDec draft attention pins
# --------------------------------------------------------------------------
def _rope_f64(x, pos, theta):
    """Half-split rotary turn of x [..., D] (float64) by position pos, with
    math.cos / math.sin / math.pow, the C library the oracle calls."""
    D = x.shape[-1]
    out = x.copy()
    for d in range(D // 2):
        a = pos * math.pow(theta, -2.0 * d / D)
        c, s_ = math.cos(a), math.sin(a)
        out[..., d] = x[..., d] * c - x[..., d + D // 2] * s_
        out[..., d + D // 2] = x[..., d + D // 2] * c + x[..., d] * s_
    return out


def _md_case(rng, L, Hq, Hkv, D, shuffle=True):
    B, T = len(L), int(max(L))
    Kl = _f32_to_bf16_bits(rng.integers(-3, 4, size=(B, Hkv, T, D)).astype(np.float32))
    Vl = _rand_bf16_bits(rng, (B, Hkv, T, D))
    kc, vc, bt = _paged_from_logical(Kl, Vl, L, rng)
    q = _rand_bf16_bits(rng, (B, Hq, D), scale=0.2)
    return q, Kl, Vl, kc, vc, bt


def pin_magicdec_without_rotation_is_sink_window(lib):
    """theta = 0: exactly the sink + window attention of the draft definition
    (the same visible set, read through the block table)."""
    rng = np.random.default_rng(51)
    L = np.array([1, 3, 66, 130, 200], dtype=np.int32)
    q, Kl, Vl, kc, vc, bt = _md_case(rng, L, 4, 2, 16)
    got, nb = oracle.magicdec(q, kc, vc, bt, L, 2, 64, 0.0, lib=lib)
    want, nb2 = oracle.draft_logical(q, Kl, Vl, L, 2, 64, lib=lib)
    assert nb == 0 and nb2 == 0
    np.testing.assert_allclose(got, want, rtol=1e-14, atol=1e-14)


def pin_magicdec_uniform_query_closed_form(lib):
    """q = 0 (any rotation leaves it 0): the mean of the visible values; value
    j carries its own position, so the mean is the closed form of the sink +
    window positions."""
    rng = np.random.default_rng(52)
    L = np.array([1, 5, 70, 129, 250], dtype=np.int32)   # positions exact in bf16
    n_sink, window, D = 3, 20, 8
    q, Kl, _, _, _, _ = _md_case(rng, L, 2, 1, D)
    q[:] = 0
    T = int(L.max())
    vals = np.zeros((len(L), 1, T, D), dtype=np.float32)
    vals[..., 0] = np.arange(T)[None, None, :]
    vals[..., 1] = 1.0
    Vl = _f32_to_bf16_bits(vals)
    kc, vc, bt = _paged_from_logical(Kl, Vl, L, rng)
    got, nb = oracle.magicdec(q, kc, vc, bt, L, n_sink, window, 10000.0, lib=lib)
    assert nb == 0
    for b, t in enumerate(L):
        np.testing.assert_allclose(got[b, :, 0], _draft_positions_closed_form(int(t), n_sink, window),
                                   rtol=1e-12)
        np.testing.assert_allclose(got[b, :, 1], 1.0, rtol=1e-14)


def pin_magicdec_full_window_is_rotary_decoding(lib):
    """window >= t: cache indices equal text positions, so keys keep their
    stored rotation and the query turns by t - 1: plain rotary decoding
    (the verify definition at k = 0 with that query)."""
    rng = np.random.default_rng(53)
    L = np.array([1, 7, 64, 100], dtype=np.int32)
    theta, D = 10000.0, 16
    q, _, _, kc, vc, bt = _md_case(rng, L, 4, 2, D)
    got, nb = oracle.magicdec(q, kc, vc, bt, L, 1, 128, theta, lib=lib)
    assert nb == 0
    qf = _bits_to_f64(q)
    qe = np.zeros_like(q)
    for b, t in enumerate(L):
        r = _rope_f64(qf[b], float(t - 1), theta)
        qe[b] = np.array([[oracle.round_bf16(v, lib=lib) for v in row] for row in r],
                         dtype=np.uint16)
    want, nb2 = oracle.verify(qe[:, None], kc, vc, bt, L, 0, lib=lib)
    assert nb2 == 0
    np.testing.assert_allclose(got, want[:, 0], rtol=1e-13, atol=1e-13)


def pin_magicdec_positions_are_cache_indices(lib):
    """The same visible tokens (keys stored turned by their own text
    positions) at two different context lengths give the same attention: only
    positions inside the reduced cache matter.  Equal up to the bf16 rounding
    of the stored and re-turned keys."""
    rng = np.random.default_rng(54)
    n_sink, window, D, Hkv, Hq, theta = 2, 12, 32, 1, 2, 10000.0
    n = n_sink + window
    kraw = rng.standard_normal((Hkv, n, D))
    vraw = _rand_bf16_bits(rng, (Hkv, n, D))
    q = _rand_bf16_bits(rng, (1, Hq, D), scale=0.7)
    outs = []
    for t in (40, 300):
        Kl = np.zeros((1, Hkv, t, D), dtype=np.uint16)
        Vl = np.zeros((1, Hkv, t, D), dtype=np.uint16)
        pos = list(range(n_sink)) + list(range(t - window, t))
        for c, p_ in enumerate(pos):
            r = _rope_f64(kraw[:, c], float(p_), theta)
            Kl[0, :, p_] = torch.from_numpy(r.astype(np.float32)).to(torch.bfloat16) \
                .view(torch.int16).numpy().view(np.uint16)
            Vl[0, :, p_] = vraw[:, c]
        L = np.array([t], dtype=np.int32)
        kc, vc, bt = _paged_from_logical(Kl, Vl, L, rng)
        o, nb = oracle.magicdec(q, kc, vc, bt, L, n_sink, window, theta, lib=lib)
        assert nb == 0
        outs.append(o)
    rel = np.linalg.norm(outs[0] - outs[1]) / np.linalg.norm(outs[1])
    assert rel < 2e-2, rel


def pin_magicdec_invalid(lib):
    """t = 0, t beyond the table, or a visible page outside the cache: NaN."""
    rng = np.random.default_rng(55)
    L = np.array([0, 40, 40, 500], dtype=np.int32)
    q, _, _, kc, vc, bt = _md_case(rng, np.array([1, 40, 40, 64]), 2, 1, 8)
    bt = bt.copy()
    bt[2, 0] = 99999
    got, nb = oracle.magicdec(q, kc, vc, bt, L, 1, 8, 10000.0, lib=lib)
    assert nb == 3
    assert np.all(np.isnan(got[[0, 2, 3]])) and np.all(np.isfinite(got[1]))


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
