"""GPU parity: the CUDA path, called through the C ABI, against the fp64
oracle on the same seeded inputs, plus the exactness properties of indexing."""
import numpy as np
import pytest
import torch

import parity
import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spire():
    import paper_2504_06419_gb300 as m
    return m


DEV = "cuda"


# ---------------------------------------------------------------- verify
VERIFY_CASES = [
    # (ctx_lens, k, Hq, Hkv, D)
    ([256, 300], 4, 4, 1, 64),                 # the tiny config's shapes
    ([5, 63, 64, 65, 129], 4, 32, 8, 128),    # ragged tails around the tile size
    ([1, 2, 3, 64], 0, 8, 8, 128),             # G = 1, k = 0 (plain decoding), L = 1
    ([9, 10, 200], 8, 64, 8, 128),             # G = 8, k = 8: 72 rows per KV head
    ([2, 3000, 777], 1, 16, 2, 64),            # several splits, D = 64
    ([4100, 70, 1000, 2049], 4, 32, 8, 128),   # splits + ragged
    ([17, 33], 15, 8, 1, 128),                 # 128 rows per KV head (maximum)
    ([100, 260], 2, 6, 2, 128),                # G = 3 (rows not a multiple of 8)
    # past 64 rows per KV head (one query copy)
    ([4100, 70, 1000, 2049, 300], 8, 64, 8, 128),   # 72 rows, many split pairs
    ([700, 64, 1500], 32, 2, 1, 128),          # 66 rows
    ([300, 1200], 16, 4, 1, 128),              # 68 rows
    ([500, 90], 64, 1, 1, 128),                # 65 rows, G = 1
    ([2000, 80], 8, 64, 8, 64),                # 72 rows at D = 64
    ([1000, 129, 64], 9, 64, 8, 128),          # 80 rows
    ([300, 1500, 65], 4, 32, 2, 128),          # 80 rows, G = 16
    ([777, 2100], 4, 32, 2, 64),               # 80 rows, G = 16, D = 64
    ([800, 333], 13, 10, 2, 128),              # 70 rows, G = 5
    ([500, 70, 3000], 11, 16, 2, 128),         # 96 rows
    ([900, 300, 4100], 2, 6, 3, 128),          # 6 rows per KV head (warp-MMA kernel)
    ([300, 1000, 65], 1, 8, 2, 64),            # 8 rows at D = 64 (warp-MMA kernel)
    ([1, 64, 2000], 0, 4, 4, 64),              # decoding, G = 1, D = 64 (warp-MMA kernel)
]


@pytest.mark.parametrize("case", VERIFY_CASES, ids=[str(i) for i in range(len(VERIFY_CASES))])
def test_verify_matches_oracle(spire, case):
    L, k, Hq, Hkv, D = case
    vi = wl.make_verify(L, k, Hq, Hkv, D, seed=100 + len(L), device=DEV, poison=True,
                        spare_pages=3)
    desc = spire.verify_desc(vi.q, vi.k_cache, vi.block_table)
    ws = torch.empty(spire.spire_verify_workspace_bytes(desc, k), dtype=torch.uint8, device=DEV)
    got = spire.verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens, k,
                                 workspace=ws)
    assert spire.spire_get_device_error(ws) == 0
    ref, n_bad = parity.oracle_verify(vi)
    assert n_bad == 0
    parity.assert_close(got.cpu().numpy(), ref, "verify %s" % (case,))


def test_verify_tiny_config(spire):
    cfg = wl.CONFIGS["tiny"]
    vi = wl.make_verify(wl.sample_ctx_lens(cfg), cfg.k, cfg.num_q_heads, cfg.num_kv_heads,
                        cfg.head_dim, seed=cfg.seed, device=DEV, shuffle=False, poison=True)
    got = parity.gpu_verify(spire, vi).cpu().numpy()
    ref, _ = parity.oracle_verify(vi)
    parity.assert_close(got, ref, "tiny verify")


def test_verify_scale(spire):
    vi = wl.make_verify([130, 64], 2, 8, 2, 128, seed=7, device=DEV, q_std=1.0)
    vi.scale = 0.088388
    got = parity.gpu_verify(spire, vi).cpu().numpy()
    ref, _ = parity.oracle_verify(vi)
    parity.assert_close(got, ref, "scaled verify")


def test_verify_page_permutation_bit_exact(spire):
    L = [700, 64, 129]
    a = wl.make_verify(L, 4, 32, 8, 128, seed=9, device=DEV, shuffle=False)
    out_a = parity.gpu_verify(spire, a)
    perm = torch.randperm(a.k_cache.shape[0], generator=torch.Generator().manual_seed(1)).to(DEV)
    inv = torch.argsort(perm)
    bt = torch.where(a.block_table >= 0, inv[a.block_table.clamp(min=0).long()].int(),
                     a.block_table)
    b = wl.VerifyInputs(q=a.q, k_cache=a.k_cache[perm].contiguous(),
                        v_cache=a.v_cache[perm].contiguous(), block_table=bt,
                        ctx_lens=a.ctx_lens, k=a.k)
    out_b = parity.gpu_verify(spire, b)
    assert torch.equal(out_a, out_b)


def test_verify_nan_poison_bit_exact_and_deterministic(spire):
    L = [1000, 65, 5, 5000]
    clean = wl.make_verify(L, 4, 32, 8, 128, seed=11, device=DEV, poison=False, spare_pages=2)
    pois = wl.make_verify(L, 4, 32, 8, 128, seed=11, device=DEV, poison=True, spare_pages=2)
    o1 = parity.gpu_verify(spire, clean)
    o2 = parity.gpu_verify(spire, pois)
    o3 = parity.gpu_verify(spire, pois)
    assert torch.isfinite(o2).all()
    assert torch.equal(o1, o2)
    assert torch.equal(o2, o3)


def test_verify_causality_bit_exact(spire):
    L, k = [777, 64], 4
    vi = wl.make_verify(L, k, 32, 8, 128, seed=13, device=DEV)
    base = parity.gpu_verify(spire, vi)
    for i in range(1, k + 1):
        kc, vc = vi.k_cache.clone(), vi.v_cache.clone()
        for b, Lb in enumerate(L):
            j = Lb - k + i - 1
            page = int(vi.block_table[b, j // 64])
            kc[page, :, j % 64] = 3.0
            vc[page, :, j % 64] = 100.0
        vj = wl.VerifyInputs(q=vi.q, k_cache=kc, v_cache=vc, block_table=vi.block_table,
                             ctx_lens=vi.ctx_lens, k=k)
        out = parity.gpu_verify(spire, vj)
        assert torch.equal(out[:, :i], base[:, :i])
        assert not torch.allclose(out[:, i], base[:, i])


def test_verify_row_equals_decode(spire):
    L, k = [900, 130, 64], 4
    vi = wl.make_verify(L, k, 32, 8, 128, seed=17, device=DEV)
    out = parity.gpu_verify(spire, vi).cpu().numpy()
    for i in range(k + 1):
        di = wl.VerifyInputs(q=vi.q[:, i:i + 1].contiguous(), k_cache=vi.k_cache,
                             v_cache=vi.v_cache, block_table=vi.block_table,
                             ctx_lens=(vi.ctx_lens - k + i).contiguous(), k=0)
        dec = parity.gpu_verify(spire, di).cpu().numpy()
        rel, mx = parity.errors(out[:, i], dec[:, 0])
        assert rel <= 1e-5 and mx <= 1e-5, (i, rel, mx)


def test_verify_constant_v(spire):
    vi = wl.make_verify([300, 5000], 4, 32, 8, 128, seed=19, device=DEV)
    vi.v_cache.fill_(0.8125)
    out = parity.gpu_verify(spire, vi)
    assert torch.allclose(out, torch.full_like(out, 0.8125), rtol=0, atol=1e-6)


def test_verify_device_errors(spire):
    L = [200, 200, 200, 200]
    vi = wl.make_verify(L, 4, 8, 2, 128, seed=23, device=DEV)
    ctx = torch.tensor([200, 3, 200, 10 ** 6], dtype=torch.int32, device=DEV)  # too short / too long
    bt = vi.block_table.clone()
    bt[2, 1] = vi.k_cache.shape[0] + 5                                         # page outside cache
    v2 = wl.VerifyInputs(q=vi.q, k_cache=vi.k_cache, v_cache=vi.v_cache, block_table=bt,
                         ctx_lens=ctx, k=4)
    desc = spire.verify_desc(v2.q, v2.k_cache, v2.block_table)
    ws = torch.empty(spire.spire_verify_workspace_bytes(desc, 4), dtype=torch.uint8, device=DEV)
    out = spire.verify_attention(v2.q, v2.k_cache, v2.v_cache, v2.block_table, v2.ctx_lens, 4,
                                 workspace=ws)
    err = spire.spire_get_device_error(ws)
    assert err == 3, err                   # CTX_LEN | PAGE_ID
    assert torch.isnan(out[1:]).all()
    ref, _ = parity.oracle_verify(vi)
    parity.assert_close(out[0].cpu().numpy(), ref[0], "valid row beside bad ones")
    # a clean call on the same workspace clears the word
    spire.verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens, 4,
                           workspace=ws)
    assert spire.spire_get_device_error(ws) == 0


def test_verify_empty_batch(spire):
    desc = spire.make_desc(0, 8, 2, 128, 64, 4, 4)
    assert spire.spire_verify_attention(0, 0, 0, 0, 0, 4, desc, 0, 0, 0, 0) == 0


# ---------------------------------------------------------------- draft
DRAFT_CASES = [
    # (t, Hq, Hkv, D, n_sink, window)
    ([60, 61, 68, 69, 500], 4, 1, 64, 4, 64),     # tiny config's cache, around capacity
    ([1, 2, 16, 17, 528, 529, 9000], 32, 8, 128, 16, 512),
    ([1, 5, 6, 7, 100], 8, 8, 128, 1, 4),         # S = 5 < one tile
    ([3, 300, 5000], 64, 8, 128, 32, 2048),       # G = 8
    ([10, 20, 4000], 16, 2, 64, 0, 100),          # no sinks
    ([700, 70, 3000], 24, 8, 128, 16, 512),       # G = 3: an odd row count
    ([50, 900, 1300], 14, 2, 128, 4, 200),        # G = 7
]


@pytest.mark.parametrize("case", DRAFT_CASES, ids=[str(i) for i in range(len(DRAFT_CASES))])
def test_draft_matches_oracle(spire, case):
    t, Hq, Hkv, D, ns, w = case
    di = wl.make_draft(t, Hq, Hkv, D, ns, w, seed=200 + len(t), device=DEV, poison=True)
    got = parity.gpu_draft(spire, di).cpu().numpy()
    ref, n_bad = parity.oracle_draft(di)
    assert n_bad == 0
    parity.assert_close(got, ref, "draft %s" % (case,))


def test_draft_window_covers_context_equals_full_attention(spire):
    """window >= t: draft == verify at k = 0 over the same keys laid out as pages."""
    t = [1, 64, 150, 200]
    ns, w, Hq, Hkv, D = 2, 254, 32, 8, 128
    di = wl.make_draft(t, Hq, Hkv, D, ns, w, seed=31, device=DEV)
    dout = parity.gpu_draft(spire, di)
    S = ns + w
    pages = (S + 63) // 64
    B = len(t)
    kc = torch.zeros((B * pages, Hkv, 64, D), dtype=torch.bfloat16, device=DEV)
    vc = torch.zeros_like(kc)
    for b in range(B):
        for p in range(pages):
            lo, hi = p * 64, min(S, (p + 1) * 64)
            kc[b * pages + p, :, :hi - lo] = di.kv[b, 0, :, lo:hi]
            vc[b * pages + p, :, :hi - lo] = di.kv[b, 1, :, lo:hi]
    bt = torch.arange(B * pages, dtype=torch.int32, device=DEV).reshape(B, pages)
    vi = wl.VerifyInputs(q=di.q[:, None].contiguous(), k_cache=kc, v_cache=vc, block_table=bt,
                         ctx_lens=di.ctx_lens, k=0)
    vout = parity.gpu_verify(spire, vi)[:, 0]
    rel, mx = parity.errors(dout.cpu().numpy(), vout.cpu().numpy())
    assert rel <= 1e-5 and mx <= 1e-5


def test_draft_device_error(spire):
    di = wl.make_draft([0, 40], 8, 2, 128, 4, 64, seed=37, device=DEV)
    desc = spire.draft_desc(di.q, di.kv)
    ws = torch.empty(spire.spire_draft_workspace_bytes(desc, 4, 64), dtype=torch.uint8,
                     device=DEV)
    out = spire.draft_attention(di.q, di.kv, di.ctx_lens, 4, 64, workspace=ws)
    assert spire.spire_get_device_error(ws) == 1
    assert torch.isnan(out[0]).all() and torch.isfinite(out[1]).all()


def test_draft_slot_matches_oracle(spire):
    import oracle
    for ns, w in [(0, 1), (4, 64), (16, 512), (32, 2048), (16, 4096)]:
        for p in list(range(0, 3000, 7)) + [10 ** 6 - 1, 262143]:
            assert spire.spire_draft_slot(p, ns, w) == oracle.draft_slot(p, ns, w)


# ---------------------------------------------------------------- zero-copy outputs
def _pinned_like(t):
    return torch.empty(t.shape, dtype=t.dtype, pin_memory=True)


@pytest.mark.parametrize("case", [([700, 5], 0, 8, 8, 128),        # warp-MMA kernel, R = 1
                                  ([4100, 70, 1000], 4, 32, 8, 128),  # tcgen05, four query copies
                                  ([9, 3000, 200], 8, 64, 8, 128)],   # tcgen05, one copy (72 rows)
                         ids=["mma", "tc4", "tc1"])
def test_verify_output_in_pinned_host_memory(spire, case):
    """`out` may be mapped pinned host memory: the kernels store into it
    directly and the result equals the one written to device memory."""
    L, k, Hq, Hkv, D = case
    vi = wl.make_verify(L, k, Hq, Hkv, D, seed=61, device=DEV)
    ref = parity.gpu_verify(spire, vi)
    host = _pinned_like(ref)
    host.fill_(float("nan"))
    spire.verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens, k,
                           softmax_scale=vi.scale, out=host)
    torch.cuda.synchronize()
    assert torch.equal(host, ref.cpu())


def test_draft_and_magicdec_output_in_pinned_host_memory(spire):
    di = wl.make_draft([3, 600, 20000], 32, 8, 128, 16, 512, seed=62, device=DEV)
    ref = spire.draft_attention(di.q, di.kv, di.ctx_lens, 16, 512)
    host = _pinned_like(ref)
    host.fill_(float("nan"))
    spire.draft_attention(di.q, di.kv, di.ctx_lens, 16, 512, out=host)
    torch.cuda.synchronize()
    assert torch.equal(host, ref.cpu())
    for Hq, Hkv in ((32, 8), (64, 1)):          # fused kernel (G <= 8), gather + attention
        vi = wl.make_verify([5, 900, 9000], 0, Hq, Hkv, 128, seed=63, device=DEV)
        q = vi.q[:, 0].contiguous()
        ref = spire.magicdec_attention(q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens,
                                       4, 256, 10000.0)
        host = _pinned_like(ref)
        host.fill_(float("nan"))
        spire.magicdec_attention(q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens, 4, 256,
                                 10000.0, out=host)
        torch.cuda.synchronize()
        assert torch.equal(host, ref.cpu()), (Hq, Hkv)


# ---------------------------------------------------------------- per-CTA timing record
def test_cta_times_cover_every_cta(spire):
    L = [4100, 70, 1000, 2049, 30000, 5]
    for k, Hq, Hkv in ((4, 32, 8), (0, 8, 8)):        # tcgen05 and warp-MMA kernels
        vi = wl.make_verify(L, k, Hq, Hkv, 128, seed=64, device=DEV)
        desc = spire.verify_desc(vi.q, vi.k_cache, vi.block_table)
        nb = spire.spire_verify_workspace_bytes(desc, k)
        ws = torch.full((nb,), 0xff, dtype=torch.uint8, device=DEV)
        spire.verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens, k,
                               workspace=ws)
        t = spire.spire_get_cta_times(ws, nb)
        sms = torch.cuda.get_device_properties(0).multi_processor_count
        assert len(t) == min(sms, 512)
        starts = np.array([a for a, _ in t], dtype=np.float64)
        ends = np.array([b for _, b in t], dtype=np.float64)
        assert np.all(ends >= starts)
        assert ends.max() - starts.min() < 1e9             # one call: well under a second
        with pytest.raises(spire.SpireError):
            spire.spire_get_cta_times(ws, 1024)           # too small for the record
    di = wl.make_draft([3, 600, 20000], 32, 8, 128, 16, 512, seed=65, device=DEV)
    desc = spire.draft_desc(di.q, di.kv)
    nb = spire.spire_draft_workspace_bytes(desc, 16, 512)
    ws = torch.full((nb,), 0xff, dtype=torch.uint8, device=DEV)
    spire.draft_attention(di.q, di.kv, di.ctx_lens, 16, 512, workspace=ws)
    t = spire.spire_get_cta_times(ws, nb)
    assert len(t) >= 1 and all(b >= a for a, b in t)


# ---------------------------------------------------------------- workspace reuse
def test_workspace_needs_no_initialisation_and_survives_reuse(spire):
    """Every call resets the merge counters it uses before its attention
    kernel reads them, so any starting content works and one workspace can
    serve calls of other shapes in turn (ordered on one stream)."""
    L = [30000, 4100, 70]                       # three sequences: every pair is split
    vi = wl.make_verify(L, 4, 32, 8, 128, seed=66, device=DEV)
    di = wl.make_draft([5, 9000, 600, 40, 3000], 32, 8, 128, 16, 512, seed=67, device=DEV)
    ref_v = parity.gpu_verify(spire, vi)
    ref_d = parity.gpu_draft(spire, di)
    vdesc = spire.verify_desc(vi.q, vi.k_cache, vi.block_table)
    ddesc = spire.draft_desc(di.q, di.kv)
    nb = max(spire.spire_verify_workspace_bytes(vdesc, 4),
             spire.spire_draft_workspace_bytes(ddesc, 16, 512))
    g = torch.Generator(device="cpu").manual_seed(68)
    fills = [torch.zeros(nb, dtype=torch.uint8), torch.full((nb,), 255, dtype=torch.uint8),
             torch.randint(0, 256, (nb,), dtype=torch.uint8, generator=g)]
    for fill in fills:
        ws = fill.to(DEV)
        for _ in range(2):
            out = spire.verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table,
                                         vi.ctx_lens, 4, workspace=ws)
            dout = spire.draft_attention(di.q, di.kv, di.ctx_lens, 16, 512, workspace=ws)
            torch.cuda.synchronize()
            assert torch.equal(out, ref_v)
            assert torch.equal(dout, ref_d)
            assert spire.spire_get_device_error(ws) == 0


# ---------------------------------------------------------------- split invariance
def test_split_plan_invariance(spire):
    """The same sequences under different split plans (alone, with a few
    companions, inside a large batch: every call cuts the KV range across
    the SMs differently) agree to fp32 rounding with one another and with the
    oracle.  The caches are shared; only q, the block-table rows and ctx_lens
    of the chosen sequences change."""
    L = [20000, 5000] + [3000] * 40
    vi = wl.make_verify(L, 4, 32, 8, 128, seed=69, device=DEV)
    full = parity.gpu_verify(spire, vi)

    def sub(idx):
        idx_t = torch.as_tensor(idx, dtype=torch.long, device=DEV)
        v = wl.VerifyInputs(q=vi.q[idx_t].contiguous(), k_cache=vi.k_cache, v_cache=vi.v_cache,
                            block_table=vi.block_table[idx_t].contiguous(),
                            ctx_lens=vi.ctx_lens[idx_t].contiguous(), k=vi.k)
        return parity.gpu_verify(spire, v)

    alone = sub([0])
    pair = sub([1, 0])
    ref, _ = parity.oracle_verify(wl.VerifyInputs(
        q=vi.q[:2], k_cache=vi.k_cache, v_cache=vi.v_cache, block_table=vi.block_table[:2],
        ctx_lens=vi.ctx_lens[:2], k=vi.k))
    for got, row in ((full[0], 0), (alone[0], 0), (pair[1], 0), (full[1], 1), (pair[0], 1)):
        parity.assert_close(got.cpu().numpy(), ref[row], "split plan, sequence %d" % row)
    for a, b in ((full[0], alone[0]), (full[0], pair[1]), (full[1], pair[0])):
        rel, mx = parity.errors(a.cpu().numpy(), b.cpu().numpy())
        assert rel <= 1e-5 and mx <= 1e-5, (rel, mx)
    # draft: one sequence alone and inside a batch of 64
    di = wl.make_draft([9000] + [2000] * 63, 32, 8, 128, 16, 512, seed=70, device=DEV)
    dfull = parity.gpu_draft(spire, di)
    d1 = wl.DraftInputs(q=di.q[:1].contiguous(), kv=di.kv[:1].contiguous(),
                        ctx_lens=di.ctx_lens[:1].contiguous(), n_sink=16, window=512)
    done = parity.gpu_draft(spire, d1)
    rel, mx = parity.errors(dfull[0].cpu().numpy(), done[0].cpu().numpy())
    assert rel <= 1e-5 and mx <= 1e-5, (rel, mx)


@pytest.mark.parametrize("case", [(200000, 4, 4, 1), (100000, 8, 8, 1), (150000, 1, 32, 8)],
                         ids=["four-copies", "one-copy", "eight-pairs"])
def test_one_long_sequence_cut_across_every_sm(spire, case):
    """A single sequence (one or a few pairs) cut into ~150 segments: every CTA
    holds a piece of the same pair, and the completing CTA merges them all."""
    L, k, Hq, Hkv = case
    vi = wl.make_verify([L], k, Hq, Hkv, 128, seed=71, device=DEV, poison=True)
    ws = torch.empty(spire.spire_verify_workspace_bytes(spire.verify_desc(vi.q, vi.k_cache,
                                                                          vi.block_table), k),
                     dtype=torch.uint8, device=DEV)
    got = spire.verify_attention(vi.q, vi.k_cache, vi.v_cache, vi.block_table, vi.ctx_lens, k,
                                 workspace=ws)
    assert spire.spire_get_device_error(ws) == 0
    ref, n_bad = parity.oracle_verify(vi)
    assert n_bad == 0
    parity.assert_close(got.cpu().numpy(), ref, "one sequence, %s" % (case,))


def test_draft_one_sequence_cut_into_one_tile_segments(spire):
    """One pair of 8208 slots (129 tiles) over the SMs: a segment per tile."""
    di = wl.make_draft([20000], 4, 1, 128, 16, 8192, seed=72, device=DEV, poison=True)
    got = parity.gpu_draft(spire, di).cpu().numpy()
    ref, n_bad = parity.oracle_draft(di)
    assert n_bad == 0
    parity.assert_close(got, ref, "draft, one sequence of 129 tiles")


# ---------------------------------------------------------------- empty batches
def test_every_call_accepts_an_empty_batch(spire):
    """B = 0 is a no-op for every call: empty results, no device error."""
    bf, f32, i32 = torch.bfloat16, torch.float32, torch.int32
    q = torch.empty((0, 32, 128), dtype=bf, device=DEV)
    kv = torch.empty((0, 2, 8, 528, 128), dtype=bf, device=DEV)
    ctx = torch.empty((0,), dtype=i32, device=DEV)
    assert spire.draft_attention(q, kv, ctx, 16, 512).shape == (0, 32, 128)
    x = torch.empty((3, 0, 256), dtype=bf, device=DEV)
    mix = torch.zeros((2, 3), dtype=f32, device=DEV)
    w = torch.zeros((2, 2 * 2 * 64, 256), dtype=bf, device=DEV)
    cache = torch.empty((2, 0, 2, 2, 7, 64), dtype=bf, device=DEV)
    spire.feedback_append(x, mix, w, torch.empty((0,), dtype=i32, device=DEV), cache, 2, 5)
    p = torch.empty((0, 5, 1000), dtype=f32, device=DEV)
    toks, n_acc = spire.verify_tokens(p, torch.empty((0, 4, 1000), dtype=f32, device=DEV),
                                      torch.empty((0, 4), dtype=i32, device=DEV),
                                      torch.empty((0, 4), dtype=f32, device=DEV),
                                      torch.empty((0, 1000), dtype=f32, device=DEV))
    assert toks.shape == (0, 5) and n_acc.shape == (0,)
    kc = torch.zeros((4, 8, 64, 128), dtype=bf, device=DEV)
    bt = torch.empty((0, 1), dtype=i32, device=DEV)
    assert spire.magicdec_attention(q, kc, kc, bt, ctx, 1, 64, 1e4).shape == (0, 32, 128)
    torch.cuda.synchronize()
