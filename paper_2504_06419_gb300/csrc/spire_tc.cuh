// spire_tc.cuh -- attention kernel on the Blackwell tensor cores (tcgen05,
// accumulators and P in tensor memory).
//
// Roles in a CTA (one CTA per SM, 7 warps):
//   warp 0 (producer)   the TMA producer shared with the warp-MMA kernel:
//                       K/V tiles into an NST-deep stage ring and each pair's
//                       query rows into the Q buffer (one copy).
//   warp 1 (QK issuer)  allocates tensor memory; one thread issues
//                         S[sb]  = Q K^T   (M=128 rows, N=64 keys, K=D)
//   warp 6 (PV issuer)  one thread issues
//                         O     += P V     (M=128, N=D, K=64)
//                       Both use tcgen05.mma with the A operand (Q, P) in
//                       tensor memory and B (K, V tiles) in shared memory and
//                       signal completion with tcgen05.commit.  One thread can
//                       issue an MMA only every ~45 cycles, so QK and PV get a
//                       thread each; they follow the stage ring independently
//                       and the softmax of tile n overlaps QK of tile n+1.
//   warps 2..5          softmax, one thread per tensor-memory lane.
//
// Query copies.  A pair has R = G*(k+1) <= 128 query rows, but the tile has
// 128.  The spare rows are used: the Q buffer holds NC = 128 / (32*ceil(R/32))
// copies of the R rows (NC = 4 for R <= 32, 2 for R <= 64, else 1), and copy c
// is responsible only for keys [c*64/NC, (c+1)*64/NC) of every tile -- its P
// is zero elsewhere.  So each of the four softmax warps handles 64/NC keys per
// tile instead of one warp handling all 64.  Every copy keeps its own running
// max m and sum l (fp32, base 2); at the end of a segment the copies are
// merged through shared memory with weights 2^(m_c - max_c m_c).
//
// Per tile, a softmax thread reads its slice of the S row from tensor memory,
// masks keys past its row's causal / length limit, updates m lazily (only
// when a score exceeds m by more than 2^8, so O is rescaled in tensor memory
// only rarely and P stays <= 2^8), and writes P = P_hi + P_lo (two bf16 parts,
// ~16 mantissa bits together) back to tensor memory.
//
// Tensor memory: S double buffer in columns [0, 128), O in [128, 128 + D),
// P double buffer in [256, 384) (per buffer: 32 columns of packed P_hi, then
// 32 of P_lo; key 2j in the low half of column j), Q double buffer in
// [384, 384 + D) (D/2 packed columns per buffer).  The QK issuer copies each
// pair's query rows from the TMA buffer in shared memory into tensor memory
// with tcgen05.cp (in order with its MMAs), so QK reads only the K tile from
// shared memory and the next pair's QK overlaps this pair's epilogue.  Double buffers let the
// softmax of tile n+1 run while PV of tile n still reads its P.  Every tile,
// bad or not, is acknowledged on its stage's p_full barrier by the softmax
// warps and the QK issuer before the PV issuer releases the stage.
#pragma once

#include "spire_common.cuh"

namespace spire {

template <int D, int NC, int NST>
struct TcCfg {
    static constexpr int THREADS = 224;
    static constexpr int TILE = kPage * D * 2;     // one K (or V) tile
    static constexpr int STAGE = 2 * TILE;
    // one copy of the query rows in shared memory (128 / NC rows of 64 columns
    // per half); tcgen05.cp replicates it into the NC copies in tensor memory
    static constexpr int QROWS = 128 / NC;
    static constexpr int QHALF = QROWS * 128;
    static constexpr int QBUF = (D / 64) * QHALF;
    static constexpr int KW = kPage / NC;          // keys of a tile per copy
    static constexpr int RB = 4 / NC;              // 32-row blocks per copy
    static constexpr int SCR_ROWS = (NC - 1) * 32 * RB;   // rows of copies 1 .. NC-1
    // floats per scratch row; 16-byte chunk q of row t sits at q ^ (t % 8), so
    // the 8 lanes of a 16-byte access phase, one row each, never share a bank
    static constexpr int SCR_LD = 32;
    static constexpr int OFF_Q = NST * STAGE;
    static constexpr int OFF_SCR = OFF_Q + QBUF;   // one Q buffer: copied to TMEM at once
    static constexpr int OFF_ML = OFF_SCR + 2 * SCR_ROWS * SCR_LD * 4;   // two scratch buffers
    static constexpr int OFF_META = OFF_ML + 128 * 8;
    static constexpr int OFF_SCHED = OFF_META + NST * 32;
    static constexpr int OFF_MISC = OFF_SCHED + ((int(sizeof(SchedShared)) + 15) / 16) * 16;
    static constexpr int OFF_BAR = OFF_MISC + 16;
    static constexpr int NBAR = 3 * NST + 15;
    static constexpr int SMEM = OFF_BAR + NBAR * 8 + 1024;   // + alignment slack
    static constexpr uint32_t TMEM_COLS = 512;
    static constexpr int S_COL = 0, O_COL = 128, P_COL = 256, Q_COL = 384;
    static_assert(NC == 1 || NC == 2 || NC == 4, "1, 2 or 4 query copies");
    static_assert(STAGE % 1024 == 0 && OFF_Q % 1024 == 0 && QHALF % 1024 == 0,
                  "swizzled regions must be 1024-byte aligned");
    static_assert(O_COL + D <= P_COL && Q_COL + D <= (int)TMEM_COLS, "tensor memory budget");
};

constexpr float kLazy = 8.0f;   // log2 units: rescale O only when the max grows by > 2^8

template <int D, int NC, int NST, bool kStall = false>
__global__ void __launch_bounds__(224, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmap_k,
                   const __grid_constant__ CUtensorMap tmap_v,
                   const __grid_constant__ CUtensorMap tmap_q, const AttnParams p) {
    using C = TcCfg<D, NC, NST>;
    constexpr int KW = C::KW;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* const sbase = smem_raw + (base - raw);
    int4* const meta = reinterpret_cast<int4*>(sbase + C::OFF_META);
    SchedShared* const sh = reinterpret_cast<SchedShared*>(sbase + C::OFF_SCHED);
    uint32_t* const misc = reinterpret_cast<uint32_t*>(sbase + C::OFF_MISC);  // [0] TMEM base, [1] merge flag
    float* const scr = reinterpret_cast<float*>(sbase + C::OFF_SCR);
    float2* const mls = reinterpret_cast<float2*>(sbase + C::OFF_ML);
    const uint32_t qsm = base + C::OFF_Q;
    const uint32_t bar0 = base + C::OFF_BAR;
    const uint32_t bar_full = bar0, bar_empty = bar0 + 8 * NST, bar_pfull = bar0 + 16 * NST;
    const uint32_t bar_qfull = bar0 + 24 * NST, bar_qempty = bar_qfull + 16;
    const uint32_t bar_sfull = bar_qempty + 16, bar_sfree = bar_sfull + 16;
    const uint32_t bar_obar = bar_sfree + 16;
    const uint32_t bar_grp = bar_obar + 16, bar_drain = bar_grp + 8;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, 1);
            mbar_init(bar_pfull + 8 * s, 5);   // softmax warps and the QK issuer are done with it
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar_qfull + 8 * b, 1);
            mbar_init(bar_qempty + 8 * b, 1);    // the rows were copied into tensor memory
            mbar_init(bar_sfull + 8 * b, 1);
            mbar_init(bar_sfree + 8 * b, 4);
            mbar_init(bar_obar + 8 * b, 1);    // PV reading P buffer b has completed
        }
        mbar_init(bar_grp, 128);
        mbar_init(bar_drain, 1);
        mbar_init(bar_drain + 8, 1);
        fence_barrier_init();
    }
    // Q rows of padding stay zero for the whole kernel
    for (int i = threadIdx.x; i < C::QBUF / 16; i += blockDim.x)
        reinterpret_cast<uint4*>(sbase + C::OFF_Q)[i] = make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async();
    if (warp == 1) {
        tmem_alloc(base + C::OFF_MISC, C::TMEM_COLS);
        tmem_relinquish();
        tc_fence_before();
    }
    // Global memory is touched only after the kernel before (the counter reset,
    // which itself waits for all earlier work) has completed; then the next
    // call's kernels may launch and start their prologue on freed SMs.
    grid_dep_wait();
    grid_dep_launch_dependents();
    if (threadIdx.x == 0) {
        if (blockIdx.x == 0) p.header[0] = gridDim.x;
        p.err[blockIdx.x] = 0;
    }
    sched_setup(p, sh);   // ends with __syncthreads()
    tc_fence_after();
    if (threadIdx.x == 0) p.stamps[2 * blockIdx.x] = globaltimer_ns();
    const uint32_t tmem = misc[0];
    uint32_t err = 0;

    if (warp == 0) {
        // ------------------------------------------------------ producer
        if (lane == 0) {
            // one copy of the query rows: tcgen05.cp replicates them
            const ProducerSmem ps{base, qsm, (uint32_t)C::QHALF, meta, bar_full,
                                  bar_empty, bar_qfull, bar_qempty, 1, 0, 1, false};
            err |= produce<D, NST, kStall>(p, *sh, &tmap_k, &tmap_v, &tmap_q, ps);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------ QK issuer
        if (lane == 0) {
            constexpr uint32_t ID_QK = idesc_bf16(128, 64, false);
            uint32_t st = 0, ph = 0, cq = 0, n_qk = 0;
            int qb = 1;                       // tensor-memory Q buffer of the current segment
            bool have_q = false, ok = true;
            for (;;) {
                if (!mbar_wait(bar_full + 8 * st, ph)) { ok = false; break; }
                const int4 mb = meta[2 * st + 1];
                const int flags = mb.x & 0xff, qflag = mb.x >> 8;
                if (flags & kTerm) break;
                if (flags & kFirst) {
                    have_q = qflag & 16;
                    if (have_q) {
                        // the pair's query rows: the smem TMA buffer -> tensor-memory
                        // buffer qb (two, alternating, so this copy never overwrites
                        // rows that QKs of the previous segment may still read)
                        qb ^= 1;
                        if (!mbar_wait(bar_qfull, cq)) { ok = false; break; }
                        cq ^= 1;
                        tc_fence_after();
                        const uint32_t qaddr = qsm;
                        const uint32_t qdst = tmem + C::Q_COL + qb * (D / 2);
                        if constexpr (NC == 1) {
#pragma unroll
                            for (int ks = 0; ks < D / 16; ++ks)   // 32 bytes of each row
                                tmem_cp_128x256b(qdst + ks * 8,
                                                 sdesc_sw128(qaddr + (ks >> 2) * C::QHALF + (ks & 3) * 32,
                                                             16, 1024));
                        } else {
                            // 16 bytes of each row at a time, into every copy at once
#pragma unroll
                            for (int j = 0; j < D / 8; ++j) {
                                const uint64_t sd =
                                    sdesc_sw128(qaddr + (j >> 3) * C::QHALF + (j & 7) * 16, 16, 1024);
                                if constexpr (NC == 4) tmem_cp_32x128b_x4(qdst + j * 4, sd);
                                else                   tmem_cp_64x128b_x2(qdst + j * 4, sd);
                            }
                        }
                        umma_commit(bar_qempty);   // smem buffer free once copied
                    }
                }
                if (!(flags & kBad)) {
                    const uint32_t sb = n_qk & 1;
                    if (!mbar_wait(bar_sfree + 8 * sb, ((n_qk >> 1) & 1) ^ 1)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t kaddr = base + st * C::STAGE;
                    const uint32_t qcol = tmem + C::Q_COL + qb * (D / 2);
#pragma unroll
                    for (int ks = 0; ks < D / 16; ++ks) {
                        const uint64_t b = sdesc_sw128(kaddr + (ks >> 2) * 8192 + (ks & 3) * 32, 16, 1024);
                        umma_bf16_ts(tmem + C::S_COL + sb * 64, qcol + ks * 8, b, ID_QK, ks > 0);
                    }
                    umma_commit(bar_sfull + 8 * sb);
                    ++n_qk;
                }
                mbar_arrive(bar_pfull + 8 * st);   // done with this stage's meta and K tile
                if (++st == NST) { st = 0; ph ^= 1; }
            }
            if (!ok) err |= kErrTimeout;
            // every issued tensor-core operation has finished before TMEM is freed
            umma_commit(bar_drain);
            if (!mbar_wait(bar_drain, 0)) err |= kErrTimeout;
        }
        __syncwarp();
    } else if (warp == 6) {
        // ------------------------------------------------------ PV issuer
        if (lane == 0) {
            constexpr uint32_t ID_PV = idesc_bf16(128, D, true);
            uint32_t st = 0, ph = 0, n_pv = 0;
            int seg_nonbad = 0;
            bool ok = true;
            for (;;) {
                if (!mbar_wait(bar_full + 8 * st, ph)) { ok = false; break; }
                const int flags = meta[2 * st + 1].x & 0xff;
                if (flags & kTerm) break;
                if (flags & kFirst) seg_nonbad = 0;
                // P written (or the tile acknowledged) by all its readers
                if (!mbar_wait(bar_pfull + 8 * st, ph)) { ok = false; break; }
                tc_fence_after();
                if (!(flags & kBad)) {
                    const uint32_t accum = seg_nonbad > 0;   // first PV of a segment overwrites O
                    ++seg_nonbad;
                    const uint32_t vaddr = base + st * C::STAGE + C::TILE;
                    const uint32_t pcol = tmem + C::P_COL + (n_pv & 1) * 64;
#pragma unroll
                    for (int part = 0; part < 2; ++part) {        // P_hi, then P_lo
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {
                            const uint64_t b = sdesc_sw128(vaddr + kk * 2048, 8192, 1024);
                            umma_bf16_ts(tmem + C::O_COL, pcol + part * 32 + kk * 8, b, ID_PV,
                                         (accum | part | kk) != 0);
                        }
                    }
                    umma_commit(bar_obar + 8 * (n_pv & 1));
                    umma_commit(bar_empty + 8 * st);
                    ++n_pv;
                } else {
                    mbar_arrive(bar_empty + 8 * st);
                }
                if (++st == NST) { st = 0; ph ^= 1; }
            }
            if (!ok) err |= kErrTimeout;
            umma_commit(bar_drain + 8);
            if (!mbar_wait(bar_drain + 8, 0)) err |= kErrTimeout;
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------ softmax warps
        const int quarter = warp & 3;                 // TMEM lanes 32*quarter .. +31
        const int tl = 32 * quarter + lane;           // this thread's TMEM lane
        const int copy = quarter / C::RB;             // query copy (key slice) of the lane
        const int r = 32 * (quarter % C::RB) + lane;  // query row within the copy
        const bool active = 32 * (quarter % C::RB) < p.R;   // warp holds a real row
        const uint32_t trow = tmem + ((uint32_t)(32 * quarter) << 16);
        const int gtid = threadIdx.x - 64;            // 0..127
        const float NEG_INF = __int_as_float(0xff800000);
        const float NANF = __int_as_float(0x7fc00000);
        const float sl2 = p.sl2;
        const int i_r = min(r / p.G, p.kp1 - 1);      // block row of query row r
        const int kofs = copy * KW;                   // first key of this copy's slice
        uint32_t st = 0, ph = 0, n_qk = 0, n_pv = 0, gph = 0;
        float m = NEG_INF, l = 0.f;
        bool poison = false;
        int seg_pv = 0;
        int cur_b = 0, cur_g = 0, cur_slot = 0, cur_nseg = 1, cur_first = 0, leff = 0, lim = 0;
        bool ok = true;
        auto grp_sync = [&]() -> bool {
            mbar_arrive(bar_grp);
            const bool rr = mbar_wait(bar_grp, gph & 1);
            ++gph;
            return rr;
        };
        // P columns outside this copy's key slice stay zero
        {
            uint32_t z[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) z[j] = 0u;
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_st32u(trow + C::P_COL + 32 * c, z);
            tmem_wait_st();
        }
        for (;;) {
            if (!mbar_wait(bar_full + 8 * st, ph)) { ok = false; break; }
            const int4 ma = meta[2 * st], mb = meta[2 * st + 1];
            const int flags = mb.x & 0xff;
            if (flags & kTerm) break;
            if (flags & kFirst) {
                cur_b = ma.x; cur_g = ma.y; leff = ma.w;
                cur_slot = mb.y; cur_nseg = mb.z; cur_first = mb.w;
                m = NEG_INF; l = 0.f; poison = false; seg_pv = 0;
                lim = leff - (p.kp1 - 1) + i_r;
            }
            if (flags & kBad) {
                poison = true;
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_pfull + 8 * st);   // meta read: the stage may be reused
            } else {
                const int key0 = ma.z + kofs;                // first key of this slice
                const uint32_t sb = n_qk & 1;
                if (!mbar_wait(bar_sfull + 8 * sb, (n_qk >> 1) & 1)) { ok = false; break; }
                tc_fence_after();
                float sv[KW];
                // this thread's slice of the S row, with keys past the row's causal /
                // length limit masked
                auto load_scores = [&]() {
                    if constexpr (KW == 16) {
                        tmem_ld16(trow + C::S_COL + sb * 64 + kofs, sv);
                    } else {
#pragma unroll
                        for (int h = 0; h < KW / 32; ++h) {
                            float t[32];
                            tmem_ld32(trow + C::S_COL + sb * 64 + kofs + 32 * h, t);
#pragma unroll
                            for (int j = 0; j < 32; ++j) sv[32 * h + j] = t[j];
                        }
                    }
                    tmem_wait_ld();
                    if (key0 + KW > lim) {
#pragma unroll
                        for (int j = 0; j < KW; ++j)
                            if (key0 + j >= lim) sv[j] = NEG_INF;
                    }
                };
                // exponentials 2^(s sl2 - mr) in place and their sum, two lanes at a time
                auto exponentials = [&](float mr) -> float {
                    const uint64_t scale2 = f2_pack(sl2, sl2), shift2 = f2_pack(-mr, -mr);
                    uint64_t sp[4];
#pragma unroll
                    for (int j = 0; j < 4; ++j) sp[j] = 0ull;
#pragma unroll
                    for (int j = 0; j < KW / 2; ++j) {
                        float x, y;
                        f2_unpack(fma2(f2_pack(sv[2 * j], sv[2 * j + 1]), scale2, shift2), x, y);
                        sv[2 * j] = ex2(x);
                        sv[2 * j + 1] = ex2(y);
                        sp[j & 3] = add2(sp[j & 3], f2_pack(sv[2 * j], sv[2 * j + 1]));
                    }
                    float x, y;
                    f2_unpack(add2(add2(sp[0], sp[1]), add2(sp[2], sp[3])), x, y);
                    return x + y;
                };
                // With one copy (64 keys a thread) the row maximum is a tenth of
                // the per-tile work, so it is skipped where it cannot matter (fast
                // path below) and the S buffer is released only after the
                // exponentials, so that a warp can reload its scores.  With more
                // copies (16 or 32 keys a thread) the maximum is cheap and the
                // buffer is released at once, so the QK two tiles ahead never waits.
                constexpr bool kFast = (KW == 64);
                if (active) load_scores();
                if (!kFast) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(bar_sfree + 8 * sb);   // S buffer read
                }
                float factor = 1.f;
                if (active) {
                    // Fast path: exponentials against the running max m as it
                    // stands.  The max only moves when a score exceeds m by more
                    // than 2^8 (lazy rescaling), which makes some exponential
                    // > 2^8; a sum <= 2^8 rules that out, so m stays and these
                    // are exactly the values the max-first path below computes.
                    // Otherwise (the first tile of a segment, a sum above 2^8,
                    // NaN) the warp takes that path, after reloading its scores
                    // (tensor-memory loads are warp-wide).
                    float sum = 0.f;
                    bool slow = !kFast || (m == NEG_INF);
                    if (!slow) {
                        sum = exponentials(m);
                        slow = !(sum <= 256.f);           // 2^kLazy
                    }
                    if (!kFast || __any_sync(0xffffffffu, slow)) {
                        if (kFast && __any_sync(0xffffffffu, m != NEG_INF)) load_scores();
                        // independent partial maxima (three-input max) keep the chain short
                        constexpr int NP = KW / 8;        // partials of 8 scores each
                        float mp[NP];
#pragma unroll
                        for (int j = 0; j < NP; ++j) {
                            const float* v = sv + 8 * j;
                            mp[j] = fmaxf(fmax3(fmax3(v[0], v[1], v[2]), v[3], v[4]),
                                          fmax3(v[5], v[6], v[7]));
                        }
#pragma unroll
                        for (int w = NP / 2; w > 0; w /= 2)
#pragma unroll
                            for (int j = 0; j < w; ++j) mp[j] = fmaxf(mp[j], mp[j + w]);
                        const float t = mp[0] * sl2;
                        if (t > m + kLazy) {              // also true while m is -inf
                            factor = ex2(m - t);          // 0 when m is -inf
                            l *= factor;
                            m = t;
                        }
                        sum = exponentials((m == NEG_INF) ? 0.f : m);
                    }
                    l += sum;
                }
                if (kFast) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(bar_sfree + 8 * sb);   // S buffer read
                }
                ++n_qk;
                const uint32_t pb = n_pv & 1;
                if (active) {
                    // PV two tiles back read this P buffer: it must have completed
                    if (n_pv >= 2 && !mbar_wait(bar_obar + 8 * pb, ((n_pv - 2) >> 1) & 1)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    // key 2j of the slice in the low half of its column, 2j+1 in the high
                    // half; packed and stored 16 or 32 keys at a time
                    constexpr int PK = KW < 32 ? KW : 32;
                    const uint32_t pc = trow + C::P_COL + pb * 64 + kofs / 2;
#pragma unroll
                    for (int h = 0; h < KW / PK; ++h) {
                        uint32_t hi[PK / 2], lo[PK / 2];
#pragma unroll
                        for (int j = 0; j < PK / 2; ++j) {
                            const float a = sv[PK * h + 2 * j], b = sv[PK * h + 2 * j + 1];
                            hi[j] = pack_bf16(a, b);
                            float ra, rb;   // the parts bf16 rounding dropped
                            f2_unpack(sub2(f2_pack(a, b), f2_pack(bf16lo_to_f32(hi[j]), bf16hi_to_f32(hi[j]))),
                                      ra, rb);
                            lo[j] = pack_bf16(ra, rb);
                        }
                        if constexpr (PK == 16) {
                            tmem_st8u(pc + 8 * h, hi);
                            tmem_st8u(pc + 32 + 8 * h, lo);
                        } else {
                            tmem_st16u(pc + 16 * h, hi);
                            tmem_st16u(pc + 32 + 16 * h, lo);
                        }
                    }
                    tmem_wait_st();
                    if (seg_pv > 0 && __any_sync(0xffffffffu, factor != 1.f)) {
                        // rescale this row of O in tensor memory once the last PV is done;
                        // after the P store, so the exponentials are no longer live (PV of
                        // this tile waits for p_full, signalled after this)
                        if (!mbar_wait(bar_obar + 8 * (pb ^ 1), ((n_pv - 1) >> 1) & 1)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
#pragma unroll
                        for (int c = 0; c < D / 32; ++c) {
                            float ov[32];
                            tmem_ld32(trow + C::O_COL + 32 * c, ov);
                            tmem_wait_ld();
#pragma unroll
                            for (int j = 0; j < 32; ++j) ov[j] *= factor;
                            tmem_st32(trow + C::O_COL + 32 * c, ov);
                        }
                        tmem_wait_st();
                    }
                }
                if (ma.z + kPage > leff && tl < kPage && ma.z + tl >= leff) {
                    // V rows of keys no query may see: their slots may hold anything
                    uint8_t* const vt = sbase + st * C::STAGE + C::TILE + tl * 128;
#pragma unroll
                    for (int h = 0; h < D / 64; ++h)
#pragma unroll
                        for (int c = 0; c < 8; ++c)
                            *reinterpret_cast<uint4*>(vt + h * 8192 + 16 * c) = make_uint4(0u, 0u, 0u, 0u);
                    fence_proxy_async();   // the zeros before the tensor core reads V
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_pfull + 8 * st);
                ++n_pv;
                ++seg_pv;
            }
            if (flags & kLast) {
                // ---- segment end: merge the copies, write the output or a partial
                if (active && seg_pv > 0 &&
                    !mbar_wait(bar_obar + 8 * ((n_pv - 1) & 1), ((n_pv - 1) >> 1) & 1)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                // weight of this copy: 2^(m_copy - M) with M the max over copies
                if (NC > 1) {
                    mls[tl] = make_float2(m, l);
                    if (!grp_sync()) { ok = false; break; }
                }
                float wgt, inv, lse;
                {
                    float M = NEG_INF;
#pragma unroll
                    for (int c = 0; c < NC; ++c) M = fmaxf(M, NC > 1 ? mls[32 * C::RB * c + r].x : m);
                    const float Mr = (M == NEG_INF) ? 0.f : M;
                    float L = 0.f;
#pragma unroll
                    for (int c = 0; c < NC; ++c) {
                        const float2 v = NC > 1 ? mls[32 * C::RB * c + r] : make_float2(m, l);
                        L += ex2(v.x - Mr) * v.y;
                    }
                    wgt = ex2(m - Mr);
                    inv = (L > 0.f) ? 1.f / L : 0.f;
                    lse = (L > 0.f) ? M + __log2f(L) : NEG_INF;
                }
                const bool nan = poison || seg_pv == 0;
                float* dst = nullptr;
                if (copy == 0 && r < p.R)
                    dst = cur_nseg == 1 ? out_row(p, cur_b, cur_g, r, D)
                                        : p.part_o + ((long long)cur_slot * p.R + r) * D;
#pragma unroll 1
                for (int c = 0; c < D / 32; ++c) {
                    float ov[32];
                    if (active) {
                        tmem_ld32(trow + C::O_COL + 32 * c, ov);
                        tmem_wait_ld();
                    }
                    float* const sc = scr + (c & 1) * C::SCR_ROWS * C::SCR_LD;
                    if (NC > 1) {
                        if (copy > 0 && active) {
                            float4* const row =
                                reinterpret_cast<float4*>(sc + (tl - 32 * C::RB) * C::SCR_LD);
#pragma unroll
                            for (int q = 0; q < 8; ++q)
                                row[q ^ (lane & 7)] = make_float4(ov[4 * q] * wgt, ov[4 * q + 1] * wgt,
                                                                  ov[4 * q + 2] * wgt, ov[4 * q + 3] * wgt);
                        }
                        if (!grp_sync()) { ok = false; break; }
                    }
                    if (dst) {
#pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            float4 acc = make_float4(ov[4 * q] * wgt, ov[4 * q + 1] * wgt,
                                                     ov[4 * q + 2] * wgt, ov[4 * q + 3] * wgt);
#pragma unroll
                            for (int cc = 1; cc < NC; ++cc) {
                                const float4 o2 = reinterpret_cast<const float4*>(
                                    sc + (32 * C::RB * (cc - 1) + r) * C::SCR_LD)[q ^ (lane & 7)];
                                acc.x += o2.x; acc.y += o2.y; acc.z += o2.z; acc.w += o2.w;
                            }
                            ov[4 * q] = acc.x * inv;
                            ov[4 * q + 1] = acc.y * inv;
                            ov[4 * q + 2] = acc.z * inv;
                            ov[4 * q + 3] = acc.w * inv;
                        }
#pragma unroll
                        for (int j = 0; j < 32; j += 4) {
                            const float4 v = nan ? make_float4(NANF, NANF, NANF, NANF)
                                                 : make_float4(ov[j], ov[j + 1], ov[j + 2], ov[j + 3]);
                            *reinterpret_cast<float4*>(dst + 32 * c + j) = v;
                        }
                    }
                }
                if (!ok) break;
                if (dst && cur_nseg > 1) p.part_lse[(long long)cur_slot * p.R + r] = nan ? NANF : lse;
                tc_fence_before();
                if (cur_nseg > 1) {
                    // publish this segment; the CTA completing the pair merges it
                    __threadfence();
                    if (!grp_sync()) { ok = false; break; }
                    if (gtid == 0) {
                        const int old = atomicAdd(p.cnt + cur_b * p.Hkv + cur_g, 1);
                        misc[1] = (old == cur_nseg - 1);
                    }
                    if (!grp_sync()) { ok = false; break; }
                    if (misc[1]) {
                        __threadfence();
                        merge_pair<D>(p, cur_b, cur_g, cur_nseg, cur_first, gtid, 128);
                    }
                }
            }
            if (++st == NST) { st = 0; ph ^= 1; }
        }
        if (!ok) err |= kErrTimeout;
    }
    if (err) atomicOr(&p.err[blockIdx.x], (int)err);
    __syncthreads();
    if (threadIdx.x == 0) p.stamps[2 * blockIdx.x + 1] = globaltimer_ns();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

}  // namespace spire
