// spire_mma.cuh -- attention kernel on the warp-level tensor-core path
// (mma.sync m16n8k16, bf16 in / fp32 accumulate).
//
// Roles in a CTA (one CTA per SM):
//   warp NW (producer)  lane 0 walks the CTA's tile range, translates pages
//                       through the block table, and streams each K and V
//                       tile with TMA (64 keys x D, 128-byte swizzle) into
//                       an NST-deep ring of shared-memory stages.
//   warps 0..NW-1       consumer warp w owns m-tile w / KP (16 query rows)
//                       and key slice w % KP (64 / KP keys of every tile).
//                       It keeps Q in registers for the current pair, runs
//                       S = Q K^T and O += P V on the tensor cores and an
//                       fp32 online softmax in base 2.
//   warp NW+1 (epilogue) at the end of a pair's segment the consumers only
//                       hand their (O, m, l) rows to one of two shared-memory
//                       buffers and go on with the next segment; this warp
//                       merges the KP key slices and writes the result to the
//                       output, or to a partial slot that the last-arriving
//                       CTA merges (see spire_common.cuh), publishing with a
//                       fence and an atomic, off the consumers' path.
// The kernel serves pairs of at most 8 query rows (one m-tile, rows 8..15 of
// the MMA are padding), so a buffer holds 8 rows per consumer warp.
//
// Precision: P enters the PV product as P_hi + P_lo, two bf16 terms carrying
// ~16 mantissa bits, so rounding P to bf16 (~1.7e-3 rms relative) never
// reaches the output.
#pragma once

#include "spire_common.cuh"

namespace spire {

template <int D, int MT, int KP, int NST>
struct MmaCfg {
    static constexpr int NW = MT * KP;            // consumer warps
    static constexpr int THREADS = 32 * (NW + 2); // + a producer and an epilogue warp
    static constexpr int KW = kPage / KP;         // keys per consumer warp per tile
    static constexpr int NT = KW / 8;             // S n-tiles per warp
    static constexpr int KK = KW / 16;            // PV k-steps per warp
    static constexpr int TILE = kPage * D * 2;    // bytes of one K (or V) tile
    static constexpr int STAGE = 2 * TILE;
    static constexpr int SCR = D + 8;             // floats per scratch row
    static constexpr int SR = 8;                  // scratch rows per warp (R <= 8)
    static constexpr int SCR_BUF = NW * SR * SCR; // floats of one hand-over buffer
    static constexpr int OFF_SCR_O = NST * STAGE;                  // [2][NW][SR][SCR]
    static constexpr int OFF_SCR_ML = OFF_SCR_O + 2 * SCR_BUF * 4; // [2][NW][SR] float2
    static constexpr int OFF_SCR_INFO = OFF_SCR_ML + 2 * NW * SR * 8;   // [2] int4 x 2
    static constexpr int QHALF = MT * 16 * 128;         // one 64-column half of a Q buffer
    static constexpr int QBUF = (D / 64) * QHALF;       // Q of one pair (rows padded to MT*16)
    static constexpr int OFF_Q = ((OFF_SCR_INFO + 2 * 32 + 1023) / 1024) * 1024;
    static constexpr int OFF_META = OFF_Q + 2 * QBUF;
    static constexpr int OFF_SCHED = OFF_META + NST * 32;
    static constexpr int OFF_BAR = OFF_SCHED + ((int(sizeof(SchedShared)) + 15) / 16) * 16 + 16;
    static constexpr int SMEM = OFF_BAR + (2 * NST + 9) * 8 + 1024;  // + alignment slack
    static_assert(KW >= 16 && NT % 2 == 0, "each warp needs >= 16 keys of a tile");
    static_assert(MT == 1, "one m-tile: the kernel serves at most 8 query rows");
    static_assert(D % 64 == 0, "head_dim must be a multiple of 64");
    // 128-byte swizzled TMA destinations must sit on 1024-byte boundaries
    static_assert(STAGE % 1024 == 0 && OFF_Q % 1024 == 0 && QHALF % 1024 == 0,
                  "swizzled regions must be 1024-byte aligned");
};

template <int D, int MT, int KP, int NST, bool kStall = false>
__global__ void __launch_bounds__(MmaCfg<D, MT, KP, NST>::THREADS, 1)
    attn_mma_kernel(const __grid_constant__ CUtensorMap tmap_k,
                    const __grid_constant__ CUtensorMap tmap_v,
                    const __grid_constant__ CUtensorMap tmap_q, const AttnParams p) {
    using C = MmaCfg<D, MT, KP, NST>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* const sbase = smem_raw + (base - raw);
    float* const scr_o = reinterpret_cast<float*>(sbase + C::OFF_SCR_O);
    float2* const scr_ml = reinterpret_cast<float2*>(sbase + C::OFF_SCR_ML);
    int4* const meta = reinterpret_cast<int4*>(sbase + C::OFF_META);
    SchedShared* const sh = reinterpret_cast<SchedShared*>(sbase + C::OFF_SCHED);
    const uint32_t bar_full = base + C::OFF_BAR;          // NST barriers
    const uint32_t bar_empty = bar_full + NST * 8;         // NST barriers
    const uint32_t bar_qfull = bar_empty + NST * 8;        // 2 barriers: Q buffer landed
    const uint32_t bar_qempty = bar_qfull + 16;            // 2 barriers: Q buffer read
    const uint32_t bar_sfull = bar_qempty + 16;            // 2: a hand-over buffer was filled
    const uint32_t bar_sempty = bar_sfull + 16;            // 2: the epilogue is done with it
    int4* const scr_info = reinterpret_cast<int4*>(sbase + C::OFF_SCR_INFO);
    const uint32_t qsm = base + C::OFF_Q;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, C::NW);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar_qfull + 8 * b, 1);
            mbar_init(bar_qempty + 8 * b, C::NW);
            mbar_init(bar_sfull + 8 * b, C::NW);
            mbar_init(bar_sempty + 8 * b, 1);
        }
        fence_barrier_init();
    }
    // Q rows past R are never loaded: keep them zero for the whole kernel
    for (int i = threadIdx.x; i < 2 * C::QBUF / 16; i += blockDim.x)
        reinterpret_cast<uint4*>(sbase + C::OFF_Q)[i] = make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async();
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
    if (threadIdx.x == 0) p.stamps[2 * blockIdx.x] = globaltimer_ns();

    if (warp == C::NW) {
        // ------------------------------------------------------ producer
        if (lane != 0) return;
        const ProducerSmem psm{base, qsm, (uint32_t)C::QHALF, meta, bar_full,
                               bar_empty, bar_qfull, bar_qempty, 1, 0, 2, true};
        const uint32_t err = produce<D, NST, kStall>(p, *sh, &tmap_k, &tmap_v, &tmap_q, psm);
        if (err) atomicOr(&p.err[blockIdx.x], (int)err);
        return;
    }
    if (warp == C::NW + 1) {
        // ------------------------------------------------------ epilogue
        const float NEG_INF = __int_as_float(0xff800000);
        const float NANF = __int_as_float(0x7fc00000);
        constexpr int D4 = D / 4;
        for (uint32_t n = 0;; ++n) {
            const int sb = n & 1;
            if (!mbar_wait(bar_sfull + 8 * sb, (n >> 1) & 1)) {
                if (lane == 0) atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
                return;
            }
            const int4 i0 = scr_info[2 * sb], i1 = scr_info[2 * sb + 1];
            if (i1.y) {                                // the consumers have finished
                if (lane == 0) p.stamps[2 * blockIdx.x + 1] = globaltimer_ns();
                return;
            }
            const int cb = i0.x, cg = i0.y, cslot = i0.z, cnseg = i0.w, cfirst = i1.x;
            const float* so = scr_o + sb * C::SCR_BUF;
            const float2* sml = scr_ml + sb * C::NW * C::SR;
            for (int idx = lane; idx < p.R * D4; idx += 32) {
                const int r = idx / D4, d4 = idx - r * D4;
                float M = NEG_INF;
                bool nan = false;
#pragma unroll
                for (int kq = 0; kq < KP; ++kq) {
                    const float mk = sml[kq * C::SR + r].x;
                    nan |= (mk != mk);
                    M = fmaxf(M, mk);
                }
                const float Mr = (M == NEG_INF) ? 0.f : M;
                float lsum = 0.f;
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int kq = 0; kq < KP; ++kq) {
                    const float2 ml = sml[kq * C::SR + r];
                    const float wgt = ex2(ml.x - Mr);
                    lsum += wgt * ml.y;
                    const float4 ov =
                        *reinterpret_cast<const float4*>(so + (kq * C::SR + r) * C::SCR + 4 * d4);
                    acc.x += wgt * ov.x; acc.y += wgt * ov.y;
                    acc.z += wgt * ov.z; acc.w += wgt * ov.w;
                }
                float4 res;
                float lse;
                if (nan) {
                    res = make_float4(NANF, NANF, NANF, NANF);
                    lse = NANF;
                } else if (lsum > 0.f) {
                    const float inv = 1.f / lsum;
                    res = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
                    lse = M + __log2f(lsum);
                } else {  // no key of this segment is visible to this row
                    res = make_float4(0.f, 0.f, 0.f, 0.f);
                    lse = NEG_INF;
                }
                if (cnseg == 1) {
                    *reinterpret_cast<float4*>(out_row(p, cb, cg, r, D) + 4 * d4) = res;
                } else {
                    const long long row = (long long)cslot * p.R + r;
                    *reinterpret_cast<float4*>(p.part_o + row * D + 4 * d4) = res;
                    if (d4 == 0) p.part_lse[row] = lse;
                }
            }
            __syncwarp();
            // the buffer is read: the consumers may fill it again
            if (lane == 0) mbar_arrive(bar_sempty + 8 * sb);
            if (cnseg > 1) {
                // publish this segment; the CTA completing the pair merges it
                __threadfence();
                __syncwarp();
                int last = 0;
                if (lane == 0) last = atomicAdd(p.cnt + cb * p.Hkv + cg, 1) == cnseg - 1;
                last = __shfl_sync(0xffffffffu, last, 0);
                if (last) {
                    __threadfence();
                    merge_pair<D>(p, cb, cg, cnseg, cfirst, lane, 32);
                }
            }
        }
    }

    // ---------------------------------------------------------- consumers
    const int mt = warp / KP, kp = warp - (warp / KP) * KP;
    const int gq = lane >> 2, tq = lane & 3;          // mma group / thread-in-group
    const int r0 = mt * 16 + gq, r1 = r0 + 8;         // the two rows this thread holds
    const int wkey = kp * C::KW;                      // first key of this warp in a tile
    const float sl2 = p.sl2;
    const float NEG_INF = __int_as_float(0xff800000);
    const float NANF = __int_as_float(0x7fc00000);

    float o[D / 8][4];
    uint32_t qf[D / 16][4];
    float m0 = NEG_INF, m1 = NEG_INF, l0 = 0.f, l1 = 0.f;
    bool poison = false;
    int cur_b = 0, cur_g = 0, cur_slot = 0, cur_nseg = 1, cur_first = 0;
    int lim0 = 0, lim1 = 0, leff = 0;
    uint32_t st = 0, ph = 0, n_seg = 0;               // stage ring / segments handed over
    uint32_t cq[2] = {0u, 0u};                        // parity of each Q buffer

    // hand the segment's (O, m, l) rows, or the end of the work, to the epilogue
    // warp through buffer n_seg & 1 (rows r0 = gq < 8 only: rows 8..15 are padding)
    auto hand_over = [&](bool term, float lt0) -> bool {
        const int sb = n_seg & 1;
        if (!mbar_wait(bar_sempty + 8 * sb, ((n_seg >> 1) & 1) ^ 1)) return false;
        if (!term) {
            float* so = scr_o + sb * C::SCR_BUF + (warp * C::SR + gq) * C::SCR;
#pragma unroll
            for (int j = 0; j < D / 8; ++j)
                *reinterpret_cast<float2*>(so + 8 * j + 2 * tq) = make_float2(o[j][0], o[j][1]);
            if (tq == 0)
                scr_ml[sb * C::NW * C::SR + warp * C::SR + gq] =
                    make_float2(poison ? NANF : m0, lt0);
        }
        if (warp == 0 && lane == 0) {
            scr_info[2 * sb] = make_int4(cur_b, cur_g, cur_slot, cur_nseg);
            scr_info[2 * sb + 1] = make_int4(cur_first, term ? 1 : 0, 0, 0);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar_sfull + 8 * sb);
        ++n_seg;
        return true;
    };

    for (;;) {
        if (!mbar_wait(bar_full + 8 * st, ph)) {
            if (lane == 0) atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
            return;
        }
        const int4 ma = meta[2 * st], mb = meta[2 * st + 1];
        const int flags = mb.x & 0xff;
        if (flags & kTerm) {
            if (!hand_over(true, 0.f) && lane == 0) atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
            return;
        }
        if (flags & kFirst) {
            const int flags_q = mb.x;
            cur_b = ma.x; cur_g = ma.y; leff = ma.w;
            cur_slot = mb.y; cur_nseg = mb.z; cur_first = mb.w;
            poison = false;
            m0 = m1 = NEG_INF; l0 = l1 = 0.f;
#pragma unroll
            for (int j = 0; j < D / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
            // rows r = i*G + hl (block row i, head hl of the group)
            const int i0 = min(r0 / p.G, p.kp1 - 1), i1 = min(r1 / p.G, p.kp1 - 1);
            lim0 = leff - (p.kp1 - 1) + i0;
            lim1 = leff - (p.kp1 - 1) + i1;
            const int qflag = flags_q >> 8;
            if (qflag & 16) {
                const int qb = qflag & 1;
                if (!mbar_wait(bar_qfull + 8 * qb, cq[qb])) {
                    if (lane == 0) atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
                    return;
                }
                cq[qb] ^= 1;
                const uint32_t qbase = qsm + qb * C::QBUF;
                const int qrow = mt * 16 + ((lane >> 3) & 1) * 8 + (lane & 7);
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks) {
                    const int chunk = 2 * ks + (lane >> 4);
                    ldsm_x4(qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3],
                            qbase + (chunk >> 3) * C::QHALF + qrow * 128 +
                                (((chunk & 7) ^ (lane & 7)) << 4));
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_qempty + 8 * qb);
            }
        }
        if (flags & kBad) {
            poison = true;
        } else {
            const int key0 = ma.z;                           // sequence index of tile key 0
            const uint32_t kb = base + st * C::STAGE, vb = kb + C::TILE;
            // ---- S = Q K^T over this warp's KW keys
            float s[C::NT][4];
#pragma unroll
            for (int j = 0; j < C::NT; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
#pragma unroll
                for (int jp = 0; jp < C::NT / 2; ++jp) {
                    const int key = wkey + jp * 16 + ((lane >> 4) << 3) + (lane & 7);
                    const int chunk = 2 * ks + ((lane >> 3) & 1);
                    const uint32_t addr = kb + (chunk >> 3) * 8192 + key * 128 +
                                          (((chunk & 7) ^ (lane & 7)) << 4);
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4(b0, b1, b2, b3, addr);
                    mma_bf16(s[2 * jp], qf[ks], b0, b1);
                    mma_bf16(s[2 * jp + 1], qf[ks], b2, b3);
                }
            }
            // ---- causal / length mask (only tiles reaching past row 0's limit)
            if (key0 + kPage > leff - (p.kp1 - 1)) {
#pragma unroll
                for (int j = 0; j < C::NT; ++j) {
                    const int kidx = key0 + wkey + 8 * j + 2 * tq;
                    if (kidx >= lim0) s[j][0] = NEG_INF;
                    if (kidx + 1 >= lim0) s[j][1] = NEG_INF;
                    if (kidx >= lim1) s[j][2] = NEG_INF;
                    if (kidx + 1 >= lim1) s[j][3] = NEG_INF;
                }
            }
            // ---- online softmax (base 2)
            float mx0 = NEG_INF, mx1 = NEG_INF;
#pragma unroll
            for (int j = 0; j < C::NT; ++j) {
                mx0 = fmaxf(mx0, fmaxf(s[j][0], s[j][1]));
                mx1 = fmaxf(mx1, fmaxf(s[j][2], s[j][3]));
            }
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
            const float mn0 = fmaxf(m0, mx0 * sl2), mn1 = fmaxf(m1, mx1 * sl2);
            const float mr0 = (mn0 == NEG_INF) ? 0.f : mn0;
            const float mr1 = (mn1 == NEG_INF) ? 0.f : mn1;
            const float a0 = ex2(m0 - mr0), a1 = ex2(m1 - mr1);
            m0 = mn0; m1 = mn1;
            float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
            for (int j = 0; j < C::NT; ++j) {
                s[j][0] = ex2(fmaf(s[j][0], sl2, -mr0));
                s[j][1] = ex2(fmaf(s[j][1], sl2, -mr0));
                s[j][2] = ex2(fmaf(s[j][2], sl2, -mr1));
                s[j][3] = ex2(fmaf(s[j][3], sl2, -mr1));
                rs0 += s[j][0] + s[j][1];
                rs1 += s[j][2] + s[j][3];
            }
            l0 = l0 * a0 + rs0;
            l1 = l1 * a1 + rs1;
            if (__any_sync(0xffffffffu, (a0 != 1.f) || (a1 != 1.f))) {
#pragma unroll
                for (int j = 0; j < D / 8; ++j) {
                    o[j][0] *= a0; o[j][1] *= a0;
                    o[j][2] *= a1; o[j][3] *= a1;
                }
            }
            // ---- O += P V with P = P_hi + P_lo (two bf16 products)
            const bool vmask = key0 + kPage > leff;
#pragma unroll
            for (int kk = 0; kk < C::KK; ++kk) {
                uint32_t A_hi[4], A_lo[4];
                // A fragment order: a0 (row g, k 0-7), a1 (row g+8, k 0-7),
                // a2 (row g, k 8-15), a3 (row g+8, k 8-15)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const float* sj = s[2 * kk + h];
                    const uint32_t x0 = pack_bf16(sj[0], sj[1]);
                    const uint32_t x1 = pack_bf16(sj[2], sj[3]);
                    A_hi[2 * h + 0] = x0;
                    A_hi[2 * h + 1] = x1;
                    A_lo[2 * h + 0] = pack_bf16(sj[0] - bf16lo_to_f32(x0), sj[1] - bf16hi_to_f32(x0));
                    A_lo[2 * h + 1] = pack_bf16(sj[2] - bf16lo_to_f32(x1), sj[3] - bf16hi_to_f32(x1));
                }
                const int kA = key0 + wkey + 16 * kk + 2 * tq;   // keys of b0/b2 (b1/b3: +8)
#pragma unroll
                for (int nn = 0; nn < D / 16; ++nn) {
                    const int key = wkey + 16 * kk + (((lane >> 3) & 1) << 3) + (lane & 7);
                    const int chunk = 2 * nn + (lane >> 4);
                    const uint32_t addr = vb + (chunk >> 3) * 8192 + key * 128 +
                                          (((chunk & 7) ^ (lane & 7)) << 4);
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_trans(b0, b1, b2, b3, addr);
                    if (vmask) {
                        // zero V of keys no row may see (their slots may hold anything)
                        const uint32_t mA = (kA < leff ? 0x0000ffffu : 0u) |
                                            (kA + 1 < leff ? 0xffff0000u : 0u);
                        const uint32_t mB = (kA + 8 < leff ? 0x0000ffffu : 0u) |
                                            (kA + 9 < leff ? 0xffff0000u : 0u);
                        b0 &= mA; b2 &= mA; b1 &= mB; b3 &= mB;
                    }
                    mma_bf16(o[2 * nn], A_hi, b0, b1);
                    mma_bf16(o[2 * nn], A_lo, b0, b1);
                    mma_bf16(o[2 * nn + 1], A_hi, b2, b3);
                    mma_bf16(o[2 * nn + 1], A_lo, b2, b3);
                }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar_empty + 8 * st);

        if (flags & kLast) {
            // ---- segment end: the row sums over the quad, then hand over
            float lt0 = l0 + __shfl_xor_sync(0xffffffffu, l0, 1);
            lt0 += __shfl_xor_sync(0xffffffffu, lt0, 2);
            if (!hand_over(false, lt0)) {
                if (lane == 0) atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
                return;
            }
        }
        if (++st == NST) { st = 0; ph ^= 1; }
    }
}

}  // namespace spire
