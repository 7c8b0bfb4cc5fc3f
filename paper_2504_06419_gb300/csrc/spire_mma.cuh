// spire_mma.cuh -- attention kernel on the warp-level tensor-core path
// (mma.sync m16n8k16, bf16 in / fp32 accumulate).
//
// Roles in a CTA (one CTA per SM):
//   warp NCW (producer) lane 0 walks the CTA's tile range, translates pages
//                       through the block table, and streams each K and V
//                       tile with TMA (64 keys x D, 128-byte swizzle) into
//                       an NST-deep ring of shared-memory stages.
//   warps 0..NCW-1      NG = 2 groups of NW = 4 consumer warps; the groups
//                       take turns by segment of the walk, so each SM
//                       sub-partition runs two independent consumer chains.
//                       Consumer warp w of a group owns key slice w (16 keys
//                       of every tile).  It keeps Q^T in registers for the
//                       current pair, runs S^T = K Q^T and O^T += V^T P^T on
//                       the tensor cores (keys and head dimensions as the
//                       MMA's 16 rows, the pair's query rows as its 8
//                       columns) and an fp32 online softmax in base 2.
//   warp NCW+1 (epilogue) at the end of a pair's segment the owning group only
//                       hands its (O, m, l) rows to one of two shared-memory
//                       buffers and goes on; this warp merges the NW key
//                       slices and writes the result to the output, or to a
//                       partial slot that the last-arriving CTA merges (see
//                       spire_common.cuh), publishing with a fence and an
//                       atomic, off the consumers' path.
// The kernel serves pairs of at most 8 query rows (the MMA's N = 8), so a
// buffer holds 8 rows per consumer warp.
//
// Precision: P enters the PV product as P_hi + P_lo, two bf16 terms carrying
// ~16 mantissa bits, so rounding P to bf16 (~1.7e-3 rms relative) never
// reaches the output.
#pragma once

#include "spire_common.cuh"

namespace spire {

template <int D, int MT, int KP, int NST>
struct MmaCfg {
    static constexpr int NW = MT * KP;            // consumer warps of a group (one per key slice)
    static constexpr int NG = 2;                  // consumer groups: they take turns by segment
    static constexpr int NCW = NW * NG;           // consumer warps
    static constexpr int THREADS = 32 * (NCW + 2);  // + a producer and an epilogue warp
    static constexpr int KW = kPage / KP;         // keys per consumer warp per tile
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
    static_assert(KW == 16, "each consumer warp owns one 16-key MMA slice of a tile");
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
            mbar_init(bar_empty + 8 * s, C::NCW);
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

    if (warp == C::NCW) {
        // ------------------------------------------------------ producer
        if (lane != 0) return;
        const ProducerSmem psm{base, qsm, (uint32_t)C::QHALF, meta, bar_full,
                               bar_empty, bar_qfull, bar_qempty, 1, 0, 2, true};
        const uint32_t err = produce<D, NST, kStall>(p, *sh, &tmap_k, &tmap_v, &tmap_q, psm);
        if (err) atomicOr(&p.err[blockIdx.x], (int)err);
        return;
    }
    if (warp == C::NCW + 1) {
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
    // NG groups of NW warps take turns by segment (group n % NG computes the
    // n-th segment of the CTA's walk), so each SM sub-partition runs NG
    // independent consumer warps; every consumer warp still waits for every
    // stage and reads its tile record, and the other groups' warps release a
    // stage as soon as they have read it.  Segment n is handed to the epilogue
    // warp through buffer n % 2; the epilogue takes them in segment order.
    // Warp w of a group owns keys [w KW, (w + 1) KW) of every tile (KW = 16).  The keys
    // are the MMA rows (M = 16) and the pair's R <= 8 query rows its columns
    // (N = 8), so at most 8 - R columns and no row of an MMA are padding:
    //   S^T  = K Q^T          A = the warp's K slice, B = Q^T (registers)
    //   O^T += V^T (P^T)      A = the V slice read transposed, B = P^T moved
    //                         into the B layout with movmatrix.trans
    // Lane (gq, tq) = (lane / 4, lane % 4) holds S^T of slice keys gq and
    // gq + 8 for query rows ra = 2 tq and rb = 2 tq + 1, and O^T of
    // dimensions 16 j + gq and 16 j + gq + 8 (j < D / 16) of the same rows.
    const int gq = lane >> 2, tq = lane & 3;
    const int ra = 2 * tq, rb = ra + 1;
    const int grp = warp / C::NW, slice = warp - grp * C::NW;
    const int wkey = slice * C::KW;                   // first key of this warp in a tile
    const float sl2 = p.sl2;
    const float NEG_INF = __int_as_float(0xff800000);
    const float NANF = __int_as_float(0x7fc00000);
    constexpr uint32_t FULL = 0xffffffffu;

    float o[D / 16][4];
    uint32_t qf[D / 16][2];
    float ma = NEG_INF, mb = NEG_INF, la = 0.f, lb = 0.f;
    bool poison = false, own = false;                 // own: this group computes the segment
    int cur_b = 0, cur_g = 0, cur_slot = 0, cur_nseg = 1, cur_first = 0;
    int lima = 0, limb = 0, leff = 0;
    uint32_t st = 0, ph = 0, n_seg = 0;               // stage ring / segments ended so far
    uint32_t cq[2] = {0u, 0u};                        // parity of each Q buffer

    // hand the segment's (O, m, l) rows, or the end of the work, to the epilogue
    // warp through buffer n_seg & 1 (rows < R only; the others are padding)
    auto hand_over = [&](bool term, float lta, float ltb) -> bool {
        const int sb = n_seg & 1;
        if (!mbar_wait(bar_sempty + 8 * sb, ((n_seg >> 1) & 1) ^ 1)) return false;
        if (!term) {
            float* so = scr_o + sb * C::SCR_BUF + slice * C::SR * C::SCR;
            if (ra < p.R) {
#pragma unroll
                for (int j = 0; j < D / 16; ++j) {
                    so[ra * C::SCR + 16 * j + gq] = o[j][0];
                    so[ra * C::SCR + 16 * j + gq + 8] = o[j][2];
                }
            }
            if (rb < p.R) {
#pragma unroll
                for (int j = 0; j < D / 16; ++j) {
                    so[rb * C::SCR + 16 * j + gq] = o[j][1];
                    so[rb * C::SCR + 16 * j + gq + 8] = o[j][3];
                }
            }
            if (gq == 0) {
                float2* ml = scr_ml + sb * C::NW * C::SR + slice * C::SR;
                ml[ra] = make_float2(poison ? NANF : ma, lta);
                ml[rb] = make_float2(poison ? NANF : mb, ltb);
            }
        }
        if (slice == 0 && lane == 0) {
            scr_info[2 * sb] = make_int4(cur_b, cur_g, cur_slot, cur_nseg);
            scr_info[2 * sb + 1] = make_int4(cur_first, term ? 1 : 0, 0, 0);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar_sfull + 8 * sb);
        return true;
    };

    for (;;) {
        if (!mbar_wait(bar_full + 8 * st, ph)) {
            if (lane == 0) atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
            return;
        }
        const int4 mta = meta[2 * st], mtb = meta[2 * st + 1];
        const int flags = mtb.x & 0xff;
        if (flags & kTerm) {
            // the group that would take the next segment tells the epilogue
            if ((int)(n_seg % C::NG) == grp && !hand_over(true, 0.f, 0.f) && lane == 0)
                atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
            return;
        }
        if (flags & kFirst) {
            own = (int)(n_seg % C::NG) == grp;
            const int flags_q = mtb.x;
            cur_b = mta.x; cur_g = mta.y; leff = mta.w;
            cur_slot = mtb.y; cur_nseg = mtb.z; cur_first = mtb.w;
            poison = false;
            ma = mb = NEG_INF; la = lb = 0.f;
#pragma unroll
            for (int j = 0; j < D / 16; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
            // rows r = i*G + hl (block row i, head hl of the group)
            const int ia = min(ra / p.G, p.kp1 - 1), ib = min(rb / p.G, p.kp1 - 1);
            lima = leff - (p.kp1 - 1) + ia;
            limb = leff - (p.kp1 - 1) + ib;
            const int qflag = flags_q >> 8;
            if ((qflag & 16) && !own) {
                cq[qflag & 1] ^= 1;     // the other group reads this Q buffer phase
            } else if (qflag & 16) {
                const int qb = qflag & 1;
                if (!mbar_wait(bar_qfull + 8 * qb, cq[qb])) {
                    if (lane == 0) atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
                    return;
                }
                cq[qb] ^= 1;
                // B = Q^T: lane (gq, tq) takes row gq, columns 2 tq, 2 tq + 1 of
                // the 8x8 blocks at 16-byte chunks 2 ks and 2 ks + 1
                const uint32_t qbase = qsm + qb * C::QBUF;
                const int qrow = lane & 7;
#pragma unroll
                for (int ks = 0; ks < D / 16; ks += 2) {
                    const int chunk = 2 * ks + (lane >> 3);
                    ldsm_x4(qf[ks][0], qf[ks][1], qf[ks + 1][0], qf[ks + 1][1],
                            qbase + (chunk >> 3) * C::QHALF + qrow * 128 +
                                (((chunk & 7) ^ qrow) << 4));
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_qempty + 8 * qb);
            }
        }
        if (!own) {
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_empty + 8 * st);
        } else if (flags & kBad) {
            poison = true;
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_empty + 8 * st);
        } else {
            const int key0 = mta.z;                          // sequence index of tile key 0
            const uint32_t kb = base + st * C::STAGE, vb = kb + C::TILE;
            // ---- this warp's K and V fragments into registers, then the stage is
            // released: it is refilled while the tile is computed, which keeps
            // more bytes in flight than holding it through the math
            uint32_t kf[D / 16][4], vf[D / 16][4];
            const int krow = wkey + ((lane >> 3) & 1) * 8 + (lane & 7);
            const int vrow = wkey + ((lane >> 4) << 3) + (lane & 7);
#pragma unroll
            for (int j = 0; j < D / 16; ++j) {
                const int kc = 2 * j + (lane >> 4), vc = 2 * j + ((lane >> 3) & 1);
                ldsm_x4(kf[j][0], kf[j][1], kf[j][2], kf[j][3],
                        kb + (kc >> 3) * 8192 + krow * 128 + (((kc & 7) ^ (lane & 7)) << 4));
                ldsm_x4_trans(vf[j][0], vf[j][1], vf[j][2], vf[j][3],
                              vb + (vc >> 3) * 8192 + vrow * 128 + (((vc & 7) ^ (lane & 7)) << 4));
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_empty + 8 * st);
            // ---- S^T = K Q^T over this warp's 16 keys: two accumulation chains
            float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
                if (ks & 1) mma_bf16(s1, kf[ks], qf[ks][0], qf[ks][1]);
                else        mma_bf16(s0, kf[ks], qf[ks][0], qf[ks][1]);
            }
            float s[4] = {s0[0] + s1[0], s0[1] + s1[1], s0[2] + s1[2], s0[3] + s1[3]};
            // ---- causal / length mask (only tiles reaching past row 0's limit)
            if (key0 + kPage > leff - (p.kp1 - 1)) {
                const int kx = key0 + wkey + gq;
                if (kx >= lima) s[0] = NEG_INF;
                if (kx >= limb) s[1] = NEG_INF;
                if (kx + 8 >= lima) s[2] = NEG_INF;
                if (kx + 8 >= limb) s[3] = NEG_INF;
            }
            // ---- online softmax (base 2); a row's 16 keys sit in the 8 lanes of its tq
            float xa = fmaxf(s[0], s[2]), xb = fmaxf(s[1], s[3]);
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                xa = fmaxf(xa, __shfl_xor_sync(FULL, xa, off));
                xb = fmaxf(xb, __shfl_xor_sync(FULL, xb, off));
            }
            const float mna = fmaxf(ma, xa * sl2), mnb = fmaxf(mb, xb * sl2);
            const float mra = (mna == NEG_INF) ? 0.f : mna;
            const float mrb = (mnb == NEG_INF) ? 0.f : mnb;
            const float aa = ex2(ma - mra), ab = ex2(mb - mrb);
            ma = mna; mb = mnb;
            s[0] = ex2(fmaf(s[0], sl2, -mra));
            s[1] = ex2(fmaf(s[1], sl2, -mrb));
            s[2] = ex2(fmaf(s[2], sl2, -mra));
            s[3] = ex2(fmaf(s[3], sl2, -mrb));
            la = la * aa + (s[0] + s[2]);
            lb = lb * ab + (s[1] + s[3]);
            if (__any_sync(FULL, (aa != 1.f) || (ab != 1.f))) {
#pragma unroll
                for (int j = 0; j < D / 16; ++j) {
                    o[j][0] *= aa; o[j][1] *= ab;
                    o[j][2] *= aa; o[j][3] *= ab;
                }
            }
            // ---- P^T = P_hi + P_lo (two bf16 terms) in the B layout
            const uint32_t h0 = pack_bf16(s[0], s[1]);      // key gq: rows ra, rb
            const uint32_t h1 = pack_bf16(s[2], s[3]);      // key gq + 8
            const uint32_t l0 = pack_bf16(s[0] - bf16lo_to_f32(h0), s[1] - bf16hi_to_f32(h0));
            const uint32_t l1 = pack_bf16(s[2] - bf16lo_to_f32(h1), s[3] - bf16hi_to_f32(h1));
            const uint32_t bh0 = movm_trans(h0), bh1 = movm_trans(h1);
            const uint32_t bl0 = movm_trans(l0), bl1 = movm_trans(l1);
            // ---- O^T += V^T P^T; V of keys no row may see is zeroed (their
            // slots may hold anything)
            if (key0 + kPage > leff) {
                const int kA = key0 + wkey + 2 * tq;        // keys of a0 / a1 (a2 / a3: + 8)
                const uint32_t mkA = (kA < leff ? 0x0000ffffu : 0u) | (kA + 1 < leff ? 0xffff0000u : 0u);
                const uint32_t mkB = (kA + 8 < leff ? 0x0000ffffu : 0u) | (kA + 9 < leff ? 0xffff0000u : 0u);
#pragma unroll
                for (int j = 0; j < D / 16; ++j) {
                    vf[j][0] &= mkA; vf[j][1] &= mkA; vf[j][2] &= mkB; vf[j][3] &= mkB;
                }
            }
#pragma unroll
            for (int j = 0; j < D / 16; ++j) {
                mma_bf16(o[j], vf[j], bh0, bh1);
                mma_bf16(o[j], vf[j], bl0, bl1);
            }
        }

        if (flags & kLast) {
            if (own) {
                // ---- segment end: each row's sum over its 8 lanes, then hand over
                float lta = la, ltb = lb;
#pragma unroll
                for (int off = 4; off < 32; off <<= 1) {
                    lta += __shfl_xor_sync(FULL, lta, off);
                    ltb += __shfl_xor_sync(FULL, ltb, off);
                }
                if (!hand_over(false, lta, ltb)) {
                    if (lane == 0) atomicOr(&p.err[blockIdx.x], (int)kErrTimeout);
                    return;
                }
            }
            ++n_seg;
        }
        if (++st == NST) { st = 0; ph ^= 1; }
    }
}

}  // namespace spire
