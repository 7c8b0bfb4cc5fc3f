// spire_kernels.cuh -- device code of libspire.
//
// One speculation round of SPIRe (arXiv 2504.06419) spends its attention time
// streaming KV caches: the target's full cache once for the k+1 block tokens
// (Section 2, t_verify) and the draft's bounded sink + window cache once per
// draft step (Section 3.1).  Both are the same flash-decoding shape: a few
// query rows per KV head against a long run of 64-token KV tiles.  Three
// kernels implement it:
//
//   plan_kernel    cuts every (sequence, KV head) into splits of `chunk`
//                  tiles, chosen from the ragged lengths so that the work
//                  list has ~kTargetItems items, and orders the list longest
//                  first.  Split boundaries depend only on ctx_lens.
//   split_kernel   persistent CTAs pull items from the list.  One producer
//                  warp streams K/V tiles with TMA into an NST-deep ring of
//                  shared-memory stages; consumer warps each own 16 query rows
//                  (an m-tile) and a slice of the 64 keys of every tile, run
//                  QK^T and PV on the tensor cores (bf16 mma, fp32 accumulate)
//                  and keep an fp32 online softmax.  All GQA heads and all k+1
//                  block rows of a KV head share each tile, so each KV byte is
//                  read from HBM once per call.
//   combine_kernel merges the splits of a (sequence, KV head) by log-sum-exp.
//
// Precision: scores and the softmax are fp32; P is fed to the PV product as
// the sum of two bf16 terms (hi + lo), which carries ~16 mantissa bits, so the
// bf16 rounding of P (~1.7e-3 relative rms) does not reach the output.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "spire_ptx.cuh"

namespace spire {

constexpr int kPage = 64;                // tokens per KV tile (and per page)
constexpr int kTargetItems = 1024;       // split-plan target item count
constexpr int kMinChunkVerify = 8;       // minimum tiles per split, verify
constexpr int kMinChunkDraft = 4;        // minimum tiles per split, draft
constexpr int kPlanThreads = 1024;
constexpr int kPlanSortMax = 4096;       // longest-first ordering up to this batch

constexpr uint32_t kErrCtxLen = 1u;
constexpr uint32_t kErrPageId = 2u;
constexpr uint32_t kErrTimeout = 4u;

// header words at the start of the workspace
constexpr int kHdrErr = 0, kHdrCounter = 1, kHdrItems = 2, kHdrChunk = 3;

enum Mode : int32_t { kModeVerify = 0, kModeDraft = 1 };

struct PlanParams {
    const int32_t* ctx_lens;
    int4* seq_info;     // [B]: x = visible length, y = n_split, z = split base, w = valid
    int4* items;        // work list: x = b*Hkv + g, y = first tile, z = n tiles, w = split idx
    int32_t* header;
    int32_t B, Hkv, kp1, mode, max_pages, cap;  // cap: draft slots S (draft) / unused
};

struct SplitParams {
    const __nv_bfloat16* q;   // [B, kp1, Hq, D]
    float* out;               // [B, kp1, Hq, D]
    const int32_t* block_table;
    const int4* seq_info;
    const int4* items;
    int32_t* header;
    float* part_o;            // [slots * R, D]
    float* part_lse;          // [slots * R]
    int32_t B, Hq, Hkv, G, kp1, R;
    int32_t max_pages, num_pages;
    int32_t mode;
    float sl2;                // softmax_scale * log2(e)
};

// ============================================================== split (a2)
template <int D, int MT, int KP, int NST>
struct SplitCfg {
    static constexpr int NW = MT * KP;            // consumer warps
    static constexpr int THREADS = 32 * (NW + 1); // + one producer warp
    static constexpr int KW = kPage / KP;         // keys per consumer warp per tile
    static constexpr int NT = KW / 8;             // S n-tiles per warp
    static constexpr int KK = KW / 16;            // PV k-steps per warp
    static constexpr int TILE = kPage * D * 2;    // bytes of one K (or V) tile
    static constexpr int STAGE = 2 * TILE;
    static constexpr int SCR = D + 8;             // floats per scratch row
    static constexpr int OFF_SCR_O = NST * STAGE;
    static constexpr int OFF_SCR_ML = OFF_SCR_O + NW * 16 * SCR * 4;
    static constexpr int OFF_META = OFF_SCR_ML + NW * 16 * 8;
    static constexpr int OFF_BAR = OFF_META + NST * 32;
    static constexpr int SMEM = OFF_BAR + (2 * NST + 2) * 8 + 1024;  // + alignment slack
    static_assert(KW >= 16 && NT % 2 == 0, "each warp needs >= 16 keys of a tile");
    static_assert(D % 64 == 0, "head_dim must be a multiple of 64");
};

enum : int32_t { kFirst = 1, kLast = 2, kBad = 4, kTerm = 8 };

template <int D, int MT, int KP, int NST>
__global__ void __launch_bounds__(SplitCfg<D, MT, KP, NST>::THREADS, 1)
    split_kernel(const __grid_constant__ CUtensorMap tmap_k,
                 const __grid_constant__ CUtensorMap tmap_v, const SplitParams p) {
    using C = SplitCfg<D, MT, KP, NST>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* const sbase = smem_raw + (base - raw);
    float* const scr_o = reinterpret_cast<float*>(sbase + C::OFF_SCR_O);
    float2* const scr_ml = reinterpret_cast<float2*>(sbase + C::OFF_SCR_ML);
    int4* const meta = reinterpret_cast<int4*>(sbase + C::OFF_META);
    const uint32_t bar_full = base + C::OFF_BAR;          // NST barriers
    const uint32_t bar_empty = bar_full + NST * 8;         // NST barriers
    const uint32_t bar_ep_full = bar_empty + NST * 8;
    const uint32_t bar_ep_empty = bar_ep_full + 8;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, C::NW);
        }
        mbar_init(bar_ep_full, 32 * C::NW);
        mbar_init(bar_ep_empty, 32 * C::NW);
        fence_barrier_init();
    }
    __syncthreads();

    const int n_items = p.header[kHdrItems];

    if (warp == C::NW) {
        // ------------------------------------------------------ producer
        if (lane != 0) return;
        prefetch_tensormap(&tmap_k);
        prefetch_tensormap(&tmap_v);
        const uint64_t pol = policy_evict_first();
        uint32_t st = 0, ph = 0;
        uint32_t armed = 0;            // bit s: stage s has a TMA load outstanding or done
        uint32_t armed_parity = 0;     // bit s: parity of that load's phase
        bool ok = true;
        for (;;) {
            const int it = atomicAdd(&p.header[kHdrCounter], 1);
            if (it >= n_items) break;
            const int4 item = p.items[it];
            const int b = item.x / p.Hkv, g = item.x - b * p.Hkv;
            const int4 si = p.seq_info[b];
            const int slot = (si.z + item.w) * p.Hkv + g;
            const int n = item.z > 0 ? item.z : 1;
            for (int i = 0; i < n; ++i) {
                if (!mbar_wait(bar_empty + 8 * st, ph ^ 1)) { ok = false; break; }
                const int tile = item.y + i;
                int flags = (i == 0 ? kFirst : 0) | (i == n - 1 ? kLast : 0);
                bool bad = !si.w || item.z <= 0;
                int zk = 0, zv = 0, y = 0;
                if (!bad) {
                    if (p.mode == kModeVerify) {
                        const int page = p.block_table[(long long)b * p.max_pages + tile];
                        if (page < 0 || page >= p.num_pages) {
                            bad = true;
                            atomicOr(&p.header[kHdrErr], (int)kErrPageId);
                        }
                        zk = zv = page * p.Hkv + g;
                    } else {
                        y = tile * kPage;
                        zk = (b * 2 + 0) * p.Hkv + g;
                        zv = (b * 2 + 1) * p.Hkv + g;
                    }
                }
                if (bad) flags |= kBad;
                meta[2 * st] = make_int4(b, g, tile * kPage, si.x);
                meta[2 * st + 1] = make_int4(slot, si.y, flags, 0);
                if (bad) {
                    mbar_arrive(bar_full + 8 * st);
                } else {
                    const uint32_t dk = base + st * C::STAGE, dv = dk + C::TILE;
                    mbar_arrive_expect_tx(bar_full + 8 * st, C::STAGE);
#pragma unroll
                    for (int h = 0; h < D / 64; ++h) {
                        tma_load_3d(dk + h * 8192, &tmap_k, h * 64, y, zk, bar_full + 8 * st, pol);
                        tma_load_3d(dv + h * 8192, &tmap_v, h * 64, y, zv, bar_full + 8 * st, pol);
                    }
                    armed |= 1u << st;
                    armed_parity = (armed_parity & ~(1u << st)) | (ph << st);
                }
                if (++st == NST) { st = 0; ph ^= 1; }
            }
            if (!ok) break;
        }
        if (ok && mbar_wait(bar_empty + 8 * st, ph ^ 1)) {
            meta[2 * st + 1] = make_int4(0, 0, kTerm, 0);
            mbar_arrive(bar_full + 8 * st);
        } else {
            // Consumers stopped answering: record it and wait (bounded) for
            // our own copies to land before the CTA's shared memory goes away.
            atomicOr(&p.header[kHdrErr], (int)kErrTimeout);
            for (int s = 0; s < NST; ++s)
                if (armed & (1u << s)) mbar_wait(bar_full + 8 * s, (armed_parity >> s) & 1u);
        }
        return;
    }

    // ---------------------------------------------------------- consumers
    const int mt = warp / KP, kp = warp - (warp / KP) * KP;
    const int gq = lane >> 2, tq = lane & 3;          // mma group / thread-in-group
    const int r0 = mt * 16 + gq, r1 = r0 + 8;         // the two rows this thread holds
    const int wkey = kp * C::KW;                      // first key of this warp in a tile
    const float sl2 = p.sl2;
    const float NEG_INF = __int_as_float(0xff800000);

    float o[D / 8][4];
    uint32_t qf[D / 16][4];
    float m0 = NEG_INF, m1 = NEG_INF, l0 = 0.f, l1 = 0.f;
    bool poison = false;
    int cur_b = 0, cur_g = 0, cur_slot = 0, cur_nsplit = 1, lim0 = 0, lim1 = 0, leff = 0;
    uint32_t st = 0, ph = 0, ep = 0;

    for (;;) {
        if (!mbar_wait(bar_full + 8 * st, ph)) {
            atomicOr(&p.header[kHdrErr], (int)kErrTimeout);
            return;
        }
        const int4 ma = meta[2 * st], mb = meta[2 * st + 1];
        const int flags = mb.z;
        if (flags & kTerm) return;
        if (flags & kFirst) {
            cur_b = ma.x; cur_g = ma.y; leff = ma.w; cur_slot = mb.x; cur_nsplit = mb.y;
            poison = false;
            m0 = m1 = NEG_INF; l0 = l1 = 0.f;
#pragma unroll
            for (int j = 0; j < D / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
            // rows r = i*G + hl (block row i, head hl of the group)
            const int i0 = min(r0 / p.G, p.kp1 - 1), i1 = min(r1 / p.G, p.kp1 - 1);
            lim0 = leff - (p.kp1 - 1) + i0;
            lim1 = leff - (p.kp1 - 1) + i1;
            const __nv_bfloat16* q0 = p.q + ((long long)(cur_b * p.kp1 + i0) * p.Hq +
                                             cur_g * p.G + (r0 - (r0 / p.G) * p.G)) * D;
            const __nv_bfloat16* q1 = p.q + ((long long)(cur_b * p.kp1 + i1) * p.Hq +
                                             cur_g * p.G + (r1 - (r1 / p.G) * p.G)) * D;
            const bool v0 = r0 < p.R, v1 = r1 < p.R;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
                const int c = ks * 16 + 2 * tq;
                qf[ks][0] = v0 ? *reinterpret_cast<const uint32_t*>(q0 + c) : 0u;
                qf[ks][1] = v1 ? *reinterpret_cast<const uint32_t*>(q1 + c) : 0u;
                qf[ks][2] = v0 ? *reinterpret_cast<const uint32_t*>(q0 + c + 8) : 0u;
                qf[ks][3] = v1 ? *reinterpret_cast<const uint32_t*>(q1 + c + 8) : 0u;
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
                uint32_t ah[4], al[4];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const float* sj = s[2 * kk + h];
                    const uint32_t x0 = pack_bf16(sj[0], sj[1]);
                    const uint32_t x1 = pack_bf16(sj[2], sj[3]);
                    ah[2 * h + 0] = x0;
                    ah[2 * h + 1] = x1;
                    al[2 * h + 0] = pack_bf16(sj[0] - bf16lo_to_f32(x0), sj[1] - bf16hi_to_f32(x0));
                    al[2 * h + 1] = pack_bf16(sj[2] - bf16lo_to_f32(x1), sj[3] - bf16hi_to_f32(x1));
                }
                // A fragment order: a0 (row g, k 0-7), a1 (row g+8, k 0-7),
                // a2 (row g, k 8-15), a3 (row g+8, k 8-15)
                const uint32_t A_hi[4] = {ah[0], ah[1], ah[2], ah[3]};
                const uint32_t A_lo[4] = {al[0], al[1], al[2], al[3]};
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
            // ---- epilogue: merge the KP key slices of each m-tile, write out
            float lt0 = l0 + __shfl_xor_sync(0xffffffffu, l0, 1);
            lt0 += __shfl_xor_sync(0xffffffffu, lt0, 2);
            float lt1 = l1 + __shfl_xor_sync(0xffffffffu, l1, 1);
            lt1 += __shfl_xor_sync(0xffffffffu, lt1, 2);
            if (ep > 0 && !mbar_wait(bar_ep_empty, (ep - 1) & 1)) {
                atomicOr(&p.header[kHdrErr], (int)kErrTimeout);
                return;
            }
            float* so = scr_o + warp * 16 * C::SCR;
#pragma unroll
            for (int j = 0; j < D / 8; ++j) {
                *reinterpret_cast<float2*>(so + gq * C::SCR + 8 * j + 2 * tq) =
                    make_float2(o[j][0], o[j][1]);
                *reinterpret_cast<float2*>(so + (gq + 8) * C::SCR + 8 * j + 2 * tq) =
                    make_float2(o[j][2], o[j][3]);
            }
            if (tq == 0) {
                const float NANF = __int_as_float(0x7fc00000);
                scr_ml[warp * 16 + gq] = make_float2(poison ? NANF : m0, lt0);
                scr_ml[warp * 16 + gq + 8] = make_float2(poison ? NANF : m1, lt1);
            }
            mbar_arrive(bar_ep_full);
            if (!mbar_wait(bar_ep_full, ep & 1)) {
                atomicOr(&p.header[kHdrErr], (int)kErrTimeout);
                return;
            }
            const int ctid = threadIdx.x;            // 0 .. 32*NW-1
            constexpr int D4 = D / 4;
            for (int idx = ctid; idx < MT * 16 * D4; idx += 32 * C::NW) {
                const int mtm = idx / (16 * D4);
                const int rem = idx - mtm * 16 * D4;
                const int rl = rem / D4, d4 = rem - rl * D4;
                const int r = mtm * 16 + rl;
                if (r >= p.R) continue;
                float M = NEG_INF;
                bool nan = false;
#pragma unroll
                for (int kq = 0; kq < KP; ++kq) {
                    const float mk = scr_ml[(mtm * KP + kq) * 16 + rl].x;
                    nan |= (mk != mk);
                    M = fmaxf(M, mk);
                }
                const float Mr = (M == NEG_INF) ? 0.f : M;
                float lsum = 0.f;
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int kq = 0; kq < KP; ++kq) {
                    const int w2 = mtm * KP + kq;
                    const float2 ml = scr_ml[w2 * 16 + rl];
                    const float wgt = ex2(ml.x - Mr);
                    lsum += wgt * ml.y;
                    const float4 ov =
                        *reinterpret_cast<const float4*>(scr_o + (w2 * 16 + rl) * C::SCR + 4 * d4);
                    acc.x += wgt * ov.x; acc.y += wgt * ov.y;
                    acc.z += wgt * ov.z; acc.w += wgt * ov.w;
                }
                float4 res;
                float lse;
                if (nan) {
                    const float NANF = __int_as_float(0x7fc00000);
                    res = make_float4(NANF, NANF, NANF, NANF);
                    lse = NANF;
                } else if (lsum > 0.f) {
                    const float inv = 1.f / lsum;
                    res = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
                    lse = M + __log2f(lsum);
                } else {  // no key of this split is visible to this row
                    res = make_float4(0.f, 0.f, 0.f, 0.f);
                    lse = NEG_INF;
                }
                if (cur_nsplit == 1) {
                    const int i = r / p.G, hl = r - i * p.G;
                    float* dst = p.out + ((long long)(cur_b * p.kp1 + i) * p.Hq + cur_g * p.G + hl) * D;
                    *reinterpret_cast<float4*>(dst + 4 * d4) = res;
                } else {
                    const long long row = (long long)cur_slot * p.R + r;
                    *reinterpret_cast<float4*>(p.part_o + row * D + 4 * d4) = res;
                    if (d4 == 0) p.part_lse[row] = lse;
                }
            }
            mbar_arrive(bar_ep_empty);
            ++ep;
        }
        if (++st == NST) { st = 0; ph ^= 1; }
    }
}

// ============================================================== combine (a3) params
struct CombineParams {
    const int4* seq_info;
    const float* part_o;
    const float* part_lse;
    float* out;
    int32_t B, Hq, Hkv, G, kp1, R, D;
};

}  // namespace spire
