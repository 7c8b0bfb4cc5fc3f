// spire_tokens.cu -- token verification of a speculation round (include/
// spire.h: spire_verify_tokens): the modified rejection sampling that makes
// every emitted token a sample of the target model's distribution (Section 1;
// the token verification algorithm, Section 6).
//
// Per sequence b with drafts x_1..x_k, draft distributions q_1..q_k and target
// distributions p_1..p_{k+1}:
//   j = the number of leading drafts with u_i * q_i(x_i) < p_i(x_i) (binary32)
//   the round's one draw: from w = max(0, p_{j+1} - q_{j+1}) when j < k (from
//   p_{j+1} if that residual has no positive entry), from p_{k+1} when j = k,
//   as the exponential race argmax_v w_v / E_v (E_v ~ Exp(1) given), ties to
//   the smallest v.
//
// Vocabularies that are a multiple of 4 (rows 16-byte aligned) take three
// launches:
//   tokens_accept_kernel    one warp per sequence: j from the k gathered
//                           probabilities (a ballot), and the bad-token flag;
//                           clears the device error word.
//   tokens_stream_kernel    its programmatic dependent, four CTAs per SM
//                           walking (sequence, chunk of 4096 entries) units:
//                           a producer warp copies the chunk's rows p_{j+1},
//                           q_{j+1} (only if j < k) and E into a four-stage
//                           shared-memory ring (1024 entries per stage) with
//                           bulk async copies, and eight consumer warps
//                           reduce the best (score, index) key of the
//                           residual and of p alone, dividing exactly only
//                           where an estimate reaches the warp's best so far;
//                           one partial per unit.
//   tokens_finalize_kernel  one warp per sequence: the best key over the
//                           chunks (the maximum is unique, so the order of the
//                           reduction cannot matter), the emitted tokens and j.
// Other vocabularies use tokens_race_kernel (grid (chunks of 8192, B): each
// CTA finds j itself, then streams its chunk with 4-byte loads) and the same
// finalize.
// Only the rows a round actually needs are read: about 12 V bytes per sequence
// against the (2k + 1) * 4 V bytes of all its distributions.
#include <atomic>
#include <cmath>
#include <cstdint>

#include <cuda_runtime.h>

#include "spire.h"
#include "spire_common.cuh"
#include "spire_host.h"

namespace spire {
namespace {

constexpr int kTokThreads = 256;
constexpr int kTokChunk = 8192;          // vocabulary entries per CTA (race kernel)
constexpr int kTokUnit = 4096;           // vocabulary entries per unit (stream kernel)
constexpr int kTokSub = 1024;            // entries per stage and row (4 KB), a multiple of 1024
constexpr int kTokStages = 4;
constexpr int kTokStreamCtas = 4;        // CTAs per SM (the register limit at 288 threads)
constexpr int kTokConsumers = 8;         // consumer warps of the stream kernel
constexpr int kTokStreamThreads = 32 * (kTokConsumers + 1);
constexpr int kTokMaxK = 31;
constexpr uint32_t kTokErrToken = 1u;    // SPIRE_DEVERR_CTX_LEN: a draft token outside [0, V)
constexpr uint32_t kTokErrValue = 8u;    // SPIRE_DEVERR_VALUE: an E value not > 0, or no draw

struct TokPartial {
    unsigned long long key_res;   // best residual candidate of the chunk (0: none)
    unsigned long long key_p;     // best candidate of p alone
    int32_t j;                    // accepted drafts (every CTA of b finds the same)
    int32_t flags;
};

struct TokAccept {
    int32_t j;                    // accepted drafts of the sequence
    int32_t flags;                // kTokErrToken when the walk reached a bad token
};

struct TokParams {
    const float* p;       // [B, k+1, V]
    const float* q;       // [B, k, V]
    const int32_t* x;     // [B, k]
    const float* u;       // [B, k]
    const float* e;       // [B, V]
    TokPartial* part;     // [B, S]
    TokAccept* acc;       // [B] (stream path) or null (race path)
    int32_t* header;
    int32_t* err;
    int32_t* out;         // [B, k+1]
    int32_t* n_acc;       // [B]
    int B, k, V, S;
};

// larger key = better: the score's bits (scores are >= 0, so their bit
// patterns order like their values), then the smaller index
__device__ __forceinline__ unsigned long long race_key(float w, float e, int v) {
    const float s = __fdiv_rn(w, e);
    return ((unsigned long long)__float_as_uint(s) << 32) | (unsigned long long)(~(uint32_t)v);
}

__device__ __forceinline__ unsigned long long umax64(unsigned long long a, unsigned long long b) {
    return a > b ? a : b;
}

// Approximate reciprocal (the hardware's, relative error below 2^-22 for
// normal inputs; a subnormal input gives infinity, which the filter passes).
__device__ __forceinline__ float rcp_approx(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// An estimate w * rcp(E) is within a factor (1 +- 2^-21) of the exact w / E
// (reciprocal 2^-22, product 2^-24): below best * (1 - 2^-20) it cannot reach
// the best score.
constexpr float kTokFilter = 1.0f - 0x1p-20f;

__global__ void __launch_bounds__(kTokThreads) tokens_race_kernel(const TokParams p) {
    const int s = blockIdx.x, b = blockIdx.y;
    const int k = p.k, V = p.V;
    __shared__ int s_j;
    __shared__ int s_flags;
    __shared__ unsigned long long s_kr[kTokThreads / 32], s_kp[kTokThreads / 32];
    const int c0 = s * kTokChunk, c1 = min(V, c0 + kTokChunk);
    const float* erow = p.e + (long long)b * V;
    if (threadIdx.x >= 32) {
        // the E row does not depend on the acceptance: bring it towards L2 meanwhile
        for (int v = c0 + 32 * (threadIdx.x - 32); v < c1; v += 32 * (kTokThreads - 32))
            asm volatile("prefetch.global.L2 [%0];" ::"l"(erow + v));
    }
    if (threadIdx.x < 32) {
        // acceptance of the k drafts: lane i tests draft i + 1
        bool acc = true;
        bool bad = false;
        if ((int)threadIdx.x < k) {
            const int t = p.x[(long long)b * k + threadIdx.x];
            if (t < 0 || t >= V) {
                acc = false;
                bad = true;
            } else {
                const float pv = p.p[((long long)b * (k + 1) + threadIdx.x) * V + t];
                const float qv = p.q[((long long)b * k + threadIdx.x) * V + t];
                const float uq = __fmul_rn(p.u[(long long)b * k + threadIdx.x], qv);
                acc = uq < pv;
            }
        }
        const uint32_t rej = __ballot_sync(0xffffffffu, !acc);
        const int j = rej ? __ffs(rej) - 1 : k;
        // a bad token counts only if the walk reaches it
        const uint32_t badm = __ballot_sync(0xffffffffu, bad);
        if (threadIdx.x == 0) {
            s_j = j;
            s_flags = (j < k && ((badm >> j) & 1u)) ? (int)kTokErrToken : 0;
        }
        if (s == 0 && b == 0 && threadIdx.x == 0) {
            p.header[0] = 1;
            p.err[0] = 0;
        }
    }
    __syncthreads();
    const int j = s_j;
    const bool res = j < k;
    const float* prow = p.p + ((long long)b * (k + 1) + j) * V;
    const float* qrow = res ? p.q + ((long long)b * k + j) * V : prow;
    unsigned long long kr = 0, kp = 0;
    bool bad_e = false;
    auto visit = [&](float pv, float qv, float ev, int v) {
        if (!(ev > 0.f)) {
            bad_e = true;
            return;
        }
        if (pv > 0.f) kp = umax64(kp, race_key(pv, ev, v));
        if (res) {
            const float w = __fsub_rn(pv, qv);
            if (w > 0.f) kr = umax64(kr, race_key(w, ev, v));
        }
    };
    // 16-byte loads where the rows allow it (V % 4 == 0 keeps every row aligned)
    if ((V & 3) == 0) {
#pragma unroll 2
        for (int v = c0 + 4 * threadIdx.x; v < c1; v += 4 * kTokThreads) {
            const float4 pv = __ldg(reinterpret_cast<const float4*>(prow + v));
            const float4 ev = __ldg(reinterpret_cast<const float4*>(erow + v));
            float4 qv = pv;
            if (res) qv = __ldg(reinterpret_cast<const float4*>(qrow + v));
            visit(pv.x, qv.x, ev.x, v);
            visit(pv.y, qv.y, ev.y, v + 1);
            visit(pv.z, qv.z, ev.z, v + 2);
            visit(pv.w, qv.w, ev.w, v + 3);
        }
    } else {
        for (int v = c0 + threadIdx.x; v < c1; v += kTokThreads)
            visit(__ldg(prow + v), res ? __ldg(qrow + v) : 0.f, __ldg(erow + v), v);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        kr = umax64(kr, __shfl_xor_sync(0xffffffffu, kr, o));
        kp = umax64(kp, __shfl_xor_sync(0xffffffffu, kp, o));
    }
    const bool any_bad = __syncthreads_or(bad_e);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        s_kr[warp] = kr;
        s_kp[warp] = kp;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < kTokThreads / 32; ++w) {
            kr = umax64(kr, s_kr[w]);
            kp = umax64(kp, s_kp[w]);
        }
        TokPartial t;
        t.key_res = kr;
        t.key_p = kp;
        t.j = j;
        t.flags = s_flags | (any_bad ? (int)kTokErrValue : 0);
        p.part[(long long)b * p.S + s] = t;
    }
}

// the acceptance walk of sequence b by one warp: lane i tests draft i + 1
__device__ __forceinline__ TokAccept tok_accept(const TokParams& p, int b, int lane) {
    const int k = p.k, V = p.V;
    bool acc = true, bad = false;
    if (lane < k) {
        const int t = p.x[(long long)b * k + lane];
        if (t < 0 || t >= V) {
            acc = false;
            bad = true;
        } else {
            const float pv = p.p[((long long)b * (k + 1) + lane) * V + t];
            const float qv = p.q[((long long)b * k + lane) * V + t];
            const float uq = __fmul_rn(p.u[(long long)b * k + lane], qv);
            acc = uq < pv;
        }
    }
    const uint32_t rej = __ballot_sync(0xffffffffu, !acc);
    const int j = rej ? __ffs(rej) - 1 : k;
    // a bad token counts only if the walk reaches it
    const uint32_t badm = __ballot_sync(0xffffffffu, bad);
    TokAccept a;
    a.j = j;
    a.flags = (j < k && ((badm >> j) & 1u)) ? (int)kTokErrToken : 0;
    return a;
}

__global__ void __launch_bounds__(128) tokens_accept_kernel(const TokParams p) {
    grid_dep_launch_dependents();                // the stream kernel may start its prologue
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        p.header[0] = 1;
        p.err[0] = 0;
    }
    const int b = blockIdx.x * 4 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (b >= p.B) return;
    const TokAccept a = tok_accept(p, b, lane);
    if (lane == 0) p.acc[b] = a;
}

__global__ void __launch_bounds__(kTokStreamThreads, kTokStreamCtas) tokens_stream_kernel(const TokParams p) {
    extern __shared__ __align__(128) uint8_t tsm[];   // [stage][p | q | E rows of kTokSub]
    __shared__ __align__(8) uint64_t bars[2 * kTokStages];
    __shared__ unsigned long long s_kr[kTokConsumers], s_kp[kTokConsumers];
    __shared__ int s_flags[kTokConsumers];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t sbase = smem_u32(tsm), bar_full = smem_u32(bars),
                   bar_empty = bar_full + 8 * kTokStages;
    constexpr uint32_t ROW = kTokSub * 4, STAGE = 3 * ROW;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kTokStages; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, kTokConsumers);
        }
        fence_barrier_init();
    }
    __syncthreads();
    const int k = p.k, V = p.V, S = p.S;
    const long long units = (long long)p.B * S;
    // j of every sequence comes from the accept kernel
    grid_dep_wait();

    if (warp == 0) {
        // ------------------------------------------------ producer: bulk copies
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0, armed = 0, armed_par = 0;
            bool ok = true;
            for (long long u = blockIdx.x; ok && u < units; u += gridDim.x) {
                const int b = (int)(u / S), c = (int)(u % S);
                const int j = p.acc[b].j;
                const bool res = j < k;
                const float* prow = p.p + ((long long)b * (k + 1) + j) * V;
                const float* qrow = p.q + ((long long)b * k + (res ? j : 0)) * V;
                const float* erow = p.e + (long long)b * V;
                const int c1 = min(V, (c + 1) * kTokUnit);
                for (int v0 = c * kTokUnit; v0 < c1; v0 += kTokSub) {
                    const uint32_t n = (uint32_t)min(kTokSub, c1 - v0) * 4u;
                    if (!mbar_wait(bar_empty + 8 * s, ph ^ 1)) { ok = false; break; }
                    const uint32_t dst = sbase + s * STAGE, bar = bar_full + 8 * s;
                    mbar_arrive_expect_tx(bar, n * (res ? 3u : 2u));
                    bulk_copy_g2s(dst, prow + v0, n, bar);
                    if (res) bulk_copy_g2s(dst + ROW, qrow + v0, n, bar);
                    bulk_copy_g2s(dst + 2 * ROW, erow + v0, n, bar);
                    armed |= 1u << s;
                    armed_par = (armed_par & ~(1u << s)) | (ph << s);
                    if (++s == kTokStages) { s = 0; ph ^= 1; }
                }
            }
            if (!ok)   // our copies land before shared memory goes away
                for (int q = 0; q < kTokStages; ++q)
                    if (armed & (1u << q)) mbar_wait(bar_full + 8 * q, (armed_par >> q) & 1u);
        }
        return;
    }

    // ---------------------------------------------------- consumers
    const int cw = warp - 1, ct = threadIdx.x - 32;  // consumer warp, thread 0..255
    int s = 0;
    uint32_t ph = 0;
    bool waits_ok = true;
    for (long long u = blockIdx.x; u < units; u += gridDim.x) {
        const int b = (int)(u / S), c = (int)(u % S);
        const int j = p.acc[b].j;
        const bool res = j < k;
        const int c1 = min(V, (c + 1) * kTokUnit);
        unsigned long long kr = 0, kp = 0;
        float thr_p = 0.f, thr_r = 0.f;             // filters on the estimates
        int flags = 0;
        for (int v0 = c * kTokUnit; v0 < c1; v0 += kTokSub) {
            const int n = min(kTokSub, c1 - v0);
            // after a wait that gave up the later ones are skipped (the data
            // is then garbage and flagged), but every barrier is still met
            if (waits_ok && !mbar_wait(bar_full + 8 * s, ph)) waits_ok = false;
            if (!waits_ok) flags |= (int)kErrTimeout;
            const float* sp = reinterpret_cast<const float*>(tsm + s * STAGE);
            const float* sq = reinterpret_cast<const float*>(tsm + s * STAGE + ROW);
            const float* se = reinterpret_cast<const float*>(tsm + s * STAGE + 2 * ROW);
#pragma unroll
            for (int h = 0; h < kTokSub / 1024; ++h) {   // 4 entries per consumer thread and pass
                const int i = 4 * ct + h * 1024;
                if (i >= n) continue;
                const float4 pv = *reinterpret_cast<const float4*>(sp + i);
                const float4 ev = *reinterpret_cast<const float4*>(se + i);
                const float4 qv = res ? *reinterpret_cast<const float4*>(sq + i) : pv;
                const float pa[4] = {pv.x, pv.y, pv.z, pv.w}, qa[4] = {qv.x, qv.y, qv.z, qv.w},
                            ea[4] = {ev.x, ev.y, ev.z, ev.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int v = v0 + i + e;
                    if (!(ea[e] > 0.f)) {
                        flags |= (int)kTokErrValue;
                        continue;
                    }
                    // w * rcp(E) is within 2^-21 of w / E, so an entry whose
                    // estimate is below thr cannot reach (or tie) the best
                    // score: only the rest pay the exact division
                    const float rcp = rcp_approx(ea[e]);
                    if (pa[e] > 0.f && pa[e] * rcp >= thr_p) {
                        kp = umax64(kp, race_key(pa[e], ea[e], v));
                        thr_p = fmaxf(thr_p, __uint_as_float((uint32_t)(kp >> 32)) * kTokFilter);
                    }
                    if (res) {
                        const float w = __fsub_rn(pa[e], qa[e]);
                        if (w > 0.f && w * rcp >= thr_r) {
                            kr = umax64(kr, race_key(w, ea[e], v));
                            thr_r = fmaxf(thr_r, __uint_as_float((uint32_t)(kr >> 32)) * kTokFilter);
                        }
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_empty + 8 * s);
            if (++s == kTokStages) { s = 0; ph ^= 1; }
            // the warp's best score so far sets every lane's filter: an entry
            // below it cannot be the maximum, and lanes that agree do not
            // diverge.  Scores are >= 0, so their bit patterns (a key's high
            // word) order like the values: one integer max over the warp.
            const uint32_t wp = __reduce_max_sync(0xffffffffu, (uint32_t)(kp >> 32));
            const uint32_t wr = __reduce_max_sync(0xffffffffu, (uint32_t)(kr >> 32));
            thr_p = __uint_as_float(wp) * kTokFilter;
            thr_r = __uint_as_float(wr) * kTokFilter;
        }
        // the unit's best keys over the consumer threads
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            kr = umax64(kr, __shfl_xor_sync(0xffffffffu, kr, o));
            kp = umax64(kp, __shfl_xor_sync(0xffffffffu, kp, o));
            flags |= __shfl_xor_sync(0xffffffffu, flags, o);
        }
        if (lane == 0) {
            s_kr[cw] = kr;
            s_kp[cw] = kp;
            s_flags[cw] = flags;
        }
        named_bar_sync(1, 32 * kTokConsumers);
        if (ct == 0) {
            for (int w = 1; w < kTokConsumers; ++w) {
                kr = umax64(kr, s_kr[w]);
                kp = umax64(kp, s_kp[w]);
                flags |= s_flags[w];
            }
            TokPartial t;
            t.key_res = kr;
            t.key_p = kp;
            t.j = j;
            t.flags = flags;
            p.part[(long long)b * S + c] = t;
        }
        named_bar_sync(1, 32 * kTokConsumers);   // s_kr is reused by the next unit
    }
}

__global__ void __launch_bounds__(128) tokens_finalize_kernel(const TokParams p) {
    // one warp per sequence: lanes take the chunks' partials, shuffles find the best
    grid_dep_wait();                             // the partials of the kernel before
    const int b = blockIdx.x * 4 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (b >= p.B) return;
    const int k = p.k;
    unsigned long long kr = 0, kp = 0;
    int flags = 0, j = k;
    for (int s = lane; s < p.S; s += 32) {
        const TokPartial t = p.part[(long long)b * p.S + s];
        kr = umax64(kr, t.key_res);
        kp = umax64(kp, t.key_p);
        flags |= t.flags;
        j = t.j;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        kr = umax64(kr, __shfl_xor_sync(0xffffffffu, kr, o));
        kp = umax64(kp, __shfl_xor_sync(0xffffffffu, kp, o));
        flags |= __shfl_xor_sync(0xffffffffu, flags, o);
    }
    j = __shfl_sync(0xffffffffu, j, 0);          // every chunk found the same j; lane 0 has one
    if (p.acc) {
        j = p.acc[b].j;
        flags |= p.acc[b].flags;
    }
    const unsigned long long key = (j < k && kr) ? kr : kp;
    const int y = key ? (int)(~(uint32_t)(key & 0xffffffffull)) : -1;
    if (!key) flags |= (int)kTokErrValue;
    int32_t* o = p.out + (long long)b * (k + 1);
    for (int i = lane; i <= k; i += 32)
        o[i] = i < j ? p.x[(long long)b * k + i] : (i == j ? y : -1);
    if (lane == 0) {
        p.n_acc[b] = j;
        if (flags) atomicOr(p.err, flags);
    }
}

bool tok_shape_ok(int32_t B, int32_t k, int32_t V) {
    return B >= 0 && B <= 65535 && k >= 0 && k <= kTokMaxK && V >= 1 && V <= (1 << 30) &&
           (long long)B * (k + 1) * V < (1LL << 40);
}

// workspace: header word | error word | accept records [B] | partials [B, S]
// (S of the finer stream path: shapes alone decide the size)
size_t tok_acc_bytes(int32_t B) { return ((size_t)B * sizeof(TokAccept) + 255) & ~size_t(255); }

size_t tok_ws_bytes(int32_t B, int32_t V) {
    const long long S = (V + kTokUnit - 1) / kTokUnit;
    return 512 + tok_acc_bytes(B) + (size_t)B * S * sizeof(TokPartial);
}

}  // namespace
}  // namespace spire

using namespace spire;

extern "C" {

size_t spire_verify_tokens_workspace_bytes(int32_t batch, int32_t k, int32_t vocab) {
    if (!tok_shape_ok(batch, k, vocab)) return 0;
    return tok_ws_bytes(batch, vocab);
}

spire_status spire_verify_tokens(const float* p, const float* q, const int32_t* draft_tokens,
                                 const float* u, const float* e, int32_t batch, int32_t k,
                                 int32_t vocab, int32_t* out_tokens, int32_t* n_accepted,
                                 void* workspace, size_t ws_bytes, void* stream) {
    if (!tok_shape_ok(batch, k, vocab)) {
        if (batch >= 0 && batch <= 65535 && k > kTokMaxK && vocab >= 1)
            return SPIRE_ERR_UNSUPPORTED;
        return SPIRE_ERR_INVALID_ARG;
    }
    if (batch == 0) return SPIRE_OK;              // nothing to do
    if (!p || !e || !out_tokens || !n_accepted || !workspace) return SPIRE_ERR_INVALID_ARG;
    if (k > 0 && (!q || !draft_tokens || !u)) return SPIRE_ERR_INVALID_ARG;
    if (!host_aligned(p, 4) || (q && !host_aligned(q, 4)) || !host_aligned(e, 4) ||
        (u && !host_aligned(u, 4)) || (draft_tokens && !host_aligned(draft_tokens, 4)) ||
        !host_aligned(out_tokens, 4) || !host_aligned(n_accepted, 4) ||
        !host_aligned(workspace, 256))
        return SPIRE_ERR_INVALID_ARG;
    if ((vocab & 3) == 0 && (!host_aligned(p, 16) || (q && !host_aligned(q, 16)) ||
                             !host_aligned(e, 16)))
        return SPIRE_ERR_INVALID_ARG;
    if (ws_bytes < tok_ws_bytes(batch, vocab)) return SPIRE_ERR_WORKSPACE;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char* ws = static_cast<char*>(workspace);
    TokParams tp{};
    tp.p = p;
    tp.q = q ? q : p;       // never read when k = 0
    tp.x = draft_tokens;
    tp.u = u;
    tp.e = e;
    tp.header = reinterpret_cast<int32_t*>(ws);
    tp.err = reinterpret_cast<int32_t*>(ws + 256);
    tp.out = out_tokens;
    tp.n_acc = n_accepted;
    tp.B = batch;
    tp.k = k;
    tp.V = vocab;
    if ((vocab & 3) != 0) {
        // rows not 16-byte aligned: the chunks are streamed with 4-byte loads
        tp.acc = nullptr;
        tp.part = reinterpret_cast<TokPartial*>(ws + 512 + tok_acc_bytes(batch));
        tp.S = (vocab + kTokChunk - 1) / kTokChunk;
        tokens_race_kernel<<<dim3((unsigned)tp.S, (unsigned)batch), kTokThreads, 0, st>>>(tp);
        if (cudaGetLastError() != cudaSuccess) return SPIRE_ERR_CUDA;
        tokens_finalize_kernel<<<(unsigned)((batch + 3) / 4), 128, 0, st>>>(tp);
        return cudaGetLastError() == cudaSuccess ? SPIRE_OK : SPIRE_ERR_CUDA;
    }
    int sms = 0, smem_optin = 0;
    if (host_device_info(&sms, &smem_optin) != SPIRE_OK) return SPIRE_ERR_CUDA;
    constexpr int kStreamSmem = kTokStages * 3 * kTokSub * 4;
    if (smem_optin < kStreamSmem + 1024) return SPIRE_ERR_UNSUPPORTED;
    static std::atomic<int> smem_set[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SPIRE_ERR_CUDA;
    if (dev < 0 || dev >= 64 || !smem_set[dev].load(std::memory_order_acquire)) {
        if (cudaFuncSetAttribute(tokens_stream_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kStreamSmem) != cudaSuccess)
            return SPIRE_ERR_CUDA;
        if (dev >= 0 && dev < 64) smem_set[dev].store(1, std::memory_order_release);
    }
    tp.acc = reinterpret_cast<TokAccept*>(ws + 512);
    tp.part = reinterpret_cast<TokPartial*>(ws + 512 + tok_acc_bytes(batch));
    tp.S = (vocab + kTokUnit - 1) / kTokUnit;
    tokens_accept_kernel<<<(unsigned)((batch + 3) / 4), 128, 0, st>>>(tp);
    if (cudaGetLastError() != cudaSuccess) return SPIRE_ERR_CUDA;
    const long long units = (long long)batch * tp.S;
    const long long ctas = (long long)kTokStreamCtas * sms;
    const long long grid = units < ctas ? units : ctas;
    if (launch_dependent(tokens_stream_kernel, dim3((unsigned)grid), dim3(kTokStreamThreads),
                         (size_t)kStreamSmem, st, tp) != cudaSuccess)
        return SPIRE_ERR_CUDA;
    return launch_dependent(tokens_finalize_kernel, dim3((unsigned)((batch + 3) / 4)), dim3(128),
                            0, st, tp) == cudaSuccess
               ? SPIRE_OK
               : SPIRE_ERR_CUDA;
}

}  // extern "C"
