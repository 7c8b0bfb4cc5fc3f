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
// Two launches:
//   tokens_race_kernel      grid (vocabulary chunks, B).  Each CTA finds j from
//                           the k gathered probabilities, streams its chunk of
//                           the rows p_{j+1}, q_{j+1} and E with 16-byte loads
//                           and reduces the best (score, index) key of the
//                           residual and of p alone; one partial per CTA.
//   tokens_finalize_kernel  one warp per sequence: the best key over the
//                           chunks (the maximum is unique, so the order of the
//                           reduction cannot matter), the emitted tokens and j.
// Only the rows a round actually needs are read: about 12 V bytes per sequence
// against the (2k + 1) * 4 V bytes of all its distributions.
#include <cmath>
#include <cstdint>

#include <cuda_runtime.h>

#include "spire.h"
#include "spire_common.cuh"
#include "spire_host.h"

namespace spire {
namespace {

constexpr int kTokThreads = 256;
constexpr int kTokChunk = 8192;          // vocabulary entries per CTA
constexpr int kTokMaxK = 31;
constexpr uint32_t kTokErrToken = 1u;    // SPIRE_DEVERR_CTX_LEN: a draft token outside [0, V)
constexpr uint32_t kTokErrValue = 8u;    // SPIRE_DEVERR_VALUE: an E value not > 0, or no draw

struct TokPartial {
    unsigned long long key_res;   // best residual candidate of the chunk (0: none)
    unsigned long long key_p;     // best candidate of p alone
    int32_t j;                    // accepted drafts (every CTA of b finds the same)
    int32_t flags;
};

struct TokParams {
    const float* p;       // [B, k+1, V]
    const float* q;       // [B, k, V]
    const int32_t* x;     // [B, k]
    const float* u;       // [B, k]
    const float* e;       // [B, V]
    TokPartial* part;     // [B, S]
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

__global__ void __launch_bounds__(128) tokens_finalize_kernel(const TokParams p) {
    // one warp per sequence: lanes take the chunks' partials, shuffles find the best
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
    return B >= 1 && B <= 65535 && k >= 0 && k <= kTokMaxK && V >= 1 && V <= (1 << 30) &&
           (long long)B * (k + 1) * V < (1LL << 40);
}

size_t tok_ws_bytes(int32_t B, int32_t V) {
    const long long S = (V + kTokChunk - 1) / kTokChunk;
    return 512 + (size_t)B * S * sizeof(TokPartial);
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
    if (!p || !e || !out_tokens || !n_accepted || !workspace) return SPIRE_ERR_INVALID_ARG;
    if (k > 0 && (!q || !draft_tokens || !u)) return SPIRE_ERR_INVALID_ARG;
    if (!tok_shape_ok(batch, k, vocab)) {
        if (batch >= 1 && k > kTokMaxK && vocab >= 1) return SPIRE_ERR_UNSUPPORTED;
        return SPIRE_ERR_INVALID_ARG;
    }
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
    tp.part = reinterpret_cast<TokPartial*>(ws + 512);
    tp.header = reinterpret_cast<int32_t*>(ws);
    tp.err = reinterpret_cast<int32_t*>(ws + 256);
    tp.out = out_tokens;
    tp.n_acc = n_accepted;
    tp.B = batch;
    tp.k = k;
    tp.V = vocab;
    tp.S = (vocab + kTokChunk - 1) / kTokChunk;
    tokens_race_kernel<<<dim3((unsigned)tp.S, (unsigned)batch), kTokThreads, 0, st>>>(tp);
    if (cudaGetLastError() != cudaSuccess) return SPIRE_ERR_CUDA;
    tokens_finalize_kernel<<<(unsigned)((batch + 3) / 4), 128, 0, st>>>(tp);
    return cudaGetLastError() == cudaSuccess ? SPIRE_OK : SPIRE_ERR_CUDA;
}

}  // extern "C"
