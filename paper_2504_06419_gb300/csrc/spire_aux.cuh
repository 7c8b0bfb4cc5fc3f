// spire_aux.cuh -- the split planner (a1) and the log-sum-exp combine (a3)
// kernels of libspire; included by exactly one translation unit.
#pragma once

#include "spire_kernels.cuh"

namespace spire {

// ============================================================== plan (a1)
__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_sums, int* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int s = (lane < (int)(blockDim.x >> 5)) ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += y;
        }
        warp_sums[lane] = s;   // inclusive prefix over warps
    }
    __syncthreads();
    int before = (warp > 0 ? warp_sums[warp - 1] : 0) + x - v;
    *total = warp_sums[(blockDim.x >> 5) - 1];
    __syncthreads();
    return before;
}

__global__ void __launch_bounds__(kPlanThreads) plan_kernel(PlanParams p) {
    __shared__ int warp_sums[32];
    __shared__ unsigned long long s_work;
    __shared__ int s_tail[kPlanSortMax];
    const int tid = threadIdx.x;
    if (tid == 0) {
        p.header[kHdrErr] = 0;
        p.header[kHdrCounter] = 0;
        s_work = 0ull;
    }
    __syncthreads();

    // pass 1: visible length and tile count per sequence; total work
    unsigned long long work = 0;
    for (int b = tid; b < p.B; b += blockDim.x) {
        const int L = p.ctx_lens[b];
        int valid, Leff;
        if (p.mode == kModeVerify) {
            valid = (L >= p.kp1) && ((long long)L <= (long long)p.max_pages * kPage);
            Leff = L;
        } else {
            valid = L >= 1;
            Leff = L < p.cap ? L : p.cap;
        }
        if (!valid) {
            atomicOr(&p.header[kHdrErr], (int)kErrCtxLen);
            Leff = 0;
        }
        const int tiles = (Leff + kPage - 1) / kPage;
        work += (unsigned long long)tiles;
        p.seq_info[b] = make_int4(Leff, tiles, 0, valid);
    }
    atomicAdd(&s_work, work);
    __syncthreads();
    const unsigned long long W = s_work * (unsigned long long)p.Hkv;
    const int min_chunk = p.mode == kModeVerify ? kMinChunkVerify : kMinChunkDraft;
    int chunk = (int)((W + kTargetItems - 1) / kTargetItems);
    if (chunk < min_chunk) chunk = min_chunk;

    // pass 2: splits per sequence and their prefix sums (chunks of blockDim)
    int carry = 0;
    for (int base = 0; base < p.B; base += blockDim.x) {
        const int b = base + tid;
        int4 si = b < p.B ? p.seq_info[b] : make_int4(0, 0, 0, 0);
        const int nsplit = (b < p.B) ? (si.w ? (si.y + chunk - 1) / chunk : 1) : 0;
        int total;
        const int excl = block_exclusive_scan(nsplit, warp_sums, &total);
        if (b < p.B) {
            const int tail = si.w ? si.y - chunk * (nsplit - 1) : 0;
            if (b < kPlanSortMax) s_tail[b] = tail;
            p.seq_info[b] = make_int4(si.x, nsplit, carry + excl, si.w);
        }
        carry += total;
    }
    const int n_full = (carry - p.B) * p.Hkv;   // splits before each sequence's last
    if (tid == 0) {
        p.header[kHdrItems] = n_full + p.B * p.Hkv;
        p.header[kHdrChunk] = chunk;
    }
    __syncthreads();

    // pass 3: emit items.  Full-length splits first; then each sequence's
    // last (shorter or equal) split, longest first, ties by sequence index.
    for (int b = tid; b < p.B; b += blockDim.x) {
        const int4 si = p.seq_info[b];
        const int nsplit = si.y;
        const int fbase = si.z - b;
        for (int s = 0; s < nsplit - 1; ++s)
            for (int g = 0; g < p.Hkv; ++g)
                p.items[(long long)(fbase + s) * p.Hkv + g] =
                    make_int4(b * p.Hkv + g, s * chunk, chunk, s);
        const int tail = si.w ? (si.x + kPage - 1) / kPage - chunk * (nsplit - 1) : 0;
        int rank = b;
        if (p.B <= kPlanSortMax) {
            rank = 0;
            for (int c = 0; c < p.B; ++c) {
                const int tc = s_tail[c];
                rank += (tc > tail) || (tc == tail && c < b);
            }
        }
        for (int g = 0; g < p.Hkv; ++g)
            p.items[(long long)n_full + (long long)rank * p.Hkv + g] =
                make_int4(b * p.Hkv + g, (nsplit - 1) * chunk, tail, nsplit - 1);
    }
}

// ============================================================== combine (a3)

__global__ void __launch_bounds__(256) combine_kernel(const CombineParams p) {
    const int pair = blockIdx.x;
    const int b = pair / p.Hkv, g = pair - b * p.Hkv;
    const int4 si = p.seq_info[b];
    const int nsplit = si.y;
    if (nsplit <= 1) return;
    const int D4 = p.D / 4;
    const float NEG_INF = __int_as_float(0xff800000);
    for (int idx = threadIdx.x; idx < p.R * D4; idx += blockDim.x) {
        const int r = idx / D4, d4 = idx - r * D4;
        float M = NEG_INF;
        bool nan = false;
        for (int s = 0; s < nsplit; ++s) {
            const float l = p.part_lse[(long long)((si.z + s) * p.Hkv + g) * p.R + r];
            nan |= (l != l);
            M = fmaxf(M, l);
        }
        const float Mr = (M == NEG_INF) ? 0.f : M;
        float den = 0.f;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s = 0; s < nsplit; ++s) {
            const long long row = (long long)((si.z + s) * p.Hkv + g) * p.R + r;
            const float w = ex2(p.part_lse[row] - Mr);
            den += w;
            const float4 v = *reinterpret_cast<const float4*>(p.part_o + row * p.D + 4 * d4);
            acc.x += w * v.x; acc.y += w * v.y; acc.z += w * v.z; acc.w += w * v.w;
        }
        float4 res;
        if (nan || !(den > 0.f)) {
            const float NANF = __int_as_float(0x7fc00000);
            res = make_float4(NANF, NANF, NANF, NANF);
        } else {
            const float inv = 1.f / den;
            res = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
        }
        const int i = r / p.G, hl = r - i * p.G;
        float* dst = p.out + ((long long)(b * p.kp1 + i) * p.Hq + g * p.G + hl) * p.D;
        *reinterpret_cast<float4*>(dst + 4 * d4) = res;
    }
}

}  // namespace spire
