// spire_append.cu -- the draft step's feedback-memory append (include/spire.h:
// spire_feedback_append): per draft layer i and sequence b
//     m[i, b]  = softmax(w_i)-weighted mean of the activations x[0..n_act-1, b]
//     y[i, b]  = W_i m[i, b]      (W_i = [key rows; value rows], F = 2*Hkv*D rows)
// keys optionally turned by the entry's position, rounded to bf16 and stored
// in slot(pos[b]) of layer i's bounded cache (Section 3.3, per-layer memory
// equation; Section 3.1 for the cache and the position).
//
// Three launches on the caller's stream:
//   append_mix_kernel       m[i, b, :] in fp32 from x and softmax(w_i), stored
//                           as two bf16 arrays m_hi = bf16(m), m_lo =
//                           bf16(m - m_hi) in the workspace (~16 significant
//                           bits together); clears the device error word.
//   append_gemm_kernel      tcgen05 GEMM, split over K.  CTA (i, 128-row block
//                           of W_i, token block of N, K range) accumulates
//                           W_i[rows, K range] . m[tokens, K range]^T in tensor
//                           memory: warp 0 streams, per 64 columns, the W tile
//                           (128 rows) and the m_hi and m_lo tiles (N tokens)
//                           with TMA (128-byte swizzle), the m_lo tile right
//                           after the m_hi tile; warp 1 issues one MMA per 16
//                           columns (M = 128, N = 2 x tokens, K = 16, A = W
//                           tile, B = the m_hi rows then the m_lo rows), so
//                           accumulator columns j and N + j hold the two parts
//                           of token j; warps 2..5 add them and write the sum
//                           (one TMEM lane = one row of W) as fp32 partials
//                           [split][i][token][row].
//   append_finalize_kernel  per four key / value pairs (d, d + D/2): sums the
//                           partials in split order, turns key pairs by the
//                           angle pos * theta^(-2d/D) (product and reduction
//                           modulo 2 pi in double, sine and cosine of the
//                           reduced angle in fp32), rounds to bf16 and writes
//                           the slot.  A negative position writes nothing and
//                           sets the device error word.
//
// The GEMM and the finalize are launched with programmatic dependent launch:
// their prologues overlap the kernel before them, and they wait
// (griddepcontrol.wait) only before reading what it wrote.  The rotary
// frequencies theta^(-2d/D) are per-call constants computed on the host in
// double and passed to the finalize.
//
// The weights are read once (the only large operand: n_dl * F * d_model * 2
// bytes); m (2 * n_dl * B * d_model * 2 bytes) is re-read from L2 by every row
// block.  With fp32 accumulation an entry is within one bf16 unit of the
// exactly rounded value plus ~2^-16 of sum_c |W_c m_c|.
#include <atomic>
#include <cmath>
#include <cstdint>

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "spire.h"
#include "spire_common.cuh"
#include "spire_host.h"

namespace spire {
namespace {

constexpr int kAppendThreads = 192;       // producer, MMA issuer, 4 epilogue warps
constexpr int kAppendMaxStages = 8;
constexpr int kAppendMaxSplit = 8;
constexpr int kAppendMaxN = 128;          // tokens per CTA (MMA N = 2 x tokens: m_hi, m_lo)
constexpr int kATile = 128 * 64 * 2;      // one W tile: 128 rows x 64 columns bf16

struct AppendMixParams {
    const __nv_bfloat16* x;   // [n_act, B, d_model]
    const float* mix_w;       // [n_dl, n_act]
    __nv_bfloat16* m;         // [2 (hi, lo), n_dl, B, d_model]
    int32_t* header;          // header[0] = number of error words
    int32_t* err;
    int B, n_act, n_dl, d_model;
};

struct AppendGemmParams {
    float* part;              // [ksplit, n_dl, B, F]
    int32_t* err;
    int B, n_dl, F, N, ntb, mtiles, ksplit, kblocks, nst;
};

struct AppendFinalParams {
    const float* part;
    const int32_t* pos;
    __nv_bfloat16* kv;        // [n_dl, B, 2, Hkv, S, D]
    int32_t* err;
    int B, n_dl, F, Hkv, D, S, n_sink, window, ksplit, rotate;
    double freq[64];          // theta^(-2d/D), d < D/2
};

// Shared-memory layout of one stage: the W tile, then the m_hi and m_lo tiles
// (N rows of 128 bytes each, 128-byte swizzled).  All parts start 1024-byte
// aligned.
__host__ __device__ constexpr int stage_bytes(int N) { return kATile + 2 * N * 128; }

__global__ void __launch_bounds__(256) append_mix_kernel(const AppendMixParams p) {
    __shared__ float a[16 * 16];                 // softmax(w_i), [n_dl][n_act]
    grid_dep_launch_dependents();                // the GEMM may start its prologue
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        p.header[0] = 1;
        p.err[0] = 0;
    }
    if (threadIdx.x < p.n_dl) {
        const int i = threadIdx.x;
        float wmax = -INFINITY;
        for (int l = 0; l < p.n_act; ++l) wmax = fmaxf(wmax, p.mix_w[i * p.n_act + l]);
        float z = 0.f;
        for (int l = 0; l < p.n_act; ++l) {
            const float e = expf(p.mix_w[i * p.n_act + l] - wmax);
            a[i * 16 + l] = e;
            z += e;
        }
        for (int l = 0; l < p.n_act; ++l) a[i * 16 + l] /= z;
    }
    __syncthreads();
    const int c8 = p.d_model / 8;                // 8-column groups per row
    const long long total = (long long)p.n_dl * p.B * c8;
    const long long plane = (long long)p.n_dl * p.B * p.d_model;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c = (int)(idx % c8);
        const long long ib = idx / c8;           // i * B + b
        const int b = (int)(ib % p.B), i = (int)(ib / p.B);
        float m[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) m[e] = 0.f;
        for (int l = 0; l < p.n_act; ++l) {
            const uint4 v = __ldg(reinterpret_cast<const uint4*>(
                p.x + ((long long)l * p.B + b) * p.d_model + 8 * c));
            const float w = a[i * 16 + l];
            const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                m[2 * e] = fmaf(w, bf16lo_to_f32(w4[e]), m[2 * e]);
                m[2 * e + 1] = fmaf(w, bf16hi_to_f32(w4[e]), m[2 * e + 1]);
            }
        }
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            hi[e] = pack_bf16(m[2 * e], m[2 * e + 1]);
            lo[e] = pack_bf16(m[2 * e] - bf16lo_to_f32(hi[e]), m[2 * e + 1] - bf16hi_to_f32(hi[e]));
        }
        const long long o = ib * p.d_model + 8 * c;
        *reinterpret_cast<uint4*>(p.m + o) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        *reinterpret_cast<uint4*>(p.m + plane + o) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    }
}

__global__ void __launch_bounds__(kAppendThreads, 1)
    append_gemm_kernel(const __grid_constant__ CUtensorMap tmap_w,
                       const __grid_constant__ CUtensorMap tmap_m, const AppendGemmParams p) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t bars[2 * kAppendMaxStages + 2];
    __shared__ uint32_t tmem_slot;

    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    const int STG = stage_bytes(p.N);
    const uint32_t mbytes = (uint32_t)p.N * 128;
    const uint32_t bar0 = smem_u32(bars);
    const uint32_t bar_full = bar0, bar_empty = bar0 + 8 * kAppendMaxStages;
    const uint32_t bar_acc = bar0 + 16 * kAppendMaxStages, bar_drain = bar_acc + 8;

    // this CTA's tile: layer i, W rows [128 mt, +128), tokens [N nt, +N), K blocks [kb0, kb1)
    int t = blockIdx.x;
    const int ks = t % p.ksplit; t /= p.ksplit;
    const int nt = t % p.ntb; t /= p.ntb;
    const int mt = t % p.mtiles;
    const int li = t / p.mtiles;
    const int kb0 = (int)((long long)ks * p.kblocks / p.ksplit);
    const int kb1 = (int)((long long)(ks + 1) * p.kblocks / p.ksplit);
    const int nst = p.nst;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t tcols = 32;
    while ((int)tcols < 2 * p.N) tcols <<= 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < nst; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, 1);
        }
        mbar_init(bar_acc, 1);
        mbar_init(bar_drain, 1);
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(&tmem_slot), tcols);
        tmem_relinquish();
        tc_fence_before();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    uint32_t err = 0;
    grid_dep_launch_dependents();                // the finalize may start its prologue
    // m and the cleared error word come from the mix kernel
    grid_dep_wait();

    if (warp == 0) {
        // ------------------------------------------------ W, m_hi, m_lo tiles by TMA
        if (lane == 0) {
            prefetch_tensormap(&tmap_w);
            prefetch_tensormap(&tmap_m);
            const uint64_t pol = policy_evict_first();
            const int yh = li * p.B + nt * p.N;          // m_hi rows; m_lo rows n_dl * B later
            const int yl = yh + p.n_dl * p.B;
            uint32_t armed = 0, armed_par = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int kb = kb0; kb < kb1; ++kb) {
                if (!mbar_wait(bar_empty + 8 * s, ph ^ 1)) { ok = false; break; }
                const uint32_t dst = base + s * STG, bar = bar_full + 8 * s;
                mbar_arrive_expect_tx(bar, kATile + 2 * mbytes);
                tma_load_2d(dst, &tmap_w, kb * 64, li * p.F + mt * 128, bar, pol);
                tma_load_2d(dst + kATile, &tmap_m, kb * 64, yh, bar, pol);
                tma_load_2d(dst + kATile + mbytes, &tmap_m, kb * 64, yl, bar, pol);
                armed |= 1u << s;
                armed_par = (armed_par & ~(1u << s)) | (ph << s);
                if (++s == nst) { s = 0; ph ^= 1; }
            }
            if (!ok) {
                err |= kErrTimeout;
                for (int q = 0; q < nst; ++q)   // our copies land before shared memory goes away
                    if (armed & (1u << q)) mbar_wait(bar_full + 8 * q, (armed_par >> q) & 1u);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, 2 * p.N, false);
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int kb = kb0; kb < kb1; ++kb) {
                if (!mbar_wait(bar_full + 8 * s, ph)) { ok = false; break; }
                tc_fence_after();
                const uint32_t a0 = base + s * STG, bm = a0 + kATile;   // m_hi rows, then m_lo
#pragma unroll
                for (int k16 = 0; k16 < 4; ++k16)
                    umma_bf16(tmem, sdesc_sw128(a0 + 32 * k16, 16, 1024),
                              sdesc_sw128(bm + 32 * k16, 16, 1024), idesc,
                              (kb > kb0 || k16 > 0) ? 1u : 0u);
                umma_commit(bar_empty + 8 * s);
                if (++s == nst) { s = 0; ph ^= 1; }
            }
            if (ok) umma_commit(bar_acc);
            else err |= kErrTimeout;
            umma_commit(bar_drain);   // every MMA has finished before TMEM is freed
            if (!mbar_wait(bar_drain, 0)) err |= kErrTimeout;
        }
        __syncwarp();
    } else {
        // ------------------------------------------------ epilogue: TMEM lane = W row
        if (!mbar_wait(bar_acc, 0)) {
            err |= kErrTimeout;
        } else {
            tc_fence_after();
            const int quarter = warp & 3;
            const int row = mt * 128 + 32 * quarter + lane;
            const uint32_t taddr = tmem + ((uint32_t)(32 * quarter) << 16);
            float* const dst = p.part + ((long long)ks * p.n_dl + li) * p.B * p.F + row;
            for (int c0 = 0; c0 < p.N; c0 += 16) {
                float vh[16], vl[16];
                tmem_ld16(taddr + c0, vh);
                tmem_ld16(taddr + p.N + c0, vl);
                tmem_wait_ld();
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int b = nt * p.N + c0 + j;
                    if (b < p.B) dst[(long long)b * p.F] = vh[j] + vl[j];
                }
            }
        }
        tc_fence_before();
    }
    if (err) atomicOr(p.err, (int)err);
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, tcols);
    }
}

__global__ void __launch_bounds__(64) append_finalize_kernel(const AppendFinalParams p) {
    grid_dep_wait();                             // the GEMM's partials
    const int half = p.D / 2, q4 = half / 4;     // four pairs (d .. d + 3, + D/2) per thread
    const double kTwoPi = 6.283185307179586476925286766559;
    const double kInvTwoPi = 0.15915494309189533576888376337251;
    const long long total = (long long)p.n_dl * p.B * p.Hkv * q4;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        long long r = idx;
        const int d = 4 * (int)(r % q4); r /= q4;
        const int g = (int)(r % p.Hkv); r /= p.Hkv;
        const int b = (int)(r % p.B);
        const int li = (int)(r / p.B);
        const int pos = p.pos[b];
        if (pos < 0) {
            if (d == 0 && g == 0 && li == 0) atomicOr(p.err, (int)kErrCtxLen);
            continue;
        }
        // the split partials of the key (kvi 0) and value (kvi 1) pairs, summed in split order
        float y[2][2][4];
#pragma unroll
        for (int kvi = 0; kvi < 2; ++kvi)
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int e = 0; e < 4; ++e) y[kvi][h][e] = 0.f;
        for (int ks = 0; ks < p.ksplit; ++ks) {
            const float* src = p.part + (((long long)ks * p.n_dl + li) * p.B + b) * p.F;
#pragma unroll
            for (int kvi = 0; kvi < 2; ++kvi)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const float4 v = __ldg(reinterpret_cast<const float4*>(
                        src + (kvi * p.Hkv + g) * p.D + h * half + d));
                    y[kvi][h][0] += v.x; y[kvi][h][1] += v.y;
                    y[kvi][h][2] += v.z; y[kvi][h][3] += v.w;
                }
        }
        if (p.rotate) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                // the angle is exact enough only in double (pos up to 2^31); the reduced
                // angle in [-pi, pi] keeps fp32 accuracy through sincosf
                const double ang = (double)pos * p.freq[d + e];
                const double red = fma(-kTwoPi, rint(ang * kInvTwoPi), ang);
                float sn, cs;
                sincosf((float)red, &sn, &cs);
                const float r0 = y[0][0][e] * cs - y[0][1][e] * sn;
                const float r1 = y[0][1][e] * cs + y[0][0][e] * sn;
                y[0][0][e] = r0;
                y[0][1][e] = r1;
            }
        }
        const int slot = pos < p.n_sink ? pos : p.n_sink + (pos - p.n_sink) % p.window;
#pragma unroll
        for (int kvi = 0; kvi < 2; ++kvi) {
            __nv_bfloat16* const dst =
                p.kv + ((((long long)li * p.B + b) * 2 + kvi) * p.Hkv + g) * (long long)p.S * p.D +
                (long long)slot * p.D + d;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const uint32_t w0 = pack_bf16(y[kvi][h][0], y[kvi][h][1]);
                const uint32_t w1 = pack_bf16(y[kvi][h][2], y[kvi][h][3]);
                *reinterpret_cast<uint2*>(dst + h * half) = make_uint2(w0, w1);
            }
        }
    }
}

struct AppendPlan {
    int F, N, ntb, mtiles, kblocks, ksplit_max;
};

bool plan_append(const spire_append_desc* d, AppendPlan* pl) {
    if (!d) return false;
    if (d->batch < 1 || d->num_act < 1 || d->num_act > 16 || d->num_draft_layers < 1 ||
        d->num_draft_layers > 16 || d->d_model < 64 || d->d_model > 65536 ||
        d->d_model % 64 != 0 || d->num_kv_heads < 1 || (d->head_dim != 64 && d->head_dim != 128) ||
        d->n_sink < 0 || d->window < 1 || !std::isfinite(d->rope_theta) || d->rope_theta < 0.f)
        return false;
    const long long F = 2LL * d->num_kv_heads * d->head_dim;
    if (F * d->num_draft_layers > (1LL << 30) ||
        (long long)d->n_sink + d->window > (1LL << 30) ||
        2LL * d->num_draft_layers * d->batch > (1LL << 30))
        return false;
    pl->F = (int)F;
    const int nb = d->batch < kAppendMaxN ? d->batch : kAppendMaxN;
    pl->N = (nb + 15) / 16 * 16;
    pl->ntb = (d->batch + pl->N - 1) / pl->N;
    pl->mtiles = (int)(F / 128);
    pl->kblocks = d->d_model / 64;
    const long long tiles = (long long)d->num_draft_layers * pl->mtiles * pl->ntb;
    long long km = 256 / tiles;   // split bound for any GPU of up to 256 SMs
    if (km > kAppendMaxSplit) km = kAppendMaxSplit;
    if (km > pl->kblocks) km = pl->kblocks;
    pl->ksplit_max = km < 1 ? 1 : (int)km;
    return true;
}

// workspace: header word | error word | (reserved) | m_hi, m_lo | partials
constexpr size_t kAppendHeader = 512;
constexpr size_t kAppendFreq = 512;

size_t append_m_bytes(const spire_append_desc* d) {
    return (((size_t)2 * d->num_draft_layers * d->batch * d->d_model * 2) + 255) & ~size_t(255);
}

size_t append_ws_bytes(const spire_append_desc* d, const AppendPlan& pl) {
    return kAppendHeader + kAppendFreq + append_m_bytes(d) +
           (size_t)pl.ksplit_max * d->num_draft_layers * d->batch * pl.F * 4;
}

}  // namespace
}  // namespace spire

using namespace spire;

extern "C" {

size_t spire_feedback_append_workspace_bytes(const spire_append_desc* desc) {
    AppendPlan pl;
    if (!plan_append(desc, &pl)) return 0;
    return append_ws_bytes(desc, pl);
}

spire_status spire_feedback_append(const void* x, const float* mix_w, const void* w_kv,
                                   const int32_t* pos, const spire_append_desc* desc, void* kv,
                                   void* workspace, size_t ws_bytes, void* stream) {
    AppendPlan pl;
    if (!x || !mix_w || !w_kv || !pos || !kv || !workspace) return SPIRE_ERR_INVALID_ARG;
    if (!plan_append(desc, &pl)) {
        if (desc && desc->head_dim != 64 && desc->head_dim != 128 && desc->batch >= 1)
            return SPIRE_ERR_UNSUPPORTED;
        return SPIRE_ERR_INVALID_ARG;
    }
    if (!host_aligned(x, 16) || !host_aligned(w_kv, 16) || !host_aligned(kv, 16) ||
        !host_aligned(mix_w, 4) || !host_aligned(pos, 4) || !host_aligned(workspace, 256))
        return SPIRE_ERR_INVALID_ARG;
    if (ws_bytes < append_ws_bytes(desc, pl)) return SPIRE_ERR_WORKSPACE;
    int sms = 0, smem_optin = 0;
    if (host_device_info(&sms, &smem_optin) != SPIRE_OK) return SPIRE_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);

    const int B = desc->batch, n_dl = desc->num_draft_layers;
    const long long tiles = (long long)n_dl * pl.mtiles * pl.ntb;
    long long ks = sms / tiles;
    if (ks < 1) ks = 1;
    if (ks > pl.ksplit_max) ks = pl.ksplit_max;
    const int STG = stage_bytes(pl.N);
    int nst = (smem_optin - 2048) / STG;   // 1 KB alignment slack, 1 KB for static shared memory
    if (nst > kAppendMaxStages) nst = kAppendMaxStages;
    if (nst < 2) return SPIRE_ERR_UNSUPPORTED;
    const size_t smem = 1024 + (size_t)nst * STG;

    char* ws = static_cast<char*>(workspace);
    __nv_bfloat16* const mbuf = reinterpret_cast<__nv_bfloat16*>(ws + kAppendHeader + kAppendFreq);
    CUtensorMap tw, tm;
    if (!encode_2d_bf16_map(&tw, w_kv, desc->d_model, (uint64_t)n_dl * pl.F, 64, 128) ||
        !encode_2d_bf16_map(&tm, mbuf, desc->d_model, (uint64_t)2 * n_dl * B, 64, pl.N))
        return SPIRE_ERR_CUDA;

    AppendMixParams mp{};
    mp.x = static_cast<const __nv_bfloat16*>(x);
    mp.mix_w = mix_w;
    mp.m = mbuf;
    mp.header = reinterpret_cast<int32_t*>(ws);
    mp.err = reinterpret_cast<int32_t*>(ws + 256);
    mp.B = B;
    mp.n_act = desc->num_act;
    mp.n_dl = n_dl;
    mp.d_model = desc->d_model;
    const long long mix_items = (long long)n_dl * B * (desc->d_model / 8);
    long long mblocks = (mix_items + 255) / 256;
    if (mblocks > 8LL * sms) mblocks = 8LL * sms;
    append_mix_kernel<<<(unsigned)mblocks, 256, 0, st>>>(mp);
    if (cudaGetLastError() != cudaSuccess) return SPIRE_ERR_CUDA;

    AppendGemmParams gp{};
    gp.part = reinterpret_cast<float*>(ws + kAppendHeader + kAppendFreq + append_m_bytes(desc));
    gp.err = mp.err;
    gp.B = B;
    gp.n_dl = n_dl;
    gp.F = pl.F;
    gp.N = pl.N;
    gp.ntb = pl.ntb;
    gp.mtiles = pl.mtiles;
    gp.ksplit = (int)ks;
    gp.kblocks = pl.kblocks;
    gp.nst = nst;
    // the kernel's dynamic shared memory limit, raised once per device to the
    // largest size used so far
    static std::atomic<int> smem_set[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SPIRE_ERR_CUDA;
    if (dev < 0 || dev >= 64 || smem_set[dev].load(std::memory_order_acquire) < (int)smem) {
        if (cudaFuncSetAttribute(append_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem) != cudaSuccess)
            return SPIRE_ERR_CUDA;
        if (dev >= 0 && dev < 64) {
            int cur = smem_set[dev].load(std::memory_order_acquire);
            while (cur < (int)smem &&
                   !smem_set[dev].compare_exchange_weak(cur, (int)smem, std::memory_order_acq_rel)) {
            }
        }
    }
    if (launch_dependent(append_gemm_kernel, dim3((unsigned)(tiles * ks)), dim3(kAppendThreads),
                         smem, st, tw, tm, gp) != cudaSuccess)
        return SPIRE_ERR_CUDA;

    AppendFinalParams fp{};
    fp.part = gp.part;
    fp.pos = pos;
    for (int d = 0; d < desc->head_dim / 2; ++d)     // the same libm pow as the definition
        fp.freq[d] = desc->rope_theta > 0.f
                         ? std::pow((double)desc->rope_theta, -2.0 * d / desc->head_dim)
                         : 0.0;
    fp.kv = static_cast<__nv_bfloat16*>(kv);
    fp.err = mp.err;
    fp.B = B;
    fp.n_dl = n_dl;
    fp.F = pl.F;
    fp.Hkv = desc->num_kv_heads;
    fp.D = desc->head_dim;
    fp.S = desc->n_sink + desc->window;
    fp.n_sink = desc->n_sink;
    fp.window = desc->window;
    fp.ksplit = (int)ks;
    fp.rotate = desc->rope_theta > 0.f;
    const long long total = (long long)n_dl * B * desc->num_kv_heads * (desc->head_dim / 8);
    // small blocks so that the few threads reach every SM
    long long blocks = (total + 63) / 64;
    if (blocks > 16LL * sms) blocks = 16LL * sms;
    return launch_dependent(append_finalize_kernel, dim3((unsigned)blocks), dim3(64), 0, st, fp) ==
                   cudaSuccess
               ? SPIRE_OK
               : SPIRE_ERR_CUDA;
}

}  // extern "C"
