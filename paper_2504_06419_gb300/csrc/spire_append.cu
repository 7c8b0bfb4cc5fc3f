// spire_append.cu -- the draft step's feedback-memory append (include/spire.h:
// spire_feedback_append): per draft layer i and sequence b
//     m[i, b]  = softmax(w_i)-weighted mean of the activations x[0..n_act-1, b]
//     y[i, b]  = W_i m[i, b]      (W_i = [key rows; value rows], F = 2*Hkv*D rows)
// keys optionally turned by the entry's position, rounded to bf16 and stored
// in slot(pos[b]) of layer i's bounded cache (Section 3.3, per-layer memory
// equation; Section 3.1 for the cache and the position).
//
// Two launches on the caller's stream:
//   append_gemm_kernel      tcgen05 GEMM, split over K.  CTA (i, 128-row block
//                           of W_i, token block of N, K range) accumulates
//                           W_i[rows, K range] . m[tokens, K range]^T in tensor
//                           memory: warp 0 streams W tiles with TMA (128 rows x
//                           64 columns, 128-byte swizzle); warps 2..5 build the
//                           matching m tile (N tokens x 64 columns) from x in
//                           shared memory, in the same swizzled K-major layout,
//                           as two bf16 parts m = m_hi + m_lo; warp 1 issues two
//                           MMAs per 16 columns (M = 128, N, K = 16, A = W tile,
//                           B = m_hi / m_lo) into one fp32 accumulator.  Warps
//                           2..5 then write the accumulator (one TMEM lane = one
//                           row of W) as fp32 partials [split][i][token][row].
//   append_finalize_kernel  sums the partials in split order (double), turns
//                           key pairs (d, d + D/2) by pos * theta^(-2d/D) in
//                           double precision, rounds once to bf16 and writes the
//                           slot.  A negative position writes nothing and sets
//                           the device error word.
//
// The weights are read once (the only large operand: n_dl * F * d_model * 2
// bytes); x (n_act * B * d_model * 2 bytes) is re-read from L2 by every row
// block.  The m split keeps about 16 significant bits of the fp32 mix, and
// the accumulation is fp32, so the stored entry is within one bf16 unit of
// the exactly rounded value.
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

constexpr int kAppendThreads = 192;       // producer, MMA issuer, 4 mix / epilogue warps
constexpr int kAppendMaxStages = 8;
constexpr int kAppendMaxSplit = 8;
constexpr int kAppendMaxN = 256;          // tokens per CTA (MMA N)
constexpr int kATile = 128 * 64 * 2;      // one W tile: 128 rows x 64 columns bf16

struct AppendGemmParams {
    const __nv_bfloat16* x;   // [n_act, B, d_model]
    const float* mix_w;       // [n_dl, n_act]
    float* part;              // [ksplit, n_dl, B, F]
    int32_t* header;          // header[0] = number of error words
    int32_t* err;
    int B, n_act, n_dl, d_model, F, N, ntb, mtiles, ksplit, kblocks, nst;
};

struct AppendFinalParams {
    const float* part;
    const int32_t* pos;
    __nv_bfloat16* kv;        // [n_dl, B, 2, Hkv, S, D]
    int32_t* err;
    int B, n_dl, F, Hkv, D, S, n_sink, window, ksplit;
    double theta;
};

// Shared-memory layout of one stage: the W tile, then m_hi and m_lo (N rows
// of 128 bytes each, 128-byte swizzled).  All parts start 1024-byte aligned.
__host__ __device__ constexpr int stage_bytes(int N) { return kATile + 2 * N * 128; }

__global__ void __launch_bounds__(kAppendThreads, 1)
    append_gemm_kernel(const __grid_constant__ CUtensorMap tmap_w, const AppendGemmParams p) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t bars[3 * kAppendMaxStages + 2];
    __shared__ uint32_t tmem_slot;
    __shared__ float mixw[16];

    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* const sbase = smem_raw + (base - raw);
    const int STG = stage_bytes(p.N);
    const uint32_t bar0 = smem_u32(bars);
    const uint32_t bar_afull = bar0, bar_bfull = bar0 + 8 * kAppendMaxStages;
    const uint32_t bar_empty = bar0 + 16 * kAppendMaxStages;
    const uint32_t bar_acc = bar0 + 24 * kAppendMaxStages, bar_drain = bar_acc + 8;

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
    while ((int)tcols < p.N) tcols <<= 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < nst; ++s) {
            mbar_init(bar_afull + 8 * s, 1);
            mbar_init(bar_bfull + 8 * s, 4);
            mbar_init(bar_empty + 8 * s, 1);
        }
        mbar_init(bar_acc, 1);
        mbar_init(bar_drain, 1);
        fence_barrier_init();
        if (blockIdx.x == 0) {
            p.header[0] = 1;
            p.err[0] = 0;
        }
    }
    if (threadIdx.x < 32) {
        // softmax of this layer's mixing weights, in fp32
        float wmax = -INFINITY;
        for (int l = 0; l < p.n_act; ++l) wmax = fmaxf(wmax, p.mix_w[li * p.n_act + l]);
        float z = 0.f, a = 0.f;
        for (int l = 0; l < p.n_act; ++l) {
            const float e = expf(p.mix_w[li * p.n_act + l] - wmax);
            z += e;
            if (l == lane) a = e;
        }
        if (lane < p.n_act) mixw[lane] = a / z;
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

    if (warp == 0) {
        // ------------------------------------------------ W tiles by TMA
        if (lane == 0) {
            prefetch_tensormap(&tmap_w);
            const uint64_t pol = policy_evict_first();
            uint32_t armed = 0, armed_par = 0;
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int kb = kb0; kb < kb1; ++kb) {
                if (!mbar_wait(bar_empty + 8 * s, ph ^ 1)) { ok = false; break; }
                mbar_arrive_expect_tx(bar_afull + 8 * s, kATile);
                tma_load_2d(base + s * STG, &tmap_w, kb * 64, li * p.F + mt * 128, bar_afull + 8 * s,
                            pol);
                armed |= 1u << s;
                armed_par = (armed_par & ~(1u << s)) | (ph << s);
                if (++s == nst) { s = 0; ph ^= 1; }
            }
            if (!ok) {
                err |= kErrTimeout;
                for (int q = 0; q < nst; ++q)   // our copies land before shared memory goes away
                    if (armed & (1u << q)) mbar_wait(bar_afull + 8 * q, (armed_par >> q) & 1u);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, p.N, false);
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int kb = kb0; kb < kb1; ++kb) {
                if (!mbar_wait(bar_afull + 8 * s, ph) || !mbar_wait(bar_bfull + 8 * s, ph)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = base + s * STG, bh = a0 + kATile, bl = bh + p.N * 128;
#pragma unroll
                for (int k16 = 0; k16 < 4; ++k16) {
                    const uint64_t a = sdesc_sw128(a0 + 32 * k16, 16, 1024);
                    umma_bf16(tmem, a, sdesc_sw128(bh + 32 * k16, 16, 1024), idesc,
                              (kb > kb0 || k16 > 0) ? 1u : 0u);
                    umma_bf16(tmem, a, sdesc_sw128(bl + 32 * k16, 16, 1024), idesc, 1u);
                }
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
        // ------------------------------------------------ m tiles, then the epilogue
        const int tid = threadIdx.x - 64;          // 0..127
        const int c = tid & 7;                     // 16-byte chunk of the 128-byte row
        const int n_first = tid >> 3;              // rows n_first + 16 j
        int s = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int kb = kb0; kb < kb1 && ok; ++kb) {
            if (!mbar_wait(bar_empty + 8 * s, ph ^ 1)) { ok = false; break; }
            uint8_t* const bh = sbase + s * STG + kATile;
            uint8_t* const bl = bh + p.N * 128;
            for (int n = n_first; n < p.N; n += 16) {
                const int b = nt * p.N + n;
                float m[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) m[e] = 0.f;
                if (b < p.B) {
                    for (int l = 0; l < p.n_act; ++l) {
                        const uint4 v = __ldg(reinterpret_cast<const uint4*>(
                            p.x + ((long long)l * p.B + b) * p.d_model + kb * 64 + 8 * c));
                        const float a = mixw[l];
                        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            m[2 * e] = fmaf(a, bf16lo_to_f32(w4[e]), m[2 * e]);
                            m[2 * e + 1] = fmaf(a, bf16hi_to_f32(w4[e]), m[2 * e + 1]);
                        }
                    }
                }
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    hi[e] = pack_bf16(m[2 * e], m[2 * e + 1]);
                    lo[e] = pack_bf16(m[2 * e] - bf16lo_to_f32(hi[e]),
                                      m[2 * e + 1] - bf16hi_to_f32(hi[e]));
                }
                // row n of a 128-byte-swizzled K-major tile: 8-row atoms of 1024 bytes,
                // chunk c of row r stored at chunk c ^ (r mod 8)
                const int off = (n >> 3) * 1024 + (n & 7) * 128 + ((c ^ (n & 7)) << 4);
                *reinterpret_cast<uint4*>(bh + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                *reinterpret_cast<uint4*>(bl + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
            fence_proxy_async();   // the tile before the tensor core reads it
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_bfull + 8 * s);
            if (++s == nst) { s = 0; ph ^= 1; }
        }
        // epilogue: TMEM lane = W row, column = token
        if (ok && !mbar_wait(bar_acc, 0)) ok = false;
        if (!ok) {
            err |= kErrTimeout;
        } else {
            tc_fence_after();
            const int quarter = warp & 3;
            const int row = mt * 128 + 32 * quarter + lane;
            const uint32_t taddr = tmem + ((uint32_t)(32 * quarter) << 16);
            float* const dst = p.part + ((long long)ks * p.n_dl + li) * p.B * p.F + row;
            for (int c0 = 0; c0 < p.N; c0 += 16) {
                float v[16];
                tmem_ld16(taddr + c0, v);
                tmem_wait_ld();
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int b = nt * p.N + c0 + j;
                    if (b < p.B) dst[(long long)b * p.F] = v[j];
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

__global__ void __launch_bounds__(256) append_finalize_kernel(const AppendFinalParams p) {
    const int half = p.D / 2;
    const long long total = (long long)p.n_dl * p.B * 2 * p.Hkv * half;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        long long r = idx;
        const int d = (int)(r % half); r /= half;
        const int g = (int)(r % p.Hkv); r /= p.Hkv;
        const int kvi = (int)(r % 2); r /= 2;
        const int b = (int)(r % p.B);
        const int li = (int)(r / p.B);
        const int pos = p.pos[b];
        if (pos < 0) {
            if (d == 0 && g == 0 && kvi == 0 && li == 0) atomicOr(p.err, (int)kErrCtxLen);
            continue;
        }
        const int f0 = (kvi * p.Hkv + g) * p.D + d;
        double y0 = 0.0, y1 = 0.0;
        for (int ks = 0; ks < p.ksplit; ++ks) {
            const float* src = p.part + (((long long)ks * p.n_dl + li) * p.B + b) * p.F;
            y0 += (double)src[f0];
            y1 += (double)src[f0 + half];
        }
        if (kvi == 0 && p.theta > 0.0) {
            double sn, cs;
            sincos((double)pos * pow(p.theta, -2.0 * d / p.D), &sn, &cs);
            const double r0 = y0 * cs - y1 * sn, r1 = y1 * cs + y0 * sn;
            y0 = r0;
            y1 = r1;
        }
        const int slot = pos < p.n_sink ? pos : p.n_sink + (pos - p.n_sink) % p.window;
        __nv_bfloat16* const dst =
            p.kv + ((((long long)li * p.B + b) * 2 + kvi) * p.Hkv + g) * (long long)p.S * p.D +
            (long long)slot * p.D + d;
        dst[0] = __double2bfloat16(y0);
        dst[half] = __double2bfloat16(y1);
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
        (long long)d->n_sink + d->window > (1LL << 30))
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

constexpr size_t kAppendHeader = 512;   // header word + error word, then the partials

size_t append_ws_bytes(const spire_append_desc* d, const AppendPlan& pl) {
    return kAppendHeader + (size_t)pl.ksplit_max * d->num_draft_layers * d->batch * pl.F * 4;
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

    CUtensorMap tw;
    if (!encode_2d_bf16_map(&tw, w_kv, desc->d_model, (uint64_t)n_dl * pl.F, 64, 128))
        return SPIRE_ERR_CUDA;

    char* ws = static_cast<char*>(workspace);
    AppendGemmParams gp{};
    gp.x = static_cast<const __nv_bfloat16*>(x);
    gp.mix_w = mix_w;
    gp.part = reinterpret_cast<float*>(ws + kAppendHeader);
    gp.header = reinterpret_cast<int32_t*>(ws);
    gp.err = reinterpret_cast<int32_t*>(ws + 256);
    gp.B = B;
    gp.n_act = desc->num_act;
    gp.n_dl = n_dl;
    gp.d_model = desc->d_model;
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
    append_gemm_kernel<<<(unsigned)(tiles * ks), kAppendThreads, smem, st>>>(tw, gp);
    if (cudaGetLastError() != cudaSuccess) return SPIRE_ERR_CUDA;

    AppendFinalParams fp{};
    fp.part = gp.part;
    fp.pos = pos;
    fp.kv = static_cast<__nv_bfloat16*>(kv);
    fp.err = gp.err;
    fp.B = B;
    fp.n_dl = n_dl;
    fp.F = pl.F;
    fp.Hkv = desc->num_kv_heads;
    fp.D = desc->head_dim;
    fp.S = desc->n_sink + desc->window;
    fp.n_sink = desc->n_sink;
    fp.window = desc->window;
    fp.ksplit = (int)ks;
    fp.theta = (double)desc->rope_theta;
    const long long total = (long long)n_dl * B * pl.F / 2;
    long long blocks = (total + 255) / 256;
    if (blocks > 4LL * sms * 8) blocks = 4LL * sms * 8;
    append_finalize_kernel<<<(unsigned)blocks, 256, 0, st>>>(fp);
    return cudaGetLastError() == cudaSuccess ? SPIRE_OK : SPIRE_ERR_CUDA;
}

}  // extern "C"
