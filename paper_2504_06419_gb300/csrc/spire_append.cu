// spire_append.cu -- the draft step's feedback-memory append (include/spire.h:
// spire_feedback_append): per draft layer i and sequence b
//     m[i, b]  = softmax(w_i)-weighted mean of the activations x[0..n_act-1, b]
//     y[i, b]  = W_i m[i, b]      (W_i = [key rows; value rows], F = 2*Hkv*D rows)
// keys optionally turned by the entry's position, rounded to bf16 and stored
// in slot(pos[b]) of layer i's bounded cache (Section 3.3, per-layer memory
// equation; Section 3.1 for the cache and the position).
//
// The projection is linear, so W_i m = sum_l a_il (W_i x_l) with a_i =
// softmax(w_i): the kernel multiplies the weights by the bf16 activations
// themselves (exact products, fp32 accumulation) and mixes the n_act
// accumulators with a_i in fp32 afterwards.  No memory vector is formed, so
// no rounding of m enters the result.
//
// One launch (append_kernel, programmatic dependent launch) in thread-block
// clusters of KS CTAs that split d_model (K) among them.  CTA (layer i, MT
// row tiles of 128 rows of W_i, token block of N, K range of cluster rank r),
// one per SM, 12 warps:
//   warp 0     streams the MT W tiles of each 64 columns of its K range by TMA
//              (128-byte swizzle, evict-first) into a deep ring: W comes from
//              HBM, the long-latency stream;
//   warp 2     streams the n_act activation tiles of its tokens (one 3-D box,
//              activation-major, evict-last: every row tile re-reads them,
//              mostly from L2) into a second, shallower ring;
//   warp 1     issues per 16 columns one tcgen05.mma per row tile (M = 128,
//              N = n_act x N over the adjacent activation tiles), so that
//              tensor-memory column t*TS + l*N + j (TS = n_act x N rounded up
//              to 32) holds W_t x_l for token j;
//   warps 4-11 (two per TMEM lane quarter; one lane = one row of W) mix the
//              accumulators, y = sum_l a_l acc_l in fp32, into the CTA's
//              partial [tile][token][row] over its drained rings.
// After one cluster barrier CTA q takes tokens [q N / KS, (q + 1) N / KS):
// for four adjacent key / value pairs (d .. d + 3, + D/2) at a time it reads
// the KS partials from the cluster's shared memories (16-byte loads), sums
// them in rank order, turns key pairs by the angle pos * theta^(-2d/D)
// (reduced modulo 2 pi exactly in 64-bit fixed point, sine and cosine of the
// reduced angle in fp32: no double arithmetic, whose rate on GB300 is a small
// fraction of fp32's), rounds to bf16 and writes the slot.  A second cluster
// barrier keeps every partial alive until its readers are done.  A negative
// position writes nothing and sets the device error word.
//
// Each CTA writes its own error word (a grid of more than kMaxCtas CTAs
// shares one, cleared by a one-thread kernel launched first).
//
// The weights are read once (the only large operand: n_dl * F * d_model * 2
// bytes); the activations (n_act * B * d_model * 2 bytes) are re-read from L2
// by every row tile group.  The rotary frequencies are per-call constants
// computed on the host.
#include <climits>
#include <cmath>
#include <atomic>
#include <cstdint>

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "spire.h"
#include "spire_common.cuh"
#include "spire_host.h"

namespace spire {
namespace {

constexpr int kAppendThreads = 384;       // W producer, MMA, x producer, (idle), 8 epilogue warps
constexpr int kAppendMaxStages = 8;
constexpr int kAppendMaxCluster = 8;      // K splits = CTAs of one cluster (portable size)
constexpr int kAppendMaxN = 128;          // tokens per CTA
constexpr int kAppendMaxMT = 2;           // row tiles per CTA
constexpr int kWTile = 128 * 64 * 2;      // one W tile: 128 rows x 64 columns bf16
constexpr int kAppendStatic = 2560;       // bound on the kernel's static shared memory

struct AppendParams {
    const float* mix_w;       // [n_dl, n_act]
    const int32_t* pos;       // [B]
    __nv_bfloat16* kv;        // [n_dl, B, 2, Hkv, S, D]
    int32_t* header;          // header[0] = number of error words
    int32_t* err;             // error words: one per CTA, or err[0] shared (err_shared)
    int B, n_act, n_dl, F, Hkv, D, S, n_sink, window;
    int N, ntb, mgroups, TS, ks, kblocks, nx, tcols, rotate;
    int err_shared;
    uint64_t fturn[64];       // theta^(-2d/D) / (2 pi) as 64-bit fractions, d < D/2
};

// The two stage rings: W stages of MT tiles (128 rows x 128 bytes each), then
// activation stages of n_act tiles of N rows (one 3-D box); 128-byte
// swizzle, every stage 1024-byte aligned.

// Only for grids of more than kMaxCtas CTAs, which share one error word.
__global__ void __launch_bounds__(32) append_clear_kernel(int32_t* header, int32_t* err) {
    grid_dep_launch_dependents();                // the projection may start its prologue
    if (threadIdx.x == 0) {
        header[0] = 1;
        err[0] = 0;
    }
}

static_assert(8 * (4 * kAppendMaxStages + 2) + 8 + 16 * 4 + kAppendMaxN * (4 + 4) + 64 * 8 + 64 <=
                  kAppendStatic,
              "static shared memory of append_kernel");

// MT (row tiles per CTA) is a compile-time constant: a run-time bound on the
// MMA loop costs each tcgen05.mma about 250 issue cycles instead of ~45.
template <int MT>
__global__ void __launch_bounds__(kAppendThreads, 1)
    append_kernel(const __grid_constant__ CUtensorMap tmap_w,
                  const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ AppendParams p) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t bars[4 * kAppendMaxStages + 2];
    __shared__ uint32_t tmem_slot;
    __shared__ uint32_t cta_err;
    __shared__ float amix[16];
    __shared__ int32_t spos[kAppendMaxN];      // positions of the tokens this CTA stores
    __shared__ int32_t sslot[kAppendMaxN];     // their slots (INT_MIN: past the batch, -1: bad)
    __shared__ uint64_t sturn[64];             // the rotary turn constants (lanes index them)

    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    const int N = p.N, NA = p.n_act * p.N, TS = p.TS;
    const int WST = MT * kWTile, XST = NA * 128;           // stage bytes of the two rings
    const int nx = p.nx;
    // the W ring takes what the launch's shared memory leaves after the
    // 1024-byte alignment of the base and the activation ring
    int nw = ((int)dynamic_smem_bytes() - (int)(base - raw) - nx * XST) / WST;
    if (nw > kAppendMaxStages) nw = kAppendMaxStages;
    if (nw < 2) {                                // the host plans for at least two
        if (threadIdx.x == 0) {
            p.err[p.err_shared ? 0 : blockIdx.x] = (int32_t)kErrTimeout;
            if (blockIdx.x == 0 && !p.err_shared) p.header[0] = (int32_t)gridDim.x;
        }
        return;
    }
    const uint32_t xbase = base + (uint32_t)(nw * WST);
    // this CTA's partial, fp32 [tile][token][row], lies over its drained rings
    const uint32_t bar0 = smem_u32(bars);
    const uint32_t bar_wfull = bar0, bar_wempty = bar0 + 8 * kAppendMaxStages;
    const uint32_t bar_xfull = bar0 + 16 * kAppendMaxStages, bar_xempty = bar0 + 24 * kAppendMaxStages;
    const uint32_t bar_acc = bar0 + 32 * kAppendMaxStages, bar_drain = bar_acc + 8;

    // this CTA: layer li, row tiles [MT mg, +MT), tokens [N nt, +N), K blocks [kb0, kb1)
    const uint32_t rank = cluster_ctarank();
    int t = blockIdx.x / p.ks;
    const int nt = t % p.ntb; t /= p.ntb;
    const int mg = t % p.mgroups;
    const int li = t / p.mgroups;
    const int kb0 = (int)rank * p.kblocks / p.ks;
    const int kb1 = ((int)rank + 1) * p.kblocks / p.ks;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < nw; ++s) {
            mbar_init(bar_wfull + 8 * s, 1);
            mbar_init(bar_wempty + 8 * s, 1);
        }
        for (int s = 0; s < nx; ++s) {
            mbar_init(bar_xfull + 8 * s, 1);
            mbar_init(bar_xempty + 8 * s, 1);
        }
        mbar_init(bar_acc, 1);
        mbar_init(bar_drain, 1);
        fence_barrier_init();
        cta_err = 0;
    }
    if (threadIdx.x >= 96 && threadIdx.x < 96 + 64) sturn[threadIdx.x - 96] = p.fturn[threadIdx.x - 96];
    if (warp == 1) {
        tmem_alloc(smem_u32(&tmem_slot), (uint32_t)p.tcols);
        tmem_relinquish();
        tc_fence_before();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    uint32_t err = 0;
    grid_dep_launch_dependents();
    // inputs are read only after the kernel before this one has completed
    grid_dep_wait();

    if ((warp == 0 || warp == 2) && lane == 0) {
        // ------------------------------------------------ producers: W (warp 0), x (warp 2)
        // Two rings: the W tiles come from HBM (long latency, a deep ring),
        // the activation tiles mostly from L2 (a shallower one).
        const bool is_w = warp == 0;
        const CUtensorMap* const map = is_w ? &tmap_w : &tmap_x;
        prefetch_tensormap(map);
        const uint64_t pol = is_w ? policy_evict_first() : policy_evict_last();
        const int ns = is_w ? nw : nx, stb = is_w ? WST : XST;
        const uint32_t ring = is_w ? base : xbase;
        const uint32_t full = is_w ? bar_wfull : bar_xfull, empty = is_w ? bar_wempty : bar_xempty;
        const int wrow = li * p.F + mg * MT * 128;
        uint32_t armed = 0, armed_par = 0;
        int s = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
            if (!mbar_wait(empty + 8 * s, ph ^ 1)) { ok = false; break; }
            const uint32_t dst = ring + s * stb, bar = full + 8 * s;
            mbar_arrive_expect_tx(bar, (uint32_t)stb);
            if (is_w) {
                for (int tt = 0; tt < MT; ++tt)
                    tma_load_2d(dst + tt * kWTile, map, kb * 64, wrow + tt * 128, bar, pol);
            } else {
                tma_load_3d(dst, map, kb * 64, nt * N, 0, bar, pol);
            }
            armed |= 1u << s;
            armed_par = (armed_par & ~(1u << s)) | (ph << s);
            if (++s == ns) { s = 0; ph ^= 1; }
        }
        if (!ok) {
            err |= kErrTimeout;
            for (int q = 0; q < ns; ++q)   // our copies land before shared memory is reused
                if (armed & (1u << q)) mbar_wait(full + 8 * q, (armed_par >> q) & 1u);
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, NA, false);
            int sw = 0, sx = 0;
            uint32_t pw = 0, px = 0;
            bool ok = true;
            for (int kb = kb0; kb < kb1; ++kb) {
                if (!mbar_wait(bar_wfull + 8 * sw, pw) || !mbar_wait(bar_xfull + 8 * sx, px)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t aw = base + sw * WST, bx = xbase + sx * XST;
#pragma unroll
                for (int k16 = 0; k16 < 4; ++k16) {
                    const uint64_t bdesc = sdesc_sw128(bx + 32 * k16, 16, 1024);
#pragma unroll
                    for (int tt = 0; tt < MT; ++tt)
                        umma_bf16(tmem + (uint32_t)(tt * TS),
                                  sdesc_sw128(aw + tt * kWTile + 32 * k16, 16, 1024), bdesc, idesc,
                                  (kb > kb0 || k16 > 0) ? 1u : 0u);
                }
                umma_commit(bar_wempty + 8 * sw);
                umma_commit(bar_xempty + 8 * sx);
                if (++sw == nw) { sw = 0; pw ^= 1; }
                if (++sx == nx) { sx = 0; px ^= 1; }
            }
            if (ok) umma_commit(bar_acc);
            else err |= kErrTimeout;
            umma_commit(bar_drain);   // every MMA has finished before TMEM is freed
            if (!mbar_wait(bar_drain, 0)) err |= kErrTimeout;
        }
        __syncwarp();
    } else if (warp >= 4) {
        // ------------------------------------------------ epilogue set-up
        if (warp == 4 && lane == 0) {            // a_i = softmax(w_i), as the definition
            const float* w = p.mix_w + li * p.n_act;
            float wmax = -INFINITY;
            for (int l = 0; l < p.n_act; ++l) wmax = fmaxf(wmax, w[l]);
            float z = 0.f;
            for (int l = 0; l < p.n_act; ++l) {
                const float e = expf(w[l] - wmax);
                amix[l] = e;
                z += e;
            }
            for (int l = 0; l < p.n_act; ++l) amix[l] /= z;
        }
        // position and slot of the tokens this CTA stores: CTA q of the
        // cluster stores tokens [q N / KS, (q + 1) N / KS) of the block
        const int j0 = rank * N / p.ks;
        const int nj = (rank + 1) * N / p.ks - j0;
        const int e = (int)threadIdx.x - 128;
        if (e < nj) {
            const int b = nt * N + j0 + e;
            const int pos = b < p.B ? p.pos[b] : INT_MIN;
            spos[e] = pos;
            sslot[e] = pos == INT_MIN ? INT_MIN   // no sequence: nothing to store
                                      : (int)spire_draft_slot_inline(pos, p.n_sink, p.window);
        }
        named_bar_sync(1, 256);                  // amix is written
        if (!mbar_wait(bar_acc, 0)) err |= kErrTimeout;
        tc_fence_before();
    }
    if (warp >= 4) {
        // ------------------------------------------------ epilogue: TMEM lane = W row
        // two warps per TMEM lane quarter, alternate 16-token chunks
        if (!(err & kErrTimeout)) {
            tc_fence_after();
            const int quarter = warp & 3, half = (warp - 4) >> 2;
            const int row = 32 * quarter + lane;
            const uint32_t taddr = tmem + ((uint32_t)(32 * quarter) << 16);
            float* const part = reinterpret_cast<float*>(smem_raw + (base - raw)) + row;
#pragma unroll
            for (int tt = 0; tt < MT; ++tt)
                for (int c0 = 16 * half; c0 < N; c0 += 32) {
                    float y[16];
                    for (int l0 = 0; l0 < p.n_act; l0 += 4) {
                        const int nl = p.n_act - l0 < 4 ? p.n_act - l0 : 4;
                        float v[4][16];
                        const uint32_t ta = taddr + (uint32_t)(tt * TS + l0 * N + c0);
                        tmem_ld16(ta, v[0]);
                        if (nl > 1) tmem_ld16(ta + N, v[1]);
                        if (nl > 2) tmem_ld16(ta + 2 * N, v[2]);
                        if (nl > 3) tmem_ld16(ta + 3 * N, v[3]);
                        tmem_wait_ld();
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            if (u >= nl) break;
                            const float al = amix[l0 + u];
                            if (l0 + u == 0) {
#pragma unroll
                                for (int j = 0; j < 16; ++j) y[j] = al * v[u][j];
                            } else {
#pragma unroll
                                for (int j = 0; j < 16; ++j) y[j] = fmaf(al, v[u][j], y[j]);
                            }
                        }
                    }
#pragma unroll
                    for (int j = 0; j < 16; ++j) part[(tt * N + c0 + j) * 128] = y[j];
                }
        }
        tc_fence_before();
    }
    // every CTA's partial is complete and visible cluster-wide after this
    cluster_sync_all();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, (uint32_t)p.tcols);
    }

    // ---------------------------------------------------- split sum, rotation, store
    {
        const int j0 = rank * N / p.ks;
        const int nj = (rank + 1) * N / p.ks - j0;
        const int half = p.D / 2, HD = p.Hkv * p.D;
        const bool d128 = p.D == 128;
        // four adjacent pairs (d .. d + 3, + D/2) of one token per item; the
        // KS partials of each are read from the cluster's shared memories
        const int items = MT * nj * 16;
        for (int it = threadIdx.x; it < items; it += kAppendThreads) {
            const int g4 = it & 15;
            const int jl = (it >> 4) % nj;
            const int tt = (it >> 4) / nj;
            const int slot = sslot[jl];
            if (slot == INT_MIN) continue;
            if (slot < 0) {
                if (g4 == 0 && tt == 0) err |= kErrCtxLen;
                continue;
            }
            const int pos = spos[jl];
            const int b = nt * N + j0 + jl;
            const int p0 = 4 * g4, hl = d128 ? 0 : p0 >> 5, d = d128 ? p0 : p0 & 31;
            const int r0 = hl * p.D + d;             // rows r0 .. r0 + 3 and + D/2
            const uint32_t a0 = base + (uint32_t)(((tt * N + j0 + jl) * 128 + r0) * 4);
            float4 v0[kAppendMaxCluster], v1[kAppendMaxCluster];
#pragma unroll
            for (int q = 0; q < kAppendMaxCluster; ++q)
                if (q < p.ks) {
                    v0[q] = ld_dsmem_f4(mapa_shared(a0, (uint32_t)q));
                    v1[q] = ld_dsmem_f4(mapa_shared(a0 + (uint32_t)(half * 4), (uint32_t)q));
                }
            float lo[4] = {v0[0].x, v0[0].y, v0[0].z, v0[0].w};
            float hi[4] = {v1[0].x, v1[0].y, v1[0].z, v1[0].w};
#pragma unroll
            for (int q = 1; q < kAppendMaxCluster; ++q)      // the splits in rank order
                if (q < p.ks) {
                    lo[0] += v0[q].x; lo[1] += v0[q].y; lo[2] += v0[q].z; lo[3] += v0[q].w;
                    hi[0] += v1[q].x; hi[1] += v1[q].y; hi[2] += v1[q].z; hi[3] += v1[q].w;
                }
            const int f = (mg * MT + tt) * 128 + r0;   // row of W_i: kvi, head g, column d
            const int kvi = f / HD, g = (f - kvi * HD) >> (d128 ? 7 : 6);
            if (kvi == 0 && p.rotate) {
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    float sn, cs;
                    rope_sincos(pos, sturn[d + e], &sn, &cs);
                    const float u = lo[e] * cs - hi[e] * sn;
                    const float w = hi[e] * cs + lo[e] * sn;
                    lo[e] = u;
                    hi[e] = w;
                }
            }
            __nv_bfloat16* const dst =
                p.kv + ((((long long)li * p.B + b) * 2 + kvi) * p.Hkv + g) * (long long)p.S * p.D +
                (long long)slot * p.D + d;
            *reinterpret_cast<uint2*>(dst) = make_uint2(pack_bf16(lo[0], lo[1]), pack_bf16(lo[2], lo[3]));
            *reinterpret_cast<uint2*>(dst + half) =
                make_uint2(pack_bf16(hi[0], hi[1]), pack_bf16(hi[2], hi[3]));
        }
    }
    if (err) atomicOr(&cta_err, err);
    __syncthreads();
    if (threadIdx.x == 0) {
        if (p.err_shared) {
            if (cta_err) atomicOr(p.err, (int)cta_err);
        } else {
            // every CTA writes its word, so nothing needs clearing first
            p.err[blockIdx.x] = (int32_t)cta_err;
            if (blockIdx.x == 0) p.header[0] = (int32_t)gridDim.x;
        }
    }
    // no CTA leaves while another may still read its partial
    cluster_sync_all();
}

struct AppendPlan {
    int F, N, ntb, mtiles, kblocks;
};

bool plan_append(const spire_append_desc* d, AppendPlan* pl) {
    if (!d) return false;
    if (d->batch < 0 || d->num_act < 1 || d->num_act > 16 || d->num_draft_layers < 1 ||
        d->num_draft_layers > 16 || d->d_model < 64 || d->d_model > 65536 ||
        d->d_model % 64 != 0 || d->num_kv_heads < 1 || (d->head_dim != 64 && d->head_dim != 128) ||
        d->n_sink < 0 || d->window < 1 || !std::isfinite(d->rope_theta) || d->rope_theta < 0.f)
        return false;
    const long long F = 2LL * d->num_kv_heads * d->head_dim;
    if (F * d->num_draft_layers > (1LL << 30) ||
        (long long)d->n_sink + d->window > (1LL << 30) ||
        (long long)d->num_act * d->batch > (1LL << 30) ||
        (long long)d->num_draft_layers * d->batch > (1LL << 30))
        return false;
    pl->F = (int)F;
    pl->mtiles = (int)(F / 128);
    pl->kblocks = d->d_model / 64;
    if (d->batch == 0) {           // nothing to do; the shape is still checked
        pl->N = 16;
        pl->ntb = 0;
        return true;
    }
    // one MMA covers the n_act activation tiles: n_act x N <= 256
    int nmax = (256 / d->num_act) / 16 * 16;
    if (nmax > kAppendMaxN) nmax = kAppendMaxN;
    const int nb = d->batch < nmax ? d->batch : nmax;
    pl->N = (nb + 15) / 16 * 16;
    pl->ntb = (d->batch + pl->N - 1) / pl->N;
    return true;
}

// workspace: header word (number of error words) | error words (one per CTA)
constexpr size_t kAppendHeader = 256;
constexpr size_t kAppendWorkspace = kAppendHeader + 4 * kMaxCtas;

}  // namespace
}  // namespace spire

using namespace spire;

extern "C" {

size_t spire_feedback_append_workspace_bytes(const spire_append_desc* desc) {
    AppendPlan pl;
    if (!plan_append(desc, &pl)) return 0;
    return kAppendWorkspace;
}

spire_status spire_feedback_append(const void* x, const float* mix_w, const void* w_kv,
                                   const int32_t* pos, const spire_append_desc* desc, void* kv,
                                   void* workspace, size_t ws_bytes, void* stream) {
    AppendPlan pl;
    if (!plan_append(desc, &pl)) {
        if (desc && desc->head_dim != 64 && desc->head_dim != 128 && desc->batch >= 0)
            return SPIRE_ERR_UNSUPPORTED;
        return SPIRE_ERR_INVALID_ARG;
    }
    if (desc->batch == 0) return SPIRE_OK;
    if (!x || !mix_w || !w_kv || !pos || !kv || !workspace) return SPIRE_ERR_INVALID_ARG;
    if (!host_aligned(x, 16) || !host_aligned(w_kv, 16) || !host_aligned(kv, 16) ||
        !host_aligned(mix_w, 4) || !host_aligned(pos, 4) || !host_aligned(workspace, 256))
        return SPIRE_ERR_INVALID_ARG;
    if (ws_bytes < kAppendWorkspace) return SPIRE_ERR_WORKSPACE;
    int sms = 0, smem_optin = 0;
    if (host_device_info(&sms, &smem_optin) != SPIRE_OK) return SPIRE_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);

    const int B = desc->batch, n_dl = desc->num_draft_layers, n_act = desc->num_act;
    const int NA = n_act * pl.N, TS = (NA + 31) / 32 * 32;
    // One MMA's N is NA, and an activation stage holds exactly NA rows: both
    // come from this plan, within what a kind::f16 MMA with M = 128 accepts.
    if (NA < 16 || NA > 256 || NA % 16 != 0) return SPIRE_ERR_UNSUPPORTED;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SPIRE_ERR_CUDA;
    const long long tiles1 = (long long)n_dl * pl.mtiles * pl.ntb;
    // two row tiles per CTA share each activation tile, but halve the CTAs:
    // only when one-tile CTAs would fill the GPU twice over
    const int MT = (pl.mtiles % 2 == 0 && kAppendMaxMT * TS <= 512 && tiles1 >= 2LL * sms)
                       ? kAppendMaxMT : 1;
    const long long tiles = tiles1 / MT;
    void (*const kern)(CUtensorMap, CUtensorMap, AppendParams) =
        MT == 2 ? append_kernel<2> : append_kernel<1>;
    // K splits: as many as fill the SMs (at most 8, the portable cluster
    // size), fewer while the GPU cannot hold all clusters at once
    long long ks = sms / tiles;
    if (ks < 1) ks = 1;
    if (ks > kAppendMaxCluster) ks = kAppendMaxCluster;
    if (ks > pl.kblocks) ks = pl.kblocks;
    const int WST = MT * kWTile, XST = NA * 128;
    // the kernel's static shared memory (the dynamic part gets the rest)
    static std::atomic<int> static_bytes[2];
    int static_smem = static_bytes[MT - 1].load(std::memory_order_acquire);
    if (static_smem == 0) {
        cudaFuncAttributes fa;
        if (cudaFuncGetAttributes(&fa, kern) != cudaSuccess) return SPIRE_ERR_CUDA;
        static_smem = (int)fa.sharedSizeBytes;
        if (static_smem <= 0 || static_smem > kAppendStatic) return SPIRE_ERR_UNSUPPORTED;
        static_bytes[MT - 1].store(static_smem, std::memory_order_release);
    }
    int nw = 0, nx = 0;
    size_t smem = 0;
    // a cluster's CTAs each take one SM (the shared memory is more than half
    // of one, so a second CTA, which could wait for tensor memory held by a
    // CTA waiting on its own cluster, never shares it)
    static std::atomic<int> max_clusters[2][64][kAppendMaxCluster + 1];
    for (;; ks--) {
        const long long part = (long long)MT * pl.N * 512;   // the partial, over the ring
        // dynamic shared memory: all the opt-in size leaves beside the static
        // part; the kernel sizes its W ring from it (the host plans with the
        // worst-case 1023-byte alignment slack, the kernel uses the real one)
        const int dyn = smem_optin - static_smem;
        const int avail = dyn - 1024;
        // the activation tiles mostly hit L2 (short latency): about 45 % of
        // the budget; the W tiles stream from HBM: the rest, a deeper ring
        nx = (int)((long long)avail * 9 / 20 / XST);
        if (nx < 2) nx = 2;
        if (nx > kAppendMaxStages) nx = kAppendMaxStages;
        nw = (avail - nx * XST) / WST;
        if (nw > kAppendMaxStages) nw = kAppendMaxStages;
        const long long ring = (long long)nw * WST + (long long)nx * XST;
        if (nw < 2 || part > ring) {
            if (ks == 1) return SPIRE_ERR_UNSUPPORTED;
            continue;
        }
        smem = (size_t)dyn;
        if (ks == 1) break;
        int mc = (dev >= 0 && dev < 64) ? max_clusters[MT - 1][dev][ks].load(std::memory_order_acquire)
                                        : 0;
        if (mc == 0) {
            if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     smem_optin - static_smem) != cudaSuccess)
                return SPIRE_ERR_CUDA;
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3((unsigned)ks);
            cfg.blockDim = dim3(kAppendThreads);
            cfg.dynamicSmemBytes = smem;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeClusterDimension;
            attr[0].val.clusterDim.x = (unsigned)ks;
            attr[0].val.clusterDim.y = 1;
            attr[0].val.clusterDim.z = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            int n = 0;
            if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
                cudaGetLastError();
                n = 0;
            }
            mc = n > 0 ? n : -1;
            if (dev >= 0 && dev < 64)
                max_clusters[MT - 1][dev][ks].store(mc, std::memory_order_release);
        }
        if (mc >= tiles) break;
    }
    if (tiles * ks > INT_MAX) return SPIRE_ERR_UNSUPPORTED;
    uint32_t tcols = 32;
    while ((int)tcols < MT * TS) tcols <<= 1;

    CUtensorMap tw, tx;
    if (!encode_2d_bf16_map(&tw, w_kv, desc->d_model, (uint64_t)n_dl * pl.F, 64, 128) ||
        !encode_3d_bf16_map(&tx, x, desc->d_model, (uint64_t)B, (uint64_t)n_act, 64, pl.N,
                            n_act))
        return SPIRE_ERR_CUDA;

    char* ws = static_cast<char*>(workspace);
    int32_t* const header = reinterpret_cast<int32_t*>(ws);
    int32_t* const errw = reinterpret_cast<int32_t*>(ws + kAppendHeader);
    // up to kMaxCtas CTAs write one error word each; a larger grid shares a
    // word that a one-thread kernel clears first
    const bool err_shared = tiles * ks > kMaxCtas;
    if (err_shared) {
        append_clear_kernel<<<1, 32, 0, st>>>(header, errw);
        if (cudaGetLastError() != cudaSuccess) return SPIRE_ERR_CUDA;
    }

    AppendParams ap{};
    ap.mix_w = mix_w;
    ap.pos = pos;
    ap.kv = static_cast<__nv_bfloat16*>(kv);
    ap.header = header;
    ap.err = errw;
    ap.err_shared = err_shared ? 1 : 0;
    ap.B = B;
    ap.n_act = n_act;
    ap.n_dl = n_dl;
    ap.F = pl.F;
    ap.Hkv = desc->num_kv_heads;
    ap.D = desc->head_dim;
    ap.S = desc->n_sink + desc->window;
    ap.n_sink = desc->n_sink;
    ap.window = desc->window;
    ap.N = pl.N;
    ap.ntb = pl.ntb;
    ap.mgroups = pl.mtiles / MT;
    ap.TS = TS;
    ap.ks = (int)ks;
    ap.kblocks = pl.kblocks;
    ap.nx = nx;
    ap.tcols = (int)tcols;
    ap.rotate = desc->rope_theta > 0.f;
    for (int d = 0; d < desc->head_dim / 2; ++d)     // the same libm pow as the definition
        ap.fturn[d] = desc->rope_theta > 0.f
                          ? rope_turn_fixed(std::pow((double)desc->rope_theta,
                                                     -2.0 * d / desc->head_dim))
                          : 0;
    // the kernel's dynamic shared memory limit, set once per device
    static std::atomic<int> smem_set[2][64];
    if (dev < 0 || dev >= 64 || !smem_set[MT - 1][dev].load(std::memory_order_acquire)) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
            cudaSuccess)
            return SPIRE_ERR_CUDA;
        if (dev >= 0 && dev < 64) smem_set[MT - 1][dev].store(1, std::memory_order_release);
    }
    return launch_dependent_cluster(kern, dim3((unsigned)(tiles * ks)),
                                    dim3(kAppendThreads), smem, st, (unsigned)ks, tw, tx, ap) ==
                   cudaSuccess
               ? SPIRE_OK
               : SPIRE_ERR_CUDA;
}

}  // extern "C"
