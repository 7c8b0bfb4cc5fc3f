// spire_abi.cu -- the C ABI of libspire (declared in include/spire.h): host
// validation, workspace layout, TMA descriptors and the launch on the
// caller's stream (a small kernel zeroing the pair counters, then one
// attention kernel that overlaps it through programmatic dependent launch).
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "spire.h"
#include "spire_host.h"
#include "spire_launch.h"

namespace spire {
namespace {

constexpr size_t kHeaderBytes = 256;
constexpr int kHeadTc = 4;    // per-pair fixed cost of the tcgen05 attention kernel, in tiles
constexpr int kHeadMma = 1;   // the same for the warp-MMA attention kernel
constexpr double kLog2e = 1.4426950408889634;  // log2(e): softmax runs in base 2

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct WsLayout {
    size_t err, stamps, cnt, part_lse, part_o, total;
};

// Offset of the per-CTA timing record: fixed, so that spire_get_cta_times
// needs only the workspace pointer.
constexpr size_t kStampsOffset = kHeaderBytes + ((size_t(kMaxCtas) * 4 + 255) & ~size_t(255));
static_assert(kStampsOffset % 256 == 0, "the timing record starts a 256-byte block");

// header (grid size of the last call) | per-CTA error words | per-CTA timing
// record | per-pair arrival counters | partial slots (two per CTA: a CTA
// range cuts at most its first and its last pair).
WsLayout ws_layout(long long B, long long Hkv, long long R, long long D) {
    const long long slots = 2LL * kMaxCtas;
    WsLayout w{};
    size_t off = kHeaderBytes;
    w.err = off;      off += align256(size_t(kMaxCtas) * 4);
    w.stamps = off;   off += align256(size_t(kMaxCtas) * 16);
    w.cnt = off;      off += align256(size_t(B * Hkv) * 4);
    w.part_lse = off; off += align256(size_t(slots * R) * 4);
    w.part_o = off;   off += align256(size_t(slots * R * D) * 4);
    w.total = off;
    return w;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

spire_status check_common(const spire_attn_desc* d) {
    if (!d) return SPIRE_ERR_INVALID_ARG;
    if (d->batch < 0 || d->num_q_heads < 1 || d->num_kv_heads < 1) return SPIRE_ERR_INVALID_ARG;
    if (d->num_q_heads % d->num_kv_heads != 0) return SPIRE_ERR_INVALID_ARG;
    if (!std::isfinite(d->softmax_scale) || !(d->softmax_scale > 0.f)) return SPIRE_ERR_INVALID_ARG;
    if (d->head_dim != 64 && d->head_dim != 128) return SPIRE_ERR_UNSUPPORTED;
    return SPIRE_OK;
}

int rows_per_kv_head(const spire_attn_desc* d, int kp1) {
    return (d->num_q_heads / d->num_kv_heads) * kp1;
}

// --------------------------------------------------------------- driver API
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// 3-D bf16 view {D, rows, planes} read in 64 x 64 boxes with 128-byte swizzle.
bool encode_kv_map(CUtensorMap* map, const void* base, uint64_t D, uint64_t rows,
                   uint64_t planes) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {D, rows, planes};
    cuuint64_t strides[2] = {D * 2, D * 2 * rows};
    cuuint32_t box[3] = {64, 64, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Query rows of pair (b, g): q viewed as {D, Hq, B * kp1}; one box is the
// G heads of the group for all kp1 block rows, landing as rows r = i*G + hl.
bool encode_q_map(CUtensorMap* map, const void* q, uint64_t D, uint64_t Hq, uint64_t planes,
                  uint32_t G, uint32_t kp1) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {D, Hq, planes};
    cuuint64_t strides[2] = {D * 2, D * 2 * Hq};
    cuuint32_t box[3] = {64, G, kp1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

struct DeviceInfo {
    int sms = 0;
    int smem_optin = 0;
};

spire_status device_info(DeviceInfo* out) {
    static std::mutex mu;
    static DeviceInfo cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SPIRE_ERR_CUDA;
    if (dev >= 0 && dev < 64) {
        std::lock_guard<std::mutex> g(mu);
        if (cache[dev].sms == 0) {
            if (cudaDeviceGetAttribute(&cache[dev].sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&cache[dev].smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin,
                                       dev) != cudaSuccess) {
                cache[dev].sms = 0;
                return SPIRE_ERR_CUDA;
            }
        }
        *out = cache[dev];
        return SPIRE_OK;
    }
    if (cudaDeviceGetAttribute(&out->sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&out->smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess)
        return SPIRE_ERR_CUDA;
    return SPIRE_OK;
}

}  // namespace

bool host_aligned(const void* p, uintptr_t a) { return aligned(p, a); }

spire_status host_device_info(int* sms, int* smem_optin) {
    DeviceInfo di;
    const spire_status st = device_info(&di);
    if (st != SPIRE_OK) return st;
    *sms = di.sms;
    *smem_optin = di.smem_optin;
    return SPIRE_OK;
}

bool encode_2d_bf16_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                        uint32_t box_inner, uint32_t box_outer) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {inner * 2};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

uint64_t rope_turn_fixed(double freq) {
    // 1 / (2 pi) = kInv2PiHi + kInv2PiLo to about 2^-107; freq / (2 pi) =
    // ph + pe with ph = fl(freq * hi) and pe its error plus freq * lo
    const double kInv2PiHi = 0.15915494309189535;
    const double kInv2PiLo = -9.839338337591243e-18;
    if (!(freq > 0.0)) return 0;
    const double ph = freq * kInv2PiHi;
    const double pe = std::fma(freq, kInv2PiHi, -ph) + freq * kInv2PiLo;
    const double two64 = 18446744073709551616.0;
    // ph * 2^64 < 2^62 truncates to an integer with an error below one unit
    // (none once it exceeds 2^53); pe * 2^64 adds the rest, rounded
    const double hi = std::floor(ph * two64);
    return (uint64_t)hi + (uint64_t)(int64_t)std::llround(ph * two64 - hi + pe * two64);
}

bool encode_3d_bf16_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t mid,
                        uint64_t outer, uint32_t box_inner, uint32_t box_mid, uint32_t box_outer) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {inner, mid, outer};
    cuuint64_t strides[2] = {inner * 2, inner * 2 * mid};
    cuuint32_t box[3] = {box_inner, box_mid, box_outer};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

namespace {

// Zeroes the per-pair arrival counters.  A programmatic dependent of the
// kernel before it (one CTA, it fits beside a running attention CTA): it lets
// the attention kernel after it launch at once and zeroes the counters only
// when the kernel before has completed, so back-to-back calls hide both
// launches behind the previous call's tail.
__global__ void __launch_bounds__(256) zero_counters_kernel(int32_t* cnt, int n) {
    grid_dep_launch_dependents();
    grid_dep_wait();
    for (int i = threadIdx.x; i < n; i += blockDim.x) cnt[i] = 0;
}

// ------------------------------------------------------------- stream floor
// Reads `bytes` of device memory once and computes nothing: one CTA per SM
// takes a contiguous run of 16 KB chunks and streams it through a four-stage
// ring of 32 KB in shared memory with bulk async copies (L2 evict-first, as
// the attention kernels' tiles); a consumer thread only waits for each stage
// and frees it.  Its time is the floor of any single launch that must read
// that many bytes.  Waits are bounded; a wait that gives up ends the CTA
// (with its copies landed) and the measurement is void.
constexpr uint32_t kFloorChunk = 16384;
constexpr int kFloorStages = 4;
constexpr int kFloorSmem = kFloorStages * 2 * kFloorChunk + 2 * kFloorStages * 8 + 128;

__global__ void __launch_bounds__(64, 1) stream_read_kernel(const uint8_t* src,
                                                            unsigned long long bytes) {
    extern __shared__ __align__(128) uint8_t fsm[];
    const uint32_t base = (smem_u32(fsm) + 127u) & ~127u;
    const uint32_t full = base + kFloorStages * 2 * kFloorChunk, empty = full + 8 * kFloorStages;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kFloorStages; ++s) {
            mbar_init(full + 8 * s, 1);
            mbar_init(empty + 8 * s, 1);
        }
        fence_barrier_init();
    }
    __syncthreads();
    const unsigned long long chunks = (bytes + kFloorChunk - 1) / kFloorChunk;
    const unsigned long long lo = chunks * blockIdx.x / gridDim.x,
                             hi = chunks * (blockIdx.x + 1) / gridDim.x;
    // two chunks per stage: stage i of this CTA holds chunks lo + 2i, lo + 2i + 1
    const unsigned long long n_st = (hi - lo + 1) / 2;
    if (threadIdx.x == 0) {
        const uint64_t pol = policy_evict_first();
        uint32_t s = 0, ph = 0, armed = 0, armed_par = 0;
        for (unsigned long long i = 0; i < n_st; ++i) {
            if (!mbar_wait(empty + 8 * s, ph ^ 1)) {
                for (int q = 0; q < kFloorStages; ++q)   // our copies land first
                    if (armed & (1u << q)) mbar_wait(full + 8 * q, (armed_par >> q) & 1u);
                return;
            }
            uint32_t nb = 0;
            const unsigned long long c0 = lo + 2 * i;
            uint32_t len[2] = {0u, 0u};
            for (int h = 0; h < 2; ++h) {
                const unsigned long long c = c0 + h;
                if (c < hi) {
                    const unsigned long long off = c * kFloorChunk;
                    len[h] = (uint32_t)(bytes - off < kFloorChunk ? bytes - off : kFloorChunk);
                    nb += len[h];
                }
            }
            mbar_arrive_expect_tx(full + 8 * s, nb);
            for (int h = 0; h < 2; ++h)
                if (len[h])
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes"
                        ".L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(base + (s * 2 + h) * kFloorChunk),
                        "l"(src + (c0 + h) * kFloorChunk), "r"(len[h]), "r"(full + 8 * s), "l"(pol)
                        : "memory");
            armed |= 1u << s;
            armed_par = (armed_par & ~(1u << s)) | (ph << s);
            if (++s == kFloorStages) { s = 0; ph ^= 1; }
        }
    } else if (threadIdx.x == 32) {
        uint32_t s = 0, ph = 0;
        for (unsigned long long i = 0; i < n_st; ++i) {
            if (!mbar_wait(full + 8 * s, ph)) return;
            mbar_arrive(empty + 8 * s);
            if (++s == kFloorStages) { s = 0; ph ^= 1; }
        }
    }
}

// ------------------------------------------------------------- MagicDec gather
// MagicDec's draft attends, with positions inside the reduced cache, to the
// sink + window entries of the target's own paged cache (Section 3.1
// footnote).  This kernel builds that reduced cache, one warp per item; a
// row of D bf16 sits in D/8 lanes, 16 bytes each, 32/(D/8) rows per step:
//   sequence items  n_vis[b] = number of visible entries (0 if t is out of
//                   range or a visible page id is outside the cache)
//   row items       1/8 of the visible entries of (b, g): entry c at text
//                   position p, K turned by (c - p) and rounded to bf16, V
//                   copied; the pages of a batch of rows are looked up first,
//                   then all their K and V loads issue together.  A sink keeps
//                   its position (c = p) and every window entry moves by the
//                   same s - w0, so a lane computes the sines and cosines of
//                   its eight elements once per item; the partner (d + D/2)
//                   of an element comes from the lane D/16 away (shuffle)
//   query items     q rows turned by their cache index n_vis - 1
// Angles: reduced modulo 2 pi exactly in 64-bit fixed point (rope_sincos),
// sine and cosine of the reduced angle in fp32 (positions up to 2^31 keep
// their accuracy).  The kernel also zeroes the attention's pair counters,
// and the attention kernel follows it as its programmatic dependent.
constexpr int kMdParts = 8;           // row items per (sequence, KV head)

struct MdParams {
    const __nv_bfloat16* q;        // [B, Hq, D], not rotated
    const __nv_bfloat16* k_cache;  // [num_pages, Hkv, 64, D], keys turned by text position
    const __nv_bfloat16* v_cache;
    const int32_t* block_table;
    const int32_t* ctx_lens;
    __nv_bfloat16* kv;             // [B, 2, Hkv, S, D] reduced cache
    __nv_bfloat16* q_eff;          // [B, Hq, D]
    int32_t* n_vis;                // [B]
    int32_t* cnt;                  // the attention's pair counters, zeroed here
    float* out;                    // fused path: [B, Hq, D]
    int32_t* header;               // fused path: error words (one per merge CTA)
    int32_t* err;
    int B, Hq, Hkv, D, S, n_sink, window, max_pages, num_pages, rotate;
    int G;                         // query heads per KV head
    float sl2;                     // softmax_scale * log2(e)
    uint64_t fturn[64];            // theta^(-2d/D) / (2 pi) as 64-bit fractions
};

struct MdVisible {
    int s, w0, n;
};

__device__ __forceinline__ MdVisible md_visible(const MdParams& p, int t) {
    MdVisible v{0, 0, 0};
    if (t < 1 || (long long)t > (long long)p.max_pages * kPage) return v;
    v.s = t < p.n_sink ? t : p.n_sink;
    v.w0 = t - p.window > v.s ? t - p.window : v.s;
    v.n = v.s + (t - v.w0);
    return v;
}

// sine and cosine of delta * freq[d] (delta != 0, rotation on); the turn
// constants come from shared memory (lanes index them: from kernel
// parameters the reads would serialise)
__device__ __forceinline__ void md_sincos(const uint64_t* turn, long long delta, int d, float* sn,
                                          float* cs) {
    rope_sincos(delta, turn[d], sn, cs);
}

// A row of D bf16 is spread over D/8 lanes, eight consecutive elements (16
// bytes) per lane; the pair partner (d + D/2) of a first-half lane's elements
// sits in the lane D/16 further on.  Turns this lane's vector v given its
// partner's w by the per-element sines / cosines:
//   first half   v cs - w sn
//   second half  v cs + w sn
// rounding each result to bf16.
__device__ __forceinline__ uint4 md_turn_vec(uint4 v, uint4 w, const float* sn, const float* cs,
                                             bool first_half) {
    const uint32_t a[4] = {v.x, v.y, v.z, v.w}, b[4] = {w.x, w.y, w.z, w.w};
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float a0 = bf16lo_to_f32(a[e]), a1 = bf16hi_to_f32(a[e]);
        const float b0 = bf16lo_to_f32(b[e]), b1 = bf16hi_to_f32(b[e]);
        const float r0 = first_half ? a0 * cs[2 * e] - b0 * sn[2 * e] : a0 * cs[2 * e] + b0 * sn[2 * e];
        const float r1 = first_half ? a1 * cs[2 * e + 1] - b1 * sn[2 * e + 1]
                                    : a1 * cs[2 * e + 1] + b1 * sn[2 * e + 1];
        o[e] = pack_bf16(r0, r1);
    }
    return make_uint4(o[0], o[1], o[2], o[3]);
}

// sines / cosines of delta * freq for this lane's eight elements d0 .. d0 + 7
__device__ __forceinline__ void md_lane_turn(const uint64_t* turn, long long delta, int d0,
                                             float* sn, float* cs) {
#pragma unroll
    for (int e = 0; e < 8; ++e) md_sincos(turn, delta, d0 + e, &sn[e], &cs[e]);
}

constexpr int kMdBatch = 5;    // row steps whose loads a lane issues together

__global__ void __launch_bounds__(256, 2) magicdec_gather_kernel(const MdParams p) {
    __shared__ uint64_t turn[64];
    grid_dep_launch_dependents();      // the attention kernel waits for all of this grid
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < p.B * p.Hkv; i += gridDim.x * blockDim.x)
        p.cnt[i] = 0;
    if (threadIdx.x < 64) turn[threadIdx.x] = p.fturn[threadIdx.x];
    __syncthreads();
    const int lane = threadIdx.x & 31;
    // lanes per row, rows per warp step, and this lane's place
    const int LPR = p.D / 8, RPW = 32 / LPR, HL = LPR / 2;
    const int jl = lane % LPR, sub = lane / LPR;
    const bool first_half = jl < HL;
    const int d0 = 8 * (jl % HL);
    const long long n_rows = (long long)p.B * p.Hkv * kMdParts;
    const long long n_q = ((long long)p.B * p.Hq + RPW - 1) / RPW;
    const long long total = p.B + n_rows + n_q;
    for (long long item = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5; item < total;
         item += ((long long)gridDim.x * blockDim.x) >> 5) {
        if (item < p.B) {
            // sequence item: the visible count, after checking every visible page
            const int b = (int)item;
            const int t = p.ctx_lens[b];
            const MdVisible v = md_visible(p, t);
            bool ok = v.n > 0;
            const int pg_s = v.s > 0 ? (v.s - 1) / kPage + 1 : 0;     // pages of the sinks
            const int pg_w0 = v.w0 / kPage, pg_w1 = ok ? (t - 1) / kPage : -1;
            for (int pg = lane; ok && pg < pg_s; pg += 32) {
                const int id = p.block_table[(long long)b * p.max_pages + pg];
                if (id < 0 || id >= p.num_pages) ok = false;
            }
            for (int pg = pg_w0 + lane; ok && pg <= pg_w1; pg += 32) {
                const int id = p.block_table[(long long)b * p.max_pages + pg];
                if (id < 0 || id >= p.num_pages) ok = false;
            }
            ok = __all_sync(0xffffffffu, ok);
            if (lane == 0) p.n_vis[b] = ok ? v.n : 0;
        } else if (item < p.B + n_rows) {
            // row item: 1/kMdParts of the visible entries of one (sequence, KV head)
            long long r = item - p.B;
            const int part = (int)(r % kMdParts); r /= kMdParts;
            const int g = (int)(r % p.Hkv);
            const int b = (int)(r / p.Hkv);
            const MdVisible v = md_visible(p, p.ctx_lens[b]);
            const int rpp = (v.n + kMdParts - 1) / kMdParts;
            const int c0 = part * rpp, c1 = min(v.n, c0 + rpp);
            if (c0 >= c1) continue;
            // every window entry moves by the same s - w0: one table per lane
            float wsn[8], wcs[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) { wsn[e] = 0.f; wcs[e] = 1.f; }
            if (p.rotate && v.s != v.w0) md_lane_turn(turn, (long long)v.s - v.w0, d0, wsn, wcs);
            for (int cb = c0; cb < c1; cb += RPW * kMdBatch) {
                long long src[kMdBatch];
                int row[kMdBatch];
#pragma unroll
                for (int i = 0; i < kMdBatch; ++i) {      // the entries' pages
                    const int c = cb + i * RPW + sub;
                    row[i] = -1;
                    src[i] = 0;
                    if (c < c1) {
                        const int pos = c < v.s ? c : v.w0 + (c - v.s);
                        const int id = p.block_table[(long long)b * p.max_pages + pos / kPage];
                        if (id >= 0 && id < p.num_pages) {   // else the sequence item reports it
                            row[i] = c;
                            src[i] = (((long long)id * p.Hkv + g) * kPage + pos % kPage) * p.D +
                                     8 * jl;
                        }
                    }
                }
                uint4 kvk[kMdBatch], kvv[kMdBatch];
#pragma unroll
                for (int i = 0; i < kMdBatch; ++i) {      // all rows in flight together
                    if (row[i] >= 0) {
                        kvk[i] = *reinterpret_cast<const uint4*>(p.k_cache + src[i]);
                        kvv[i] = *reinterpret_cast<const uint4*>(p.v_cache + src[i]);
                    } else {
                        kvk[i] = kvv[i] = make_uint4(0, 0, 0, 0);
                    }
                }
#pragma unroll
                for (int i = 0; i < kMdBatch; ++i) {
                    const uint4 w = shfl_xor_u4(kvk[i], HL);
                    if (row[i] < 0) continue;
                    const bool sink = row[i] < v.s;
                    const uint4 kt = (sink || !p.rotate) ? kvk[i]
                                                          : md_turn_vec(kvk[i], w, wsn, wcs, first_half);
                    const long long dk =
                        ((((long long)b * 2 + 0) * p.Hkv + g) * p.S + row[i]) * p.D + 8 * jl;
                    const long long dv =
                        ((((long long)b * 2 + 1) * p.Hkv + g) * p.S + row[i]) * p.D + 8 * jl;
                    *reinterpret_cast<uint4*>(p.kv + dk) = kt;
                    *reinterpret_cast<uint4*>(p.kv + dv) = kvv[i];
                }
            }
        } else {
            // query item: RPW rows of q, each turned by its sequence's last cache index
            const long long r = (item - p.B - n_rows) * RPW + sub;
            const bool have = r < (long long)p.B * p.Hq;
            const int b = have ? (int)(r / p.Hq) : 0;
            const MdVisible v = md_visible(p, p.ctx_lens[b]);
            uint4 x = make_uint4(0, 0, 0, 0);
            if (have) x = *reinterpret_cast<const uint4*>(p.q + r * p.D + 8 * jl);
            const uint4 w = shfl_xor_u4(x, HL);
            if (!have || v.n == 0) continue;
            uint4 y = x;
            if (p.rotate && v.n > 1) {
                float sn[8], cs[8];
                md_lane_turn(turn, v.n - 1, d0, sn, cs);
                y = md_turn_vec(x, w, sn, cs, first_half);
            }
            *reinterpret_cast<uint4*>(p.q_eff + r * p.D + 8 * jl) = y;
        }
    }
}

// ------------------------------------------------------------- MagicDec, fused
// For up to 8 query heads per KV head the draft attention is computed in one
// kernel, one CTA of kMfWarps warps per (sequence, KV head) pair (a
// grid-stride loop over pairs), on the warp-level tensor cores: the pair's
// visible entries are taken kMfChunk at a time.  For a chunk, every thread
// looks up one entry's page (all lookups in flight together), then the CTA
// copies the chunk's K and V rows into shared memory with 16-byte
// asynchronous copies (all in flight together; entries past the visible ones
// and entries on a bad page are zero-filled), turns the window keys in place
// (pairs d, d + D/2 of a row; every window entry moves by the same s - w0, so
// one sine / cosine table per pair) and rounds them to bf16.  Warp w then owns
// 16 entries of the chunk: S^T = K Q^T and O^T += V^T (P_hi + P_lo)^T with
// the entries (and for PV the head dimensions) as the MMA's 16 rows and the
// G <= 8 query heads (turned by n - 1, rounded to bf16, in shared memory) as
// its 8 columns, and an online softmax in base 2 across chunks.  At the end
// the warps' (O, m, l) rows meet in shared memory (over the K/V rows, no
// longer needed) and are merged in warp order (deterministic).  A bad page,
// or a context length out of range, gives NaN rows and SPIRE_DEVERR_CTX_LEN,
// as on the gather path.
constexpr int kMfWarps = 5;                    // 80-entry chunks: sink 1 + window 64 in one
constexpr int kMfChunk = 16 * kMfWarps;

template <int D>
struct MfSmem {
    static constexpr int HALF = kMfChunk * 128;          // one 64-column half of the K or V rows
    static constexpr int KV = (D / 64) * HALF;
    static constexpr int SCR = D + 8;                    // floats per hand-over row
    static_assert(kMfWarps * 8 * SCR * 4 + kMfWarps * 8 * 8 <= 2 * KV,
                  "the hand-over fits over the K/V rows");
};

template <int D>
__global__ void __launch_bounds__(32 * kMfWarps, 4) magicdec_fused_kernel(const MdParams p) {
    using M = MfSmem<D>;
    __shared__ __align__(128) uint8_t kvs[2 * M::KV];    // K rows, then V rows (swizzled)
    __shared__ __align__(128) uint8_t qs[(D / 64) * 1024];   // Q^T source: 8 rows, swizzled
    __shared__ uint64_t turn[64];
    __shared__ float tw_sn[D / 2], tw_cs[D / 2];         // window turn s - w0, per element
    __shared__ float tq_sn[D / 2], tq_cs[D / 2];         // query turn n - 1, per element
    __shared__ long long src[kMfChunk];                  // element offset of an entry's row
    constexpr uint32_t FULL = 0xffffffffu;
    constexpr int DT = D / 16;
    const float NEG_INF = __int_as_float(0xff800000);
    const float NANF = __int_as_float(0x7fc00000);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gq = lane >> 2, tq = lane & 3;
    const int ra = 2 * tq, rb = ra + 1;                  // query heads of this lane's columns
    const uint32_t kbase = smem_u32(kvs), vbase = kbase + M::KV, qbase = smem_u32(qs);
    float* const scr_o = reinterpret_cast<float*>(kvs);
    float2* const scr_ml = reinterpret_cast<float2*>(kvs + kMfWarps * 8 * M::SCR * 4);
    if (tid < 64) turn[tid] = p.fturn[tid];
    uint32_t cta_err = 0;
    const long long pairs = (long long)p.B * p.Hkv;
    for (long long bg = blockIdx.x; bg < pairs; bg += gridDim.x) {
        const int g = (int)(bg % p.Hkv), b = (int)(bg / p.Hkv);
        const MdVisible v = md_visible(p, p.ctx_lens[b]);
        const bool turnw = p.rotate && v.s != v.w0, turnq = p.rotate && v.n > 1;
        __syncthreads();                                 // turn[] loaded; the last pair is done
        bool pbad = v.n == 0;                            // same in every thread
        // an entry's page id (thread e < kMfChunk, entry c0 + e), or -1 past the
        // visible entries; the load is issued here and consumed later
        auto page_of = [&](int c0) -> int {
            if (tid >= kMfChunk || c0 + tid >= v.n) return -1;
            const int c = c0 + tid;
            const int pos = c < v.s ? c : v.w0 + (c - v.s);
            return p.block_table[(long long)b * p.max_pages + pos / kPage];
        };
        const int id0 = page_of(0);                      // in flight during the tables
        // the per-element turns: of the window entries (s - w0) and of the query (n - 1)
        for (int d = tid; d < D / 2; d += blockDim.x) {
            float sn = 0.f, cs = 1.f, qsn = 0.f, qcs = 1.f;
            if (turnw) md_sincos(turn, (long long)v.s - v.w0, d, &sn, &cs);
            if (turnq) md_sincos(turn, (long long)v.n - 1, d, &qsn, &qcs);
            tw_sn[d] = sn;
            tw_cs[d] = cs;
            tq_sn[d] = qsn;
            tq_cs[d] = qcs;
        }
        float o[DT][4];
        float ma = NEG_INF, mb = NEG_INF, la = 0.f, lb = 0.f;
#pragma unroll
        for (int j = 0; j < DT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
        uint32_t qf[DT][2];
        for (int c0 = 0; c0 < v.n; c0 += kMfChunk) {
            const int ne = min(kMfChunk, v.n - c0);
            const int id = c0 == 0 ? id0 : page_of(c0);
            // ---- the chunk's pages (one lookup per thread, all in flight together)
            int badpg = 0;
            if (tid < kMfChunk) {
                long long sr = -1;                       // -1: no row (zero-filled)
                if (tid < ne) {
                    const int c = c0 + tid;
                    const int pos = c < v.s ? c : v.w0 + (c - v.s);
                    if (id >= 0 && id < p.num_pages)
                        sr = (((long long)id * p.Hkv + g) * kPage + pos % kPage) * D;
                    else
                        badpg = 1;
                }
                src[tid] = sr;
            }
            if (__syncthreads_or(badpg)) pbad = true;   // the tables and src[] are in place
            // ---- K and V rows into shared memory (row e, 16-byte chunk ch at
            // half ch / 8, row e, chunk (ch % 8) ^ (e % 8)); rows past the
            // visible entries, or on a bad page, zero-filled
            for (int i = tid; i < kMfChunk * (D / 8); i += blockDim.x) {
                const int e = i / (D / 8), ch = i - e * (D / 8);
                const uint32_t off = (ch >> 3) * M::HALF + e * 128 + (((ch & 7) ^ (e & 7)) << 4);
                const long long sr = src[e];
                if (sr >= 0) {
                    cp_async16(kbase + off, p.k_cache + sr + 8 * ch);
                    cp_async16(vbase + off, p.v_cache + sr + 8 * ch);
                } else {
                    *reinterpret_cast<uint4*>(kvs + off) = make_uint4(0u, 0u, 0u, 0u);
                    *reinterpret_cast<uint4*>(kvs + M::KV + off) = make_uint4(0u, 0u, 0u, 0u);
                }
            }
            if (c0 == 0) {
                // the query heads turned by n - 1, rounded to bf16, at their
                // swizzled places (element d and d + D/2 of row h; rows >= G zero)
                __nv_bfloat16* const q16 = reinterpret_cast<__nv_bfloat16*>(qs);
                for (int i = tid; i < 8 * (D / 2); i += blockDim.x) {
                    const int h = i / (D / 2), d = i - h * (D / 2);
                    float x0 = 0.f, x1 = 0.f;
                    if (h < p.G) {
                        const __nv_bfloat16* qr =
                            p.q + ((long long)b * p.Hq + (long long)g * p.G + h) * D;
                        const float a0 = __bfloat162float(qr[d]), a1 = __bfloat162float(qr[d + D / 2]);
                        x0 = turnq ? a0 * tq_cs[d] - a1 * tq_sn[d] : a0;
                        x1 = turnq ? a1 * tq_cs[d] + a0 * tq_sn[d] : a1;
                    }
                    const int e0 = d, e1 = d + D / 2;
                    q16[(e0 >> 6) * 512 + h * 64 + ((((e0 & 63) >> 3) ^ h) << 3) + (e0 & 7)] =
                        __float2bfloat16_rn(x0);
                    q16[(e1 >> 6) * 512 + h * 64 + ((((e1 & 63) >> 3) ^ h) << 3) + (e1 & 7)] =
                        __float2bfloat16_rn(x1);
                }
            }
            cp_async_wait_all();
            __syncthreads();
            // ---- window keys turned by s - w0 and rounded to bf16, in place
            if (turnw) {
                for (int i = tid; i < kMfChunk * (D / 16); i += blockDim.x) {
                    const int e = i / (D / 16), ch = i - e * (D / 16), ch2 = ch + D / 16;
                    if (e >= ne || c0 + e < v.s || src[e] < 0) continue;   // sinks keep their turn
                    const uint32_t off1 = (ch >> 3) * M::HALF + e * 128 + (((ch & 7) ^ (e & 7)) << 4);
                    const uint32_t off2 = (ch2 >> 3) * M::HALF + e * 128 + (((ch2 & 7) ^ (e & 7)) << 4);
                    uint4* const p1 = reinterpret_cast<uint4*>(kvs + off1);
                    uint4* const p2 = reinterpret_cast<uint4*>(kvs + off2);
                    const uint4 a = *p1, w = *p2;
                    const uint32_t av[4] = {a.x, a.y, a.z, a.w}, wv[4] = {w.x, w.y, w.z, w.w};
                    uint32_t r1[4], r2[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int d = 8 * ch + 2 * q;
                        const float a0 = bf16lo_to_f32(av[q]), a1 = bf16hi_to_f32(av[q]);
                        const float b0 = bf16lo_to_f32(wv[q]), b1 = bf16hi_to_f32(wv[q]);
                        r1[q] = pack_bf16(a0 * tw_cs[d] - b0 * tw_sn[d], a1 * tw_cs[d + 1] - b1 * tw_sn[d + 1]);
                        r2[q] = pack_bf16(b0 * tw_cs[d] + a0 * tw_sn[d], b1 * tw_cs[d + 1] + a1 * tw_sn[d + 1]);
                    }
                    *p1 = make_uint4(r1[0], r1[1], r1[2], r1[3]);
                    *p2 = make_uint4(r2[0], r2[1], r2[2], r2[3]);
                }
                __syncthreads();
            }
            if (c0 == 0) {
                // B = Q^T: lane (gq, tq) takes row gq, columns 2 tq, 2 tq + 1 of the
                // 8x8 blocks at 16-byte chunks 2 ks and 2 ks + 1
                const int qrow = lane & 7;
#pragma unroll
                for (int ks = 0; ks < DT; ks += 2) {
                    const int chunk = 2 * ks + (lane >> 3);
                    ldsm_x4(qf[ks][0], qf[ks][1], qf[ks + 1][0], qf[ks + 1][1],
                            qbase + (chunk >> 3) * 1024 + qrow * 128 + (((chunk & 7) ^ qrow) << 4));
                }
            }
            // ---- this warp's 16 entries: S^T = K Q^T (two accumulation chains)
            const int wkey = 16 * warp;
            const int krow = wkey + ((lane >> 3) & 1) * 8 + (lane & 7);
            const int vrow = wkey + ((lane >> 4) << 3) + (lane & 7);
            float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int ks = 0; ks < DT; ++ks) {
                const int chunk = 2 * ks + (lane >> 4);
                uint32_t a[4];
                ldsm_x4(a[0], a[1], a[2], a[3],
                        kbase + (chunk >> 3) * M::HALF + krow * 128 + (((chunk & 7) ^ (lane & 7)) << 4));
                if (ks & 1) mma_bf16(s1, a, qf[ks][0], qf[ks][1]);
                else        mma_bf16(s0, a, qf[ks][0], qf[ks][1]);
            }
            float s[4] = {s0[0] + s1[0], s0[1] + s1[1], s0[2] + s1[2], s0[3] + s1[3]};
            if (wkey + gq >= ne) s[0] = s[1] = NEG_INF;          // past the visible entries
            if (wkey + gq + 8 >= ne) s[2] = s[3] = NEG_INF;
            // ---- online softmax (base 2); a head's 16 entries sit in the 8 lanes of its tq
            float xa = fmaxf(s[0], s[2]), xb = fmaxf(s[1], s[3]);
#pragma unroll
            for (int off = 4; off < 32; off <<= 1) {
                xa = fmaxf(xa, __shfl_xor_sync(FULL, xa, off));
                xb = fmaxf(xb, __shfl_xor_sync(FULL, xb, off));
            }
            const float mna = fmaxf(ma, xa * p.sl2), mnb = fmaxf(mb, xb * p.sl2);
            const float mra = (mna == NEG_INF) ? 0.f : mna;
            const float mrb = (mnb == NEG_INF) ? 0.f : mnb;
            const float aa = ex2(ma - mra), ab = ex2(mb - mrb);
            ma = mna; mb = mnb;
            s[0] = ex2(fmaf(s[0], p.sl2, -mra));
            s[1] = ex2(fmaf(s[1], p.sl2, -mrb));
            s[2] = ex2(fmaf(s[2], p.sl2, -mra));
            s[3] = ex2(fmaf(s[3], p.sl2, -mrb));
            la = la * aa + (s[0] + s[2]);
            lb = lb * ab + (s[1] + s[3]);
#pragma unroll
            for (int j = 0; j < DT; ++j) {
                o[j][0] *= aa; o[j][1] *= ab;
                o[j][2] *= aa; o[j][3] *= ab;
            }
            // ---- O^T += V^T (P_hi + P_lo)^T, P^T moved into the B layout
            const uint32_t h0 = pack_bf16(s[0], s[1]), h1 = pack_bf16(s[2], s[3]);
            const uint32_t l0 = pack_bf16(s[0] - bf16lo_to_f32(h0), s[1] - bf16hi_to_f32(h0));
            const uint32_t l1 = pack_bf16(s[2] - bf16lo_to_f32(h1), s[3] - bf16hi_to_f32(h1));
            const uint32_t bh0 = movm_trans(h0), bh1 = movm_trans(h1);
            const uint32_t bl0 = movm_trans(l0), bl1 = movm_trans(l1);
#pragma unroll
            for (int j = 0; j < DT; ++j) {
                const int chunk = 2 * j + ((lane >> 3) & 1);
                uint32_t a[4];
                ldsm_x4_trans(a[0], a[1], a[2], a[3],
                              vbase + (chunk >> 3) * M::HALF + vrow * 128 + (((chunk & 7) ^ (lane & 7)) << 4));
                mma_bf16(o[j], a, bh0, bh1);
                mma_bf16(o[j], a, bl0, bl1);
            }
            __syncthreads();                             // the rows are read: next chunk, or hand-over
        }
        // ---- the warps' rows meet in shared memory, merged in warp order
        float lta = la, ltb = lb;
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            lta += __shfl_xor_sync(FULL, lta, off);
            ltb += __shfl_xor_sync(FULL, ltb, off);
        }
        float* const so = scr_o + warp * 8 * M::SCR;
        if (ra < p.G) {
#pragma unroll
            for (int j = 0; j < DT; ++j) {
                so[ra * M::SCR + 16 * j + gq] = o[j][0];
                so[ra * M::SCR + 16 * j + gq + 8] = o[j][2];
            }
        }
        if (rb < p.G) {
#pragma unroll
            for (int j = 0; j < DT; ++j) {
                so[rb * M::SCR + 16 * j + gq] = o[j][1];
                so[rb * M::SCR + 16 * j + gq + 8] = o[j][3];
            }
        }
        if (gq == 0) {
            scr_ml[warp * 8 + ra] = make_float2(ma, lta);
            scr_ml[warp * 8 + rb] = make_float2(mb, ltb);
        }
        __syncthreads();
        if (pbad) cta_err |= kErrCtxLen;
        for (int i = tid; i < p.G * D; i += blockDim.x) {
            const int h = i / D, d = i - h * D;
            float Mx = NEG_INF;
#pragma unroll
            for (int w = 0; w < kMfWarps; ++w) Mx = fmaxf(Mx, scr_ml[w * 8 + h].x);
            const float Mr = (Mx == NEG_INF) ? 0.f : Mx;
            float L = 0.f, O = 0.f;
#pragma unroll
            for (int w = 0; w < kMfWarps; ++w) {
                const float2 ml = scr_ml[w * 8 + h];
                const float sc = ex2(ml.x - Mr);
                L = fmaf(ml.y, sc, L);
                O = fmaf(scr_o[(w * 8 + h) * M::SCR + d], sc, O);
            }
            p.out[((long long)b * p.Hq + (long long)g * p.G + h) * D + d] =
                (pbad || !(L > 0.f)) ? NANF : O / L;
        }
    }
    // one error word per CTA: every CTA writes its own, nothing needs clearing
    if (tid == 0) {
        p.err[blockIdx.x] = (int32_t)cta_err;
        if (blockIdx.x == 0) p.header[0] = (int32_t)gridDim.x;
    }
}

// spire_test_draft_slots: the inline slot helper evaluated on the device
__global__ void draft_slots_kernel(int64_t* out, long long n, int32_t n_sink, int32_t window) {
    for (long long p = blockIdx.x * (long long)blockDim.x + threadIdx.x; p < n;
         p += (long long)gridDim.x * blockDim.x)
        out[p] = spire_draft_slot_inline(p, n_sink, window);
}

struct MdLayout {
    size_t draft, kv, q, nvis, total;
};

// query heads per KV head padded to 1, 2, 4 or 8 (fused path), 0 if above 8
int md_fused_gp(const spire_attn_desc* d) {
    const int G = d->num_q_heads / d->num_kv_heads;
    return G <= 1 ? 1 : G <= 2 ? 2 : G <= 4 ? 4 : G <= 8 ? 8 : 0;
}

// fused path workspace: header word | error words (one per CTA)
size_t md_fused_bytes(const spire_attn_desc* d) {
    if (md_fused_gp(d) == 0) return 0;
    return kHeaderBytes + align256(size_t(kMaxCtas) * 4);
}

MdLayout md_layout(const spire_attn_desc* d, int S) {
    MdLayout l{};
    l.draft = 0;
    size_t off = ws_layout(d->batch, d->num_kv_heads, rows_per_kv_head(d, 1), d->head_dim).total;
    l.kv = off;   off += align256((size_t)d->batch * 2 * d->num_kv_heads * S * d->head_dim * 2);
    l.q = off;    off += align256((size_t)d->batch * d->num_q_heads * d->head_dim * 2);
    l.nvis = off; off += align256((size_t)d->batch * 4);
    l.total = off;
    return l;
}

// Test hook (spire_test_stall_next_call): the next attention call made by this
// host thread stalls one pair.
struct TestStall {
    bool armed = false;
    int32_t pair = -1;
};
thread_local TestStall g_test_stall;

// Launches the attention for one call: a one-CTA kernel zeroing the pair
// counters, then the attention kernel, each a programmatic dependent of the
// kernel before it (each waits for that kernel to complete before it touches
// global memory).  With counters_zeroed the kernel launched just before
// (which must have zeroed them, and may have written ctx_lens) is the
// attention kernel's dependency.
spire_status run(int mode, const void* q, const CUtensorMap& tk, const CUtensorMap& tv,
                 const int32_t* block_table, const int32_t* ctx_lens, int kp1,
                 const spire_attn_desc* d, int cap, float* out, void* workspace,
                 cudaStream_t stream, bool counters_zeroed = false) {
    DeviceInfo di;
    spire_status st = device_info(&di);
    if (st != SPIRE_OK) return st;
    if (di.smem_optin < kMaxDynSmem) return SPIRE_ERR_UNSUPPORTED;
    const int B = d->batch, Hkv = d->num_kv_heads, D = d->head_dim;
    const int R = rows_per_kv_head(d, kp1);
    const WsLayout w = ws_layout(B, Hkv, R, D);
    char* ws = static_cast<char*>(workspace);

    AttnParams ap{};
    ap.q = static_cast<const __nv_bfloat16*>(q);
    ap.out = out;
    ap.ctx_lens = ctx_lens;
    ap.block_table = block_table;
    ap.header = reinterpret_cast<int32_t*>(ws);
    ap.err = reinterpret_cast<int32_t*>(ws + w.err);
    ap.cnt = reinterpret_cast<int32_t*>(ws + w.cnt);
    ap.stamps = reinterpret_cast<unsigned long long*>(ws + w.stamps);
    ap.part_lse = reinterpret_cast<float*>(ws + w.part_lse);
    ap.part_o = reinterpret_cast<float*>(ws + w.part_o);
    ap.B = B;
    ap.Hq = d->num_q_heads;
    ap.Hkv = Hkv;
    ap.G = d->num_q_heads / Hkv;
    ap.kp1 = kp1;
    ap.R = R;
    ap.max_pages = mode == kModeVerify ? d->max_pages_per_seq : 0;
    ap.num_pages = mode == kModeVerify ? d->num_pages : 0;
    ap.cap = cap;
    ap.mode = mode;
    ap.sl2 = static_cast<float>(static_cast<double>(d->softmax_scale) * kLog2e);

    CUtensorMap tq;
    if (!encode_q_map(&tq, q, D, d->num_q_heads, uint64_t(B) * kp1, ap.G, kp1))
        return SPIRE_ERR_CUDA;
    if (!counters_zeroed) {
        if (launch_dependent(zero_counters_kernel, dim3(1), dim3(256), 0, stream, ap.cnt,
                             B * Hkv) != cudaSuccess)
            return SPIRE_ERR_CUDA;
    }
    const int ctas = di.sms < kMaxCtas ? di.sms : kMaxCtas;
    const int mt = (R + 15) / 16;
    // tcgen05 path when a KV head serves enough query rows to make QK^T and PV
    // real contractions; the warp-MMA path for the few-row draft step, whose
    // short pairs favour its lighter per-pair epilogue (measured on GB300)
    const bool use_tc = R > 8;
    // the split's per-pair weight, from per-CTA timings on GB300 (busy time
    // against planned tiles and segments): ~4 tiles for the tcgen05 kernel,
    // whose softmax warps run the segment epilogue and the merge, ~1 for the
    // warp-MMA kernel, whose epilogue warp works beside the stream
    ap.head = use_tc ? kHeadTc : kHeadMma;
    cudaError_t e;
    const int nc = R <= 32 ? 4 : (R <= 64 ? 2 : 1);   // query copies of the tcgen05 kernel
    if (g_test_stall.armed) {      // spire_test_stall_next_call: this thread's next call only
        g_test_stall.armed = false;
        if (D == 128) {
            e = launch_stall_d128(use_tc, nc, g_test_stall.pair, tk, tv, tq, ap, ctas, stream);
            return e == cudaSuccess ? SPIRE_OK : SPIRE_ERR_CUDA;
        }
    }
    if (use_tc)
        e = D == 128 ? launch_attn_tc_d128(nc, tk, tv, tq, ap, ctas, stream)
                     : launch_attn_tc_d64(nc, tk, tv, tq, ap, ctas, stream);
    else
        e = D == 128 ? launch_attn_d128(mt, tk, tv, tq, ap, ctas, stream)
                     : launch_attn_d64(mt, tk, tv, tq, ap, ctas, stream);
    return e == cudaSuccess ? SPIRE_OK : SPIRE_ERR_CUDA;
}

}  // namespace
}  // namespace spire

using namespace spire;

extern "C" {

size_t spire_verify_workspace_bytes(const spire_attn_desc* desc, int32_t k) {
    if (check_common(desc) != SPIRE_OK || k < 0 || k >= SPIRE_MAX_ROWS_PER_KV_HEAD) return 0;
    const int R = rows_per_kv_head(desc, k + 1);
    return ws_layout(desc->batch, desc->num_kv_heads, R, desc->head_dim).total;
}

size_t spire_draft_workspace_bytes(const spire_attn_desc* desc, int32_t n_sink, int32_t window) {
    if (check_common(desc) != SPIRE_OK || n_sink < 0 || window < 1) return 0;
    const int R = rows_per_kv_head(desc, 1);
    return ws_layout(desc->batch, desc->num_kv_heads, R, desc->head_dim).total;
}

spire_status spire_verify_attention(const void* q, const void* k_cache, const void* v_cache,
                                    const int32_t* block_table, const int32_t* ctx_lens,
                                    int32_t k, const spire_attn_desc* desc, float* out,
                                    void* workspace, size_t ws_bytes, void* stream) {
    spire_status st = check_common(desc);
    if (st != SPIRE_OK) return st;
    if (k < 0) return SPIRE_ERR_INVALID_ARG;
    if (desc->page_size != kPage) return SPIRE_ERR_UNSUPPORTED;
    if (desc->max_pages_per_seq < 1 || desc->num_pages < 1) return SPIRE_ERR_INVALID_ARG;
    if (rows_per_kv_head(desc, 1) > SPIRE_MAX_ROWS_PER_KV_HEAD ||
        (long long)rows_per_kv_head(desc, 1) * (k + 1LL) > SPIRE_MAX_ROWS_PER_KV_HEAD)
        return SPIRE_ERR_UNSUPPORTED;
    // TMA plane index page * Hkv + g and the block-table offset are int32
    if ((long long)desc->num_pages * desc->num_kv_heads >= (1LL << 31) ||
        (long long)desc->batch * desc->max_pages_per_seq >= (1LL << 31) ||
        (long long)desc->max_pages_per_seq * kPage >= (1LL << 31))
        return SPIRE_ERR_UNSUPPORTED;
    if (desc->batch == 0) return SPIRE_OK;
    if (!q || !k_cache || !v_cache || !block_table || !ctx_lens || !out)
        return SPIRE_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) ||
        !aligned(block_table, 4) || !aligned(ctx_lens, 4))
        return SPIRE_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) || ws_bytes < spire_verify_workspace_bytes(desc, k))
        return SPIRE_ERR_WORKSPACE;

    CUtensorMap tk, tv;
    const uint64_t planes = uint64_t(desc->num_pages) * uint64_t(desc->num_kv_heads);
    if (!encode_kv_map(&tk, k_cache, desc->head_dim, kPage, planes) ||
        !encode_kv_map(&tv, v_cache, desc->head_dim, kPage, planes))
        return SPIRE_ERR_CUDA;
    return run(kModeVerify, q, tk, tv, block_table, ctx_lens, k + 1, desc, 0, out, workspace,
               static_cast<cudaStream_t>(stream));
}

spire_status spire_draft_sparse_attention(const void* q, const void* kv, const int32_t* ctx_lens,
                                          int32_t n_sink, int32_t window,
                                          const spire_attn_desc* desc, float* out,
                                          void* workspace, size_t ws_bytes, void* stream) {
    spire_status st = check_common(desc);
    if (st != SPIRE_OK) return st;
    if (n_sink < 0 || window < 1) return SPIRE_ERR_INVALID_ARG;
    const long long S = (long long)n_sink + window;
    if (S > (1LL << 30)) return SPIRE_ERR_UNSUPPORTED;
    if (rows_per_kv_head(desc, 1) > SPIRE_MAX_ROWS_PER_KV_HEAD) return SPIRE_ERR_UNSUPPORTED;
    if ((long long)desc->batch * 2 * desc->num_kv_heads >= (1LL << 31)) return SPIRE_ERR_UNSUPPORTED;
    if (desc->batch == 0) return SPIRE_OK;
    if (!q || !kv || !ctx_lens || !out) return SPIRE_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(kv, 16) || !aligned(out, 16) || !aligned(ctx_lens, 4))
        return SPIRE_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) ||
        ws_bytes < spire_draft_workspace_bytes(desc, n_sink, window))
        return SPIRE_ERR_WORKSPACE;

    CUtensorMap tkv;
    const uint64_t planes = uint64_t(desc->batch) * 2u * uint64_t(desc->num_kv_heads);
    if (!encode_kv_map(&tkv, kv, desc->head_dim, uint64_t(S), planes)) return SPIRE_ERR_CUDA;
    return run(kModeDraft, q, tkv, tkv, nullptr, ctx_lens, 1, desc, int(S), out, workspace,
               static_cast<cudaStream_t>(stream));
}

size_t spire_magicdec_workspace_bytes(const spire_attn_desc* desc, int32_t n_sink,
                                      int32_t window) {
    if (check_common(desc) != SPIRE_OK || n_sink < 0 || window < 1 ||
        (long long)n_sink + window > 65536)
        return 0;
    const size_t gather = md_layout(desc, n_sink + window).total, fused = md_fused_bytes(desc);
    return gather > fused ? gather : fused;
}

spire_status spire_magicdec_attention(const void* q, const void* k_cache, const void* v_cache,
                                      const int32_t* block_table, const int32_t* ctx_lens,
                                      int32_t n_sink, int32_t window, float rope_theta,
                                      const spire_attn_desc* desc, float* out, void* workspace,
                                      size_t ws_bytes, void* stream) {
    spire_status st = check_common(desc);
    if (st != SPIRE_OK) return st;
    if (n_sink < 0 || window < 1 || !std::isfinite(rope_theta) || rope_theta < 0.f)
        return SPIRE_ERR_INVALID_ARG;
    if ((long long)n_sink + window > 65536) return SPIRE_ERR_UNSUPPORTED;
    if (desc->page_size != kPage) return SPIRE_ERR_UNSUPPORTED;
    if (desc->max_pages_per_seq < 1 || desc->num_pages < 1) return SPIRE_ERR_INVALID_ARG;
    if (rows_per_kv_head(desc, 1) > SPIRE_MAX_ROWS_PER_KV_HEAD) return SPIRE_ERR_UNSUPPORTED;
    if ((long long)desc->num_pages * desc->num_kv_heads >= (1LL << 31) ||
        (long long)desc->batch * desc->max_pages_per_seq >= (1LL << 31) ||
        (long long)desc->max_pages_per_seq * kPage >= (1LL << 31) ||
        (long long)desc->batch * 2 * desc->num_kv_heads >= (1LL << 31))
        return SPIRE_ERR_UNSUPPORTED;
    if (desc->batch == 0) return SPIRE_OK;
    if (!q || !k_cache || !v_cache || !block_table || !ctx_lens || !out)
        return SPIRE_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) ||
        !aligned(block_table, 4) || !aligned(ctx_lens, 4))
        return SPIRE_ERR_INVALID_ARG;
    const int S = n_sink + window;
    const MdLayout l = md_layout(desc, S);
    const size_t need = l.total > md_fused_bytes(desc) ? l.total : md_fused_bytes(desc);
    if (!workspace || !aligned(workspace, 256) || ws_bytes < need) return SPIRE_ERR_WORKSPACE;
    DeviceInfo di;
    st = device_info(&di);
    if (st != SPIRE_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    char* ws = static_cast<char*>(workspace);

    MdParams mp{};
    mp.q = static_cast<const __nv_bfloat16*>(q);
    mp.k_cache = static_cast<const __nv_bfloat16*>(k_cache);
    mp.v_cache = static_cast<const __nv_bfloat16*>(v_cache);
    mp.block_table = block_table;
    mp.ctx_lens = ctx_lens;
    mp.kv = reinterpret_cast<__nv_bfloat16*>(ws + l.kv);
    mp.q_eff = reinterpret_cast<__nv_bfloat16*>(ws + l.q);
    mp.n_vis = reinterpret_cast<int32_t*>(ws + l.nvis);
    // the attention's workspace starts the MagicDec workspace: its pair
    // counters are zeroed by the gather, so no separate zeroing launch
    mp.cnt = reinterpret_cast<int32_t*>(
        ws + ws_layout(desc->batch, desc->num_kv_heads, rows_per_kv_head(desc, 1), desc->head_dim).cnt);
    mp.B = desc->batch;
    mp.Hq = desc->num_q_heads;
    mp.Hkv = desc->num_kv_heads;
    mp.D = desc->head_dim;
    mp.S = S;
    mp.n_sink = n_sink;
    mp.window = window;
    mp.max_pages = desc->max_pages_per_seq;
    mp.num_pages = desc->num_pages;
    mp.rotate = rope_theta > 0.f;
    // the rotary frequencies theta^(-2d/D) (the same libm pow as the
    // definition) as per-call fixed-point turn constants
    for (int d = 0; d < desc->head_dim / 2; ++d)
        mp.fturn[d] = mp.rotate
                          ? rope_turn_fixed(std::pow((double)rope_theta, -2.0 * d / desc->head_dim))
                          : 0;
    const int gp = md_fused_gp(desc);
    if (gp != 0) {
        // up to 8 query heads per KV head: the fused kernel and its merge
        mp.G = desc->num_q_heads / desc->num_kv_heads;
        mp.sl2 = static_cast<float>(static_cast<double>(desc->softmax_scale) * kLog2e);
        mp.header = reinterpret_cast<int32_t*>(ws);
        mp.err = reinterpret_cast<int32_t*>(ws + kHeaderBytes);
        mp.out = out;
        const long long pairs = (long long)mp.B * mp.Hkv;
        const long long fblocks = pairs < kMaxCtas ? pairs : kMaxCtas;   // one error word each
        void (*fk)(MdParams) = desc->head_dim == 128 ? magicdec_fused_kernel<128>
                               : desc->head_dim == 64  ? magicdec_fused_kernel<64>
                                                       : nullptr;
        if (!fk) return SPIRE_ERR_UNSUPPORTED;
        fk<<<(unsigned)fblocks, 32 * kMfWarps, 0, s>>>(mp);   // after all prior work
        return cudaGetLastError() == cudaSuccess ? SPIRE_OK : SPIRE_ERR_CUDA;
    }
    const int rpw = 32 / (desc->head_dim / 8);     // query rows per warp item
    const long long items = (long long)mp.B * (1 + (long long)mp.Hkv * kMdParts) +
                            ((long long)mp.B * mp.Hq + rpw - 1) / rpw;
    long long blocks = (items * 32 + 255) / 256;
    if (blocks > 32LL * di.sms) blocks = 32LL * di.sms;
    magicdec_gather_kernel<<<(unsigned)blocks, 256, 0, s>>>(mp);   // a plain launch: after all prior work
    if (cudaGetLastError() != cudaSuccess) return SPIRE_ERR_CUDA;

    CUtensorMap tkv;
    const uint64_t planes = uint64_t(desc->batch) * 2u * uint64_t(desc->num_kv_heads);
    if (!encode_kv_map(&tkv, mp.kv, desc->head_dim, uint64_t(S), planes)) return SPIRE_ERR_CUDA;
    return run(kModeDraft, mp.q_eff, tkv, tkv, nullptr, mp.n_vis, 1, desc, S, out, workspace, s,
               true);
}

int64_t spire_draft_slot(int64_t pos, int32_t n_sink, int32_t window) {
    return spire_draft_slot_inline(pos, n_sink, window);
}

spire_status spire_test_draft_slots(int64_t* out, int64_t n, int32_t n_sink, int32_t window,
                                    void* stream) {
    if (n < 0) return SPIRE_ERR_INVALID_ARG;
    if (n == 0) return SPIRE_OK;
    if (!out || !aligned(out, 8)) return SPIRE_ERR_INVALID_ARG;
    const long long blocks = (n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096;
    draft_slots_kernel<<<(unsigned)blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        out, (long long)n, n_sink, window);
    return cudaGetLastError() == cudaSuccess ? SPIRE_OK : SPIRE_ERR_CUDA;
}

spire_status spire_get_device_error(const void* workspace, int32_t* code_out, void* stream) {
    if (!workspace || !code_out) return SPIRE_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // the header word first, then exactly the words it counts: a workspace
    // holds at least kHeaderBytes plus the words its last call wrote
    int32_t n = 0;
    if (cudaMemcpyAsync(&n, workspace, sizeof(n), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return SPIRE_ERR_CUDA;
    if (n < 0 || n > kMaxCtas) n = 0;
    int32_t buf[kMaxCtas];
    if (n > 0 && (cudaMemcpyAsync(buf, static_cast<const char*>(workspace) + kHeaderBytes,
                                  (size_t)n * 4, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
                  cudaStreamSynchronize(s) != cudaSuccess))
        return SPIRE_ERR_CUDA;
    int32_t v = 0;
    for (int c = 0; c < n; ++c) v |= buf[c];
    *code_out = v;
    return SPIRE_OK;
}

spire_status spire_get_cta_times(const void* workspace, size_t ws_bytes, uint64_t* ns_out,
                                 int32_t max_ctas, int32_t* n_out, void* stream) {
    if (!workspace || !n_out || max_ctas < 0 || (max_ctas > 0 && !ns_out))
        return SPIRE_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int32_t n = 0;
    if (ws_bytes < kHeaderBytes) return SPIRE_ERR_WORKSPACE;
    if (cudaMemcpyAsync(&n, workspace, sizeof(n), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return SPIRE_ERR_CUDA;
    if (n < 0 || n > kMaxCtas) n = 0;
    if (kStampsOffset + (size_t)n * 16 > ws_bytes) return SPIRE_ERR_WORKSPACE;
    const int m = n < max_ctas ? n : max_ctas;
    if (m > 0 && (cudaMemcpyAsync(ns_out, static_cast<const char*>(workspace) + kStampsOffset,
                                  (size_t)m * 16, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
                  cudaStreamSynchronize(s) != cudaSuccess))
        return SPIRE_ERR_CUDA;
    *n_out = n;
    return SPIRE_OK;
}

spire_status spire_test_stall_next_call(int32_t pair) {
    if (pair < 0) return SPIRE_ERR_INVALID_ARG;
    g_test_stall.armed = true;
    g_test_stall.pair = pair;
    return SPIRE_OK;
}

spire_status spire_stream_read(const void* src, size_t bytes, void* stream) {
    if (bytes == 0) return SPIRE_OK;
    if (!src || !aligned(src, 16) || bytes % 16 != 0) return SPIRE_ERR_INVALID_ARG;
    DeviceInfo di;
    const spire_status st = device_info(&di);
    if (st != SPIRE_OK) return st;
    static std::atomic<unsigned long long> done{0ull};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SPIRE_ERR_CUDA;
    const unsigned long long bit = dev >= 0 && dev < 64 ? (1ull << dev) : 0ull;
    if (!bit || !(done.load(std::memory_order_acquire) & bit)) {
        if (cudaFuncSetAttribute(stream_read_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kFloorSmem) != cudaSuccess)
            return SPIRE_ERR_CUDA;
        done.fetch_or(bit, std::memory_order_acq_rel);
    }
    stream_read_kernel<<<di.sms, 64, kFloorSmem, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint8_t*>(src), (unsigned long long)bytes);
    return cudaGetLastError() == cudaSuccess ? SPIRE_OK : SPIRE_ERR_CUDA;
}

const char* spire_status_string(spire_status status) {
    switch (status) {
        case SPIRE_OK: return "SPIRE_OK";
        case SPIRE_ERR_INVALID_ARG: return "SPIRE_ERR_INVALID_ARG";
        case SPIRE_ERR_UNSUPPORTED: return "SPIRE_ERR_UNSUPPORTED";
        case SPIRE_ERR_WORKSPACE: return "SPIRE_ERR_WORKSPACE";
        case SPIRE_ERR_CUDA: return "SPIRE_ERR_CUDA";
    }
    return "SPIRE_ERR_UNKNOWN";
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Verification attention without a caller-provided workspace.
//
// Some callers cannot allocate device memory when they call us: a serving
// engine that hands all free GPU memory to its KV-cache pool at start-up, or a
// plugin / foreign-function host that passes only input and output pointers
// and has no CUDA allocator of its own.  For them the split partials, arrival
// counters and error words live in one file-scope device array of fixed size
// that every GPU loading this library reserves until the process exits.
namespace {

constexpr size_t kStaticWsBytes = size_t(32) << 20;   // 32 MiB

static __device__ __align__(256) unsigned char g_static_ws[kStaticWsBytes];

// Unique id of the calling thread's current context, or 0 when there is none
// (or the driver lacks cuCtxGetId).  A context created after cudaDeviceReset
// gets a new id even where its handle value repeats, so a device address
// cached for an older context is never reused.
unsigned long long current_ctx_id() {
    using GetCurrent = CUresult (*)(CUcontext*);
    using GetId = CUresult (*)(CUcontext, unsigned long long*);
    static GetCurrent get_current = nullptr;
    static GetId get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<GetCurrent>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<GetId>(p);
    });
    if (!get_current || !get_id) return 0;
    CUcontext c = nullptr;
    if (get_current(&c) != CUDA_SUCCESS || !c) return 0;
    unsigned long long id = 0;
    return get_id(c, &id) == CUDA_SUCCESS ? id : 0;
}

// Device address of g_static_ws on the current device, looked up
// (cudaGetSymbolAddress, which allocates nothing) on the first call for each
// device and again whenever the device's context has changed since.
spire_status static_ws_address(void** out) {
    static std::mutex mu;
    static void* addr[64] = {};
    static unsigned long long ctx[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SPIRE_ERR_CUDA;
    std::lock_guard<std::mutex> g(mu);
    const bool slot = dev >= 0 && dev < 64;
    const unsigned long long id = current_ctx_id();
    if (slot && addr[dev] && id != 0 && ctx[dev] == id) {
        *out = addr[dev];
        return SPIRE_OK;
    }
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_ws) != cudaSuccess || !p) return SPIRE_ERR_CUDA;
    if (slot) {
        addr[dev] = p;
        ctx[dev] = current_ctx_id();   // the lookup made the primary context current if none was
    }
    *out = p;
    return SPIRE_OK;
}

}  // namespace

extern "C" spire_status spire_verify_attention_noalloc(const void* q, const void* k_cache,
                                                       const void* v_cache,
                                                       const int32_t* block_table,
                                                       const int32_t* ctx_lens, int32_t k,
                                                       const spire_attn_desc* desc, float* out,
                                                       void* stream) {
    // Invalid descriptors have no workspace size: report them exactly as the
    // workspace entry point does.  Otherwise its ordered checks see the static
    // array, so a valid, non-empty shape that needs more than it holds is the
    // only one that gets SPIRE_ERR_WORKSPACE (an empty batch is a no-op, an
    // unsupported page size SPIRE_ERR_UNSUPPORTED, as there).
    if (spire_verify_workspace_bytes(desc, k) == 0)
        return spire_verify_attention(q, k_cache, v_cache, block_table, ctx_lens, k, desc, out,
                                      nullptr, 0, stream);
    void* ws = nullptr;
    const spire_status st = static_ws_address(&ws);
    if (st != SPIRE_OK) return st;
    return spire_verify_attention(q, k_cache, v_cache, block_table, ctx_lens, k, desc, out, ws,
                                  kStaticWsBytes, stream);
}
