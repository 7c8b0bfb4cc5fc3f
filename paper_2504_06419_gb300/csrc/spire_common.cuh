// spire_common.cuh -- work decomposition shared by the libspire attention
// kernels.
//
// One speculation round of SPIRe (arXiv 2504.06419) spends its attention time
// streaming KV caches: the target's full cache once for the k+1 block tokens
// (Section 2, t_verify) and the draft's bounded sink + window cache once per
// draft step (Section 3.1).  Both are the same flash-decoding shape: a few
// query rows per KV head against a run of 64-token K/V tiles.
//
// Decomposition.  The unit of work is one 64-token tile of one
// (sequence b, KV head g) pair, plus `head` units of fixed cost per pair (its
// query load and epilogue).  Pairs are laid end to end in the order (b, g),
// each as [head units | T tile units], numbered globally 0..W-1.  CTA c
// of a grid of N takes the contiguous range [floor(cW/N), floor((c+1)W/N)):
// every SM gets the same work whatever the spread of lengths, counting the
// per-pair cost that many short pairs add.  A pair whose
// tiles straddle CTA ranges is computed in segments; each segment leaves a
// normalised partial (O, log-sum-exp) in a slot of the workspace, and the
// CTA that finishes a pair's last segment (an arrival counter decides)
// merges them.  The split depends only on ctx_lens, the shapes and N, and
// partials are merged in slot order, so results are deterministic.
//
// Every CTA derives W and its own starting pair from ctx_lens with a
// block-wide scan; there is no planning kernel.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "spire_ptx.cuh"

namespace spire {

constexpr int kPage = 64;        // tokens per K/V tile (and per page)
constexpr int kMaxCtas = 512;    // grid cap; the workspace holds 2 partial slots per CTA
// Per-pair fixed cost in tile units (AttnParams::head), chosen per kernel by
// the host: a pair's start and end (Q load, epilogue, output or partial) cost
// the tcgen05 kernel about four tiles, the warp-MMA kernel about one.

constexpr uint32_t kErrCtxLen = 1u;
constexpr uint32_t kErrPageId = 2u;
constexpr uint32_t kErrTimeout = 4u;

enum Mode : int32_t { kModeVerify = 0, kModeDraft = 1 };

// Sine and cosine of the rotary angle delta * freq for |delta| < 2^31, from
// fturn = freq / (2 pi) as a 64-bit binary fraction (the host's
// rope_turn_fixed): delta * fturn modulo 2^64 is the angle in turns modulo
// one, exact in integer arithmetic; its top 32 bits, read as a signed
// fraction of a turn, give the reduced angle in [-pi, pi) in fp32 (about
// 2e-7 rad of rounding), whose sine and cosine come from the hardware
// approximation (absolute error about 2^-21 on [-pi, pi]; the rotated values
// are rounded to bf16, 2^-9 relative).  No double arithmetic on the device:
// GB300's double-precision rate is a small fraction of its fp32 rate.
__device__ __forceinline__ void rope_sincos(long long delta, uint64_t fturn, float* sn,
                                            float* cs) {
    const uint64_t t = (uint64_t)delta * fturn;
    const float a = (float)(int32_t)(uint32_t)(t >> 32) * 1.4629180792671596e-9f;  // 2 pi / 2^32
    __sincosf(a, sn, cs);
}

// Stage flags passed from the producer to the consumers.
enum : int32_t { kFirst = 1, kLast = 2, kBad = 4, kTerm = 8 };

struct AttnParams {
    const __nv_bfloat16* q;    // [B, kp1, Hq, D]
    float* out;                // [B, kp1, Hq, D]
    const int32_t* ctx_lens;   // [B]
    const int32_t* block_table;
    int32_t* header;           // [0]: grid size of the last call
    int32_t* err;              // [kMaxCtas]: error bits of each CTA of the last call
    int32_t* cnt;              // [B * Hkv]: segment arrival counters, zero at launch
    unsigned long long* stamps;  // [2 * kMaxCtas]: per CTA, %globaltimer when its first tile
                                 // starts and when its last merge is done (last call)
    float* part_o;             // [2 * kMaxCtas * R, D]
    float* part_lse;           // [2 * kMaxCtas * R]
    int32_t B, Hq, Hkv, G, kp1, R;
    int32_t max_pages, num_pages;  // verify
    int32_t cap;                   // draft: cache slots S = n_sink + window
    int32_t mode;
    float sl2;                     // softmax_scale * log2(e)
    int32_t head;                  // per-pair fixed cost in tile units (the split's weights)
};

// Tiles of sequence b: ceil(visible length / 64); a sequence whose length
// breaks the rules occupies one pseudo-tile that yields NaN rows.
__device__ __forceinline__ int seq_tiles(const AttnParams& p, int L, int* leff, bool* valid) {
    bool ok;
    int le;
    if (p.mode == kModeVerify) {
        ok = (L >= p.kp1) && ((long long)L <= (long long)p.max_pages * kPage);
        le = L;
    } else {
        ok = L >= 1;
        le = L < p.cap ? L : p.cap;
    }
    *valid = ok;
    *leff = ok ? le : 0;
    return ok ? (le + kPage - 1) / kPage : 1;
}

// CTA whose range holds global tile x (ranges are floor(cW/N) .. floor((c+1)W/N)).
__device__ __forceinline__ int cta_of(long long x, long long W, int N) {
    return (int)(((x + 1) * N + W - 1) / W) - 1;
}

__device__ __forceinline__ long long range_lo(int c, long long W, int N) {
    return W * c / N;
}

struct SchedShared {
    long long W, lo, hi, p0;   // total tiles, this CTA's range, first tile of sequence b0
    long long p1;              // first unit of sequence b1, which holds unit hi - 1
    int b0, b1;
    int N;                     // CTAs with work: min(grid, W), so no range is empty
    int bad_len;               // some ctx_lens entry breaks the rules
    long long warp_sums[32];
};

__device__ __forceinline__ long long block_sum(long long v, SchedShared* sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) sh->warp_sums[warp] = v;
    __syncthreads();
    long long t = 0;
    for (int w = 0; w < nw; ++w) t += sh->warp_sums[w];
    return t;
}

__device__ __forceinline__ long long block_excl_scan(long long v, SchedShared* sh,
                                                     long long* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    long long x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    __syncthreads();
    if (lane == 31) sh->warp_sums[warp] = x;
    __syncthreads();
    long long before = 0, t = 0;
    for (int w = 0; w < nw; ++w) {
        if (w < warp) before += sh->warp_sums[w];
        t += sh->warp_sums[w];
    }
    *total = t;
    return before + x - v;
}

// All threads of the CTA: total work, this CTA's range and the sequence its
// range starts in.  Leaves the results in *sh (valid after the call).
__device__ inline void sched_setup(const AttnParams& p, SchedShared* sh) {
    long long acc = 0;
    int bad = 0;
    for (int b = threadIdx.x; b < p.B; b += blockDim.x) {
        int le;
        bool ok;
        acc += seq_tiles(p, p.ctx_lens[b], &le, &ok) + p.head;
        bad |= !ok;
    }
    const long long units = block_sum(acc, sh);
    const int any_bad = __syncthreads_or(bad);
    const long long W = units * p.Hkv;
    const int N = W < (long long)gridDim.x ? (int)W : (int)gridDim.x;
    const int c = blockIdx.x;
    const long long lo = c < N ? range_lo(c, W, N) : W, hi = c < N ? range_lo(c + 1, W, N) : W;
    if (threadIdx.x == 0) {
        sh->W = W; sh->lo = lo; sh->hi = hi; sh->b0 = 0; sh->p0 = 0; sh->N = N;
        sh->b1 = 0; sh->p1 = 0;
        sh->bad_len = any_bad;
    }
    long long carry = 0;
    for (int base = 0; base < p.B; base += blockDim.x) {
        const int b = base + threadIdx.x;
        int le;
        bool ok;
        const long long U = b < p.B ? seq_tiles(p, p.ctx_lens[b], &le, &ok) + p.head : 0;
        long long chunk;
        const long long P = carry + block_excl_scan(U, sh, &chunk);
        if (b < p.B && lo < hi && P * p.Hkv <= lo && lo < (P + U) * p.Hkv) {
            sh->b0 = b;
            sh->p0 = P * p.Hkv;
        }
        if (b < p.B && lo < hi && P * p.Hkv <= hi - 1 && hi - 1 < (P + U) * p.Hkv) {
            sh->b1 = b;
            sh->p1 = P * p.Hkv;
        }
        carry += chunk;
    }
    __syncthreads();
}

// One tile of work as the producer hands it to the consumers.
struct TileMeta {
    int b, g, key0, leff;      // sequence, KV head, first key of the tile, visible length
    int flags, slot, nseg, first_slot;
};

// Walks the tiles of this CTA's unit range, tracking (b, g, t) incrementally
// and stepping over head units; the segment bookkeeping (slot, number of
// segments, first slot) is computed once per segment.  With tail_first, when
// the range ends inside a pair that continues in the next CTA, that pair's
// segment is walked first and then the rest of the range from its start: the
// pair's two halves are then done near the start of both CTAs, so its merge
// overlaps the remaining work instead of trailing the kernel (used by the
// warp-MMA kernel, whose short draft ranges end in such a merge; measured
// slower for the tcgen05 kernel, whose softmax warps do the merge).  Segments,
// slots and the tiles of each segment are the same in either order.
struct TileWalker {
    long long x, end, lo, W;   // unit of the next tile, end of the current part, range start
    long long rest_end;        // end of the second part (the tail pair's first unit), or -1
    int N;
    int b, g, t, T, leff;      // current sequence / KV head / tile-in-pair, tiles per pair
    bool valid, first;
    int slot, nseg, first_slot;
    int b0;
    long long p0;

    // decode the pair and tile at unit x of sequence b (first unit pb)
    __device__ void seek(const AttnParams& p, long long at, int sb, long long pb) {
        x = at; b = sb; g = 0; t = 0; first = true;
        T = seq_tiles(p, p.ctx_lens[b], &leff, &valid);
        const long long off = x - pb;
        const int U = T + p.head;
        g = (int)(off / U);
        const int u = (int)(off - (long long)g * U);
        if (u < p.head) x += p.head - u;             // a part starting in a pair's head
        else t = u - p.head;
    }

    __device__ void init(const AttnParams& p, const SchedShared& sh, bool tail_first) {
        lo = sh.lo; W = sh.W; N = sh.N; b0 = sh.b0; p0 = sh.p0;
        slot = nseg = first_slot = 0;
        valid = false; T = 1; leff = 0; b = sh.b0; g = 0; t = 0; first = true;
        rest_end = -1;
        x = sh.lo; end = sh.hi;
        if (sh.lo >= sh.hi) return;
        // the pair holding the range's last unit
        int le1;
        bool ok1;
        const int T1 = seq_tiles(p, p.ctx_lens[sh.b1], &le1, &ok1);
        const int U1 = T1 + p.head;
        const long long g1 = (sh.hi - 1 - sh.p1) / U1;
        const long long pstart = sh.p1 + g1 * U1;
        if (tail_first && pstart > sh.lo && sh.hi - 1 - pstart >= p.head && pstart + U1 > sh.hi) {
            seek(p, pstart + p.head, sh.b1, sh.p1);  // the tail pair first
            rest_end = pstart;
        } else {
            seek(p, sh.lo, sh.b0, sh.p0);
        }
    }
    __device__ bool done() const { return x >= end && rest_end < 0; }

    // Fills m for the tile at unit x and advances; returns the tile index
    // within the pair.
    __device__ int next(const AttnParams& p, TileMeta* m) {
        int flags = 0;
        if (first || t == 0) {
            flags |= kFirst;
            // units of this pair's first / last tile and of its head
            const long long ftile = x - t, ltile = ftile + T - 1, pstart = ftile - p.head;
            const int c = blockIdx.x;
            const int c0 = cta_of(ftile, W, N), c1 = cta_of(ltile, W, N);
            slot = (lo >= pstart) ? 2 * c : 2 * c + 1;   // first segment of this CTA?
            nseg = c1 - c0 + 1;
            first_slot = (range_lo(c0, W, N) >= pstart) ? 2 * c0 : 2 * c0 + 1;
        }
        if (x == end - 1 || t == T - 1) flags |= kLast;
        if (!valid) flags |= kBad;
        m->b = b; m->g = g; m->key0 = t * kPage; m->leff = leff;
        m->flags = flags; m->slot = slot; m->nseg = nseg; m->first_slot = first_slot;
        const int tile = t;
        first = false;
        ++x;
        if (++t == T) {                            // next pair: step over its head
            t = 0;
            x += p.head;
            if (++g == p.Hkv) {
                g = 0;
                if (x < end) {
                    ++b;
                    T = seq_tiles(p, p.ctx_lens[b], &leff, &valid);
                }
            }
        }
        if (x >= end && rest_end >= 0) {           // the tail pair is done: the rest
            end = rest_end;
            rest_end = -1;
            seek(p, lo, b0, p0);
        }
        return tile;
    }
};

// Shared-memory layout the producer fills: NST stages of [K tile | V tile]
// (each D/64 boxes of 64 keys x 128 bytes, 128-byte swizzled) and `nqbuf` (1
// or 2) Q buffers of D/64 halves, each half QHALF bytes of 128-byte rows
// holding `qcopies` copies of the pair's R query rows, `qcopy_rows` rows apart.
struct ProducerSmem {
    uint32_t stages;       // shared address of stage 0
    uint32_t q;            // shared address of Q buffer 0
    uint32_t qhalf;        // bytes per 64-column half of a Q buffer
    int4* meta;            // 2 int4 per stage
    uint32_t bar_full, bar_empty, bar_qfull, bar_qempty;
    int qcopies;           // copies of the query rows per Q buffer
    int qcopy_rows;        // rows between consecutive copies
    int nqbuf;             // Q buffers in the ring (1 or 2)
    bool tail_first;       // walk a range's split last pair first (TileWalker)
};

// Pair whose loads the test instantiations (kStall) never issue, set by the
// host before such a launch (spire_test_stall_next_call); one copy per
// translation unit.  The production instantiations never read it.
static __device__ int32_t g_stall_pair = -1;

// Meta word layout: meta[2s] = {b, g, key0, leff}; meta[2s+1] = {flags |
// (qflag << 8), slot, nseg, first_slot} where qflag = 16 | Q buffer when the
// tile starts a segment whose query rows were loaded.
//
// Streams this CTA's tiles; run by one thread.  Returns the error bits it
// found.  The stage ring protocol: wait `empty` (parity ph ^ 1), fill, arrive
// on `full` with the byte count; a tile that must not be read (bad length or
// page) arrives without a copy and carries kBad.  The run ends with a stage
// that carries kTerm.  With kStall (test instantiations only) the producer
// stops before the first tile of pair g_stall_pair, issuing nothing more, so
// the consumers' waits for that tile run out.
template <int D, int NST, bool kStall = false>
__device__ uint32_t produce(const AttnParams& p, const SchedShared& sh, const CUtensorMap* tmap_k,
                            const CUtensorMap* tmap_v, const CUtensorMap* tmap_q,
                            const ProducerSmem& sm) {
    constexpr uint32_t TILE = kPage * D * 2, STAGE = 2 * TILE;
    uint32_t err = sh.bad_len ? kErrCtxLen : 0u;
    prefetch_tensormap(tmap_k);
    prefetch_tensormap(tmap_v);
    prefetch_tensormap(tmap_q);
    const uint64_t pol = policy_evict_first();
    const uint32_t qbytes = (D / 64) * sm.qcopies * p.R * 128;
    const uint32_t qbuf = (D / 64) * sm.qhalf;
    uint32_t st = 0, ph = 0, qs = 0, qph = 0;      // stage ring / Q buffer ring
    uint32_t armed = 0, armed_parity = 0;          // stages with a TMA load issued, and its phase
    uint32_t qarmed = 0, qarmed_parity = 0;
    bool ok = true;
    TileWalker wk;
    wk.init(p, sh, sm.tail_first);
    while (!wk.done()) {
        if (!mbar_wait(sm.bar_empty + 8 * st, ph ^ 1)) { ok = false; break; }
        TileMeta m;
        const int t = wk.next(p, &m);
        if constexpr (kStall) {
            if (m.b * p.Hkv + m.g == g_stall_pair) {
                ok = false;
                break;
            }
        }
        int qflag = 0;
        if ((m.flags & kFirst) && !(m.flags & kBad)) {
            // the pair's query rows r = i*G + hl, one box per 64 columns
            if (!mbar_wait(sm.bar_qempty + 8 * qs, qph ^ 1)) { ok = false; break; }
            mbar_arrive_expect_tx(sm.bar_qfull + 8 * qs, qbytes);
            for (int c = 0; c < sm.qcopies; ++c)
#pragma unroll
                for (int h = 0; h < D / 64; ++h)
                    tma_load_3d(sm.q + qs * qbuf + h * sm.qhalf + c * sm.qcopy_rows * 128, tmap_q,
                                h * 64, m.g * p.G, m.b * p.kp1, sm.bar_qfull + 8 * qs, pol);
            qarmed |= 1u << qs;
            qarmed_parity = (qarmed_parity & ~(1u << qs)) | (qph << qs);
            qflag = 16 | qs;
            if (++qs == (uint32_t)sm.nqbuf) { qs = 0; qph ^= 1; }
        }
        int zk = 0, zv = 0, y = 0;
        if (!(m.flags & kBad)) {
            if (p.mode == kModeVerify) {
                const int page = p.block_table[(long long)m.b * p.max_pages + t];
                if (page < 0 || page >= p.num_pages) {
                    m.flags |= kBad;
                    err |= kErrPageId;
                }
                zk = zv = page * p.Hkv + m.g;
            } else {
                y = m.key0;
                zk = (m.b * 2 + 0) * p.Hkv + m.g;
                zv = (m.b * 2 + 1) * p.Hkv + m.g;
            }
        }
        sm.meta[2 * st] = make_int4(m.b, m.g, m.key0, m.leff);
        sm.meta[2 * st + 1] = make_int4(m.flags | (qflag << 8), m.slot, m.nseg, m.first_slot);
        if (m.flags & kBad) {
            mbar_arrive(sm.bar_full + 8 * st);
        } else {
            const uint32_t dk = sm.stages + st * STAGE, dv = dk + TILE;
            mbar_arrive_expect_tx(sm.bar_full + 8 * st, STAGE);
#pragma unroll
            for (int h = 0; h < D / 64; ++h) {
                tma_load_3d(dk + h * 8192, tmap_k, h * 64, y, zk, sm.bar_full + 8 * st, pol);
                tma_load_3d(dv + h * 8192, tmap_v, h * 64, y, zv, sm.bar_full + 8 * st, pol);
            }
            armed |= 1u << st;
            armed_parity = (armed_parity & ~(1u << st)) | (ph << st);
        }
        if (++st == NST) { st = 0; ph ^= 1; }
    }
    if (ok && mbar_wait(sm.bar_empty + 8 * st, ph ^ 1)) {
        sm.meta[2 * st + 1] = make_int4(kTerm, 0, 0, 0);
        mbar_arrive(sm.bar_full + 8 * st);
    } else {
        // Consumers stopped answering: record it and wait (bounded) for our
        // own copies to land before the CTA's shared memory goes away.
        err |= kErrTimeout;
        for (int s = 0; s < NST; ++s)
            if (armed & (1u << s)) mbar_wait(sm.bar_full + 8 * s, (armed_parity >> s) & 1u);
        for (int s = 0; s < 2; ++s)
            if (qarmed & (1u << s)) mbar_wait(sm.bar_qfull + 8 * s, (qarmed_parity >> s) & 1u);
    }
    return err;
}

// Slot of segment j (0 .. nseg-1) of a pair whose first segment uses first_slot.
__device__ __forceinline__ int segment_slot(int j, int first_slot) {
    return j == 0 ? first_slot : 2 * ((first_slot >> 1) + j);
}

// Output row of query row r (= block row i * G + head-in-group hl) of pair (b, g).
__device__ __forceinline__ float* out_row(const AttnParams& p, int b, int g, int r, int D) {
    const int i = r / p.G, hl = r - i * p.G;
    return p.out + ((long long)(b * p.kp1 + i) * p.Hq + g * p.G + hl) * D;
}

// Merge the nseg partials of pair (b, g) into the output; executed by
// `nthreads` threads with ids 0..nthreads-1.  Partials are read around L1.
// One pass per output float4: a running maximum M of the segments' base-2
// log-sum-exps, with the sum and the weighted partial rescaled whenever M
// grows, so no load waits for another segment's result; each thread handles
// U outputs per round so that their loads are in flight together.
template <int D>
__device__ void merge_pair(const AttnParams& p, int b, int g, int nseg, int first_slot,
                           int tid, int nthreads) {
    constexpr int D4 = D / 4, U = 4;
    const float NEG_INF = __int_as_float(0xff800000);
    const float NANF = __int_as_float(0x7fc00000);
    const int total = p.R * D4;
    for (int base = tid; base < total; base += U * nthreads) {
        float M[U], den[U];
        float4 acc[U];
        bool nan[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            M[u] = NEG_INF;
            den[u] = 0.f;
            acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
            nan[u] = false;
        }
        for (int j = 0; j < nseg; ++j) {
            const long long slot_row = (long long)segment_slot(j, first_slot) * p.R;
            float lse[U];
            float4 v[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int idx = base + u * nthreads;
                if (idx < total) {
                    const int r = idx / D4, d4 = idx - r * D4;
                    lse[u] = __ldcg(p.part_lse + slot_row + r);
                    v[u] = __ldcg(reinterpret_cast<const float4*>(p.part_o + (slot_row + r) * D) + d4);
                }
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                if (base + u * nthreads >= total) continue;
                const float l = lse[u];
                nan[u] |= (l != l);
                if (l > M[u]) {            // rescale what was accumulated so far
                    const float sc = ex2(M[u] - l);   // 0 while M is -inf
                    den[u] *= sc;
                    acc[u].x *= sc; acc[u].y *= sc; acc[u].z *= sc; acc[u].w *= sc;
                    M[u] = l;
                }
                if (l != NEG_INF && !(l != l)) {
                    const float w = ex2(l - M[u]);
                    den[u] += w;
                    acc[u].x += w * v[u].x; acc[u].y += w * v[u].y;
                    acc[u].z += w * v[u].z; acc[u].w += w * v[u].w;
                }
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int idx = base + u * nthreads;
            if (idx >= total) continue;
            const int r = idx / D4, d4 = idx - r * D4;
            float4 res;
            if (nan[u] || !(den[u] > 0.f)) {
                res = make_float4(NANF, NANF, NANF, NANF);
            } else {
                const float inv = 1.f / den[u];
                res = make_float4(acc[u].x * inv, acc[u].y * inv, acc[u].z * inv, acc[u].w * inv);
            }
            *reinterpret_cast<float4*>(out_row(p, b, g, r, D) + 4 * d4) = res;
        }
    }
}

}  // namespace spire
