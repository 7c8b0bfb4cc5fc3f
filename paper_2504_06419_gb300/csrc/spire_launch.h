// spire_launch.h -- host-side launchers of the split kernel instantiations
// (one translation unit per head_dim so they compile in parallel).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include "spire_mma.cuh"
#include "spire_tc.cuh"

namespace spire {

// Launch the warp-MMA attention kernel for head_dim D with MT m-tiles (16
// query rows each; only MT = 1 is built) on a grid of `ctas` persistent CTAs.
// Returns the launch error, or cudaErrorInvalidValue for an unsupported MT.
cudaError_t launch_attn_d64(int mt, const CUtensorMap& tk, const CUtensorMap& tv,
                            const CUtensorMap& tq, const AttnParams& p, int ctas,
                            cudaStream_t stream);
cudaError_t launch_attn_d128(int mt, const CUtensorMap& tk, const CUtensorMap& tv,
                             const CUtensorMap& tq, const AttnParams& p, int ctas,
                             cudaStream_t stream);

// tcgen05 kernel (any R <= 128): one CTA per SM; nc = copies of the query
// rows (4 for R <= 32, 2 for R <= 64, else 1).
cudaError_t launch_attn_tc_d64(int nc, const CUtensorMap& tk, const CUtensorMap& tv,
                               const CUtensorMap& tq, const AttnParams& p, int ctas,
                               cudaStream_t stream);
cudaError_t launch_attn_tc_d128(int nc, const CUtensorMap& tk, const CUtensorMap& tv,
                                const CUtensorMap& tq, const AttnParams& p, int ctas,
                                cudaStream_t stream);

// Test instantiations at head_dim 128 (spire_test_stall_next_call): the
// warp-MMA kernel (tc = false) or the tcgen05 kernel with nc copies, whose
// producer issues nothing from pair `pair` on.
cudaError_t launch_stall_d128(bool tc, int nc, int32_t pair, const CUtensorMap& tk,
                              const CUtensorMap& tv, const CUtensorMap& tq, const AttnParams& p,
                              int ctas, cudaStream_t stream);

// Largest dynamic shared memory one block of this build may use (227 KB).
constexpr int kMaxDynSmem = 232448;

// Key slices per m-tile: enough consumer warps to keep the tensor pipes and
// the softmax busy, each warp still owning >= 16 keys of a tile (measured on
// GB300: 4 slices for one m-tile, 2 for two or three).  The register
// file is split across the SM's four sub-partitions, so a block of 9+ warps
// gets at most 168 registers per thread; from MT = 3 on, one slice per
// m-tile keeps the block at <= 8 warps.
constexpr int key_parts(int mt) { return mt <= 1 ? 4 : (mt <= 3 ? 2 : 1); }

// Deepest stage ring that fits next to the merge scratch.
template <int D, int MT>
constexpr int stages() {
    constexpr int kp = key_parts(MT);
    constexpr int nw = MT * kp;
    constexpr int qbuf = 2 * (D / 64) * MT * 16 * 128;
    constexpr int fixed = 2 * nw * 8 * (D + 8) * 4 +
                          ((2 * nw * 8 * 8 + 2 * 32 + 1023) / 1024) * 1024 + qbuf + 8 * 32 + 512 +
                          (2 * 8 + 9) * 8 + 1024;
    constexpr int stage = 2 * 64 * D * 2;
    constexpr int n = (kMaxDynSmem - fixed) / stage;
    return n > 8 ? 8 : n;
}

// Deepest stage ring of the tcgen05 kernel next to its Q buffer and the
// copy-merge scratch: a stage costs its K and V tiles, 32 bytes of tile
// metadata and three mbarriers.
template <int D, int NC>
constexpr int tc_stages() {
    constexpr int fixed = TcCfg<D, NC, 0>::SMEM;
    constexpr int n = (kMaxDynSmem - fixed) / (2 * 64 * D * 2 + 32 + 3 * 8);
    return n > 6 ? 6 : n;
}

}  // namespace spire
