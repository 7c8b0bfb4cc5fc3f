// spire_split_inst.cuh -- instantiates and launches the attention kernel for one
// head_dim; included by spire_split_d64.cu / spire_split_d128.cu.
#pragma once

#include <atomic>

#include "spire_launch.h"

namespace spire {

// Launch with programmatic stream serialisation: the kernel may start while
// the counter-zeroing kernel before it finishes, and waits for it
// (griddepcontrol.wait) before touching the counters.
template <typename Kern>
cudaError_t launch_pdl(Kern kern, int ctas, int threads, int smem, cudaStream_t stream,
                       const CUtensorMap& tk, const CUtensorMap& tv, const CUtensorMap& tq,
                       const AttnParams& p) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(ctas);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, tk, tv, tq, p);
}

template <int D, int MT, bool kStall = false>
cudaError_t launch_attn_t(const CUtensorMap& tk, const CUtensorMap& tv, const CUtensorMap& tq,
                          const AttnParams& p, int ctas, cudaStream_t stream) {
    constexpr int KP = key_parts(MT);
    constexpr int NST = stages<D, MT>();
    static_assert(NST >= 2, "stage ring does not fit in shared memory");
    using C = MmaCfg<D, MT, KP, NST>;
    static_assert(C::SMEM <= kMaxDynSmem, "shared memory budget exceeded");
    auto kern = attn_mma_kernel<D, MT, KP, NST, kStall>;
    // the shared-memory opt-in is per device; remember it for the first 64
    static std::atomic<unsigned long long> done{0ull};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = dev < 64 ? (1ull << dev) : 0ull;
    if (!bit || !(done.load(std::memory_order_acquire) & bit)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (e != cudaSuccess) return e;
        done.fetch_or(bit, std::memory_order_acq_rel);
    }
    // one CTA per SM: the stage ring takes most of the shared memory
    return launch_pdl(kern, ctas, C::THREADS, C::SMEM, stream, tk, tv, tq, p);
}

template <int D, int NC, bool kStall = false>
cudaError_t launch_tc_t(const CUtensorMap& tk, const CUtensorMap& tv, const CUtensorMap& tq,
                        const AttnParams& p, int ctas, cudaStream_t stream) {
    constexpr int NST = tc_stages<D, NC>();
    static_assert(NST >= 2, "stage ring does not fit in shared memory");
    using C = TcCfg<D, NC, NST>;
    static_assert(C::SMEM <= kMaxDynSmem, "shared memory budget exceeded");
    auto kern = attn_tc_kernel<D, NC, NST, kStall>;
    static std::atomic<unsigned long long> done{0ull};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = dev < 64 ? (1ull << dev) : 0ull;
    if (!bit || !(done.load(std::memory_order_acquire) & bit)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (e != cudaSuccess) return e;
        done.fetch_or(bit, std::memory_order_acq_rel);
    }
    return launch_pdl(kern, ctas, C::THREADS, C::SMEM, stream, tk, tv, tq, p);
}

template <int D>
cudaError_t launch_tc_dispatch(int nc, const CUtensorMap& tk, const CUtensorMap& tv,
                               const CUtensorMap& tq, const AttnParams& p, int ctas,
                               cudaStream_t stream) {
    switch (nc) {
        case 4: return launch_tc_t<D, 4>(tk, tv, tq, p, ctas, stream);
        case 2: return launch_tc_t<D, 2>(tk, tv, tq, p, ctas, stream);
        case 1: return launch_tc_t<D, 1>(tk, tv, tq, p, ctas, stream);
        default: return cudaErrorInvalidValue;
    }
}

// Test instantiations (spire_test_stall_next_call): the same kernels with
// kStall, after the host has set this unit's g_stall_pair.
template <int D>
cudaError_t launch_stall_dispatch(bool tc, int nc, int32_t pair, const CUtensorMap& tk,
                                  const CUtensorMap& tv, const CUtensorMap& tq,
                                  const AttnParams& p, int ctas, cudaStream_t stream) {
    cudaError_t e = cudaMemcpyToSymbolAsync(g_stall_pair, &pair, sizeof(pair), 0,
                                            cudaMemcpyHostToDevice, stream);
    if (e != cudaSuccess) return e;
    if (!tc) return launch_attn_t<D, 1, true>(tk, tv, tq, p, ctas, stream);
    switch (nc) {
        case 4: return launch_tc_t<D, 4, true>(tk, tv, tq, p, ctas, stream);
        case 2: return launch_tc_t<D, 2, true>(tk, tv, tq, p, ctas, stream);
        case 1: return launch_tc_t<D, 1, true>(tk, tv, tq, p, ctas, stream);
        default: return cudaErrorInvalidValue;
    }
}

template <int D>
cudaError_t launch_attn_dispatch(int mt, const CUtensorMap& tk, const CUtensorMap& tv,
                                 const CUtensorMap& tq, const AttnParams& p, int ctas,
                                 cudaStream_t stream) {
    // the library sends only pairs of at most 16 query rows (one m-tile) here
    if (mt != 1) return cudaErrorInvalidValue;
    return launch_attn_t<D, 1>(tk, tv, tq, p, ctas, stream);
}

}  // namespace spire
