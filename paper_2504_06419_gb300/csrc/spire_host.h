// spire_host.h -- host helpers shared by the translation units of libspire
// (defined in spire_abi.cu).
#pragma once

#include <cstdint>

#include <cuda.h>
#include <cuda_runtime.h>

#include "spire.h"

namespace spire {

// True if p is a multiple of a bytes.
bool host_aligned(const void* p, uintptr_t a);

// SM count and opt-in shared memory per block of the current device (cached).
spire_status host_device_info(int* sms, int* smem_optin);

// 3-D bf16 tensor map {inner, mid, outer} (dense, row stride inner * 2 bytes)
// read in box_inner x box_mid x box_outer boxes with 128-byte swizzle.
bool encode_3d_bf16_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t mid,
                        uint64_t outer, uint32_t box_inner, uint32_t box_mid, uint32_t box_outer);

// 2-D bf16 tensor map {inner, outer} (row stride inner * 2 bytes) read in
// box_inner x box_outer boxes with 128-byte swizzle.
bool encode_2d_bf16_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                        uint32_t box_inner, uint32_t box_outer);

// freq / (2 pi) as a 64-bit binary fraction, rounded to nearest (0 <= freq
// <= 1): the device's rope_sincos turns it into the angle modulo 2 pi for any
// integer position.  Double and fma only, so every host computes the same bits.
uint64_t rope_turn_fixed(double freq);

// Launch a kernel with programmatic dependent launch: it may start while the
// kernel before it in the stream runs (after that kernel's blocks have all
// called griddepcontrol.launch_dependents or exited); the launched kernel
// must execute griddepcontrol.wait before it reads anything that kernel wrote.
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t stream, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

// As launch_dependent, for a kernel launched in clusters of cluster_x CTAs
// along x (the grid's x extent a multiple of cluster_x).
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent_cluster(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                     cudaStream_t stream, unsigned cluster_x, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = cluster_x;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

}  // namespace spire
