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

// 2-D bf16 tensor map {inner, outer} (row stride inner * 2 bytes) read in
// box_inner x box_outer boxes with 128-byte swizzle.
bool encode_2d_bf16_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                        uint32_t box_inner, uint32_t box_outer);

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

}  // namespace spire
