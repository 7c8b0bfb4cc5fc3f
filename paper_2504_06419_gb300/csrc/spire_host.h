// spire_host.h -- host helpers shared by the translation units of libspire
// (defined in spire_abi.cu).
#pragma once

#include <cstdint>

#include <cuda.h>

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

}  // namespace spire
