// Split-kernel instantiations for head_dim 128.
#include "spire_split_inst.cuh"

namespace spire {
cudaError_t launch_split_d128(int mt, const CUtensorMap& tk, const CUtensorMap& tv,
                              const SplitParams& p, int num_sms, cudaStream_t stream) {
    return launch_split_dispatch<128>(mt, tk, tv, p, num_sms, stream);
}
}  // namespace spire
