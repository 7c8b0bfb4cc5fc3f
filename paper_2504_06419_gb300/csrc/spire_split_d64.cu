// Attention-kernel instantiations for head_dim 64.
#include "spire_split_inst.cuh"

namespace spire {
cudaError_t launch_attn_d64(int mt, const CUtensorMap& tk, const CUtensorMap& tv,
                            const CUtensorMap& tq, const AttnParams& p, int ctas,
                            cudaStream_t stream) {
    return launch_attn_dispatch<64>(mt, tk, tv, tq, p, ctas, stream);
}
cudaError_t launch_attn_tc_d64(int nc, const CUtensorMap& tk, const CUtensorMap& tv,
                               const CUtensorMap& tq, const AttnParams& p, int ctas,
                               cudaStream_t stream) {
    return launch_tc_dispatch<64>(nc, tk, tv, tq, p, ctas, stream);
}
}  // namespace spire
