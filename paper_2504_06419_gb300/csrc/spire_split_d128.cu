// Attention-kernel instantiations for head_dim 128.
#include "spire_split_inst.cuh"

namespace spire {
cudaError_t launch_attn_d128(int mt, const CUtensorMap& tk, const CUtensorMap& tv,
                            const CUtensorMap& tq, const AttnParams& p, int ctas,
                            cudaStream_t stream) {
    return launch_attn_dispatch<128>(mt, tk, tv, tq, p, ctas, stream);
}
cudaError_t launch_attn_tc_d128(int nc, const CUtensorMap& tk, const CUtensorMap& tv,
                               const CUtensorMap& tq, const AttnParams& p, int ctas,
                               cudaStream_t stream) {
    return launch_tc_dispatch<128>(nc, tk, tv, tq, p, ctas, stream);
}
cudaError_t launch_stall_d128(bool tc, int nc, int32_t pair, const CUtensorMap& tk,
                              const CUtensorMap& tv, const CUtensorMap& tq, const AttnParams& p,
                              int ctas, cudaStream_t stream) {
    return launch_stall_dispatch<128>(tc, nc, pair, tk, tv, tq, p, ctas, stream);
}
}  // namespace spire
