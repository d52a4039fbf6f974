// Two-CTA sink + window attention (MODE_SPARSE, d = 128, G even) with its epilogues.
#include "launch_impl.cuh"

namespace da {
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_BF16, false, true>(const CUtensorMap&, const CUtensorMap&,
                                                                   const CUtensorMap&, const Params&, long long,
                                                                   cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_FUSED_INTILE, false, true>(const CUtensorMap&,
                                                                           const CUtensorMap&, const CUtensorMap&,
                                                                           const Params&, long long, cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_FUSED_DELTA, false, true>(const CUtensorMap&,
                                                                          const CUtensorMap&, const CUtensorMap&,
                                                                          const Params&, long long, cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_FUSED_SMOOTH, false, true>(const CUtensorMap&,
                                                                           const CUtensorMap&, const CUtensorMap&,
                                                                           const Params&, long long, cudaStream_t);
}  // namespace da
