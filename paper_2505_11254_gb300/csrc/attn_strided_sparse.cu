// Sink + window attention at the sampled rows (MODE_STRIDED_SPARSE), building
// Delta_k = D_k - S_{k gamma} when gamma does not divide the 128-row tile.
#include "launch_impl.cuh"

namespace da {
template cudaError_t launch_attn<64, MODE_STRIDED_SPARSE, EPI_DELTA_BUILD, false>(const CUtensorMap&, const CUtensorMap&,
                                                                           const CUtensorMap&, const Params&,
                                                                           long long, cudaStream_t);
template cudaError_t launch_attn<128, MODE_STRIDED_SPARSE, EPI_DELTA_BUILD, false>(const CUtensorMap&,
                                                                            const CUtensorMap&,
                                                                            const CUtensorMap&, const Params&,
                                                                            long long, cudaStream_t);
}  // namespace da
