// Dense causal attention of the sampled rows (MODE_STRIDED_DENSE), split-K.
#include "launch_impl.cuh"

namespace da {
template cudaError_t launch_attn<64, MODE_STRIDED_DENSE, EPI_DENSE_F32, false>(const CUtensorMap&, const CUtensorMap&,
                                                                        const CUtensorMap&, const Params&,
                                                                        long long, cudaStream_t);
template cudaError_t launch_attn<128, MODE_STRIDED_DENSE, EPI_DENSE_F32, false>(const CUtensorMap&, const CUtensorMap&,
                                                                         const CUtensorMap&, const Params&,
                                                                         long long, cudaStream_t);
template cudaError_t launch_attn<64, MODE_STRIDED_DENSE, EPI_DENSE_BF16, false>(const CUtensorMap&, const CUtensorMap&,
                                                                         const CUtensorMap&, const Params&,
                                                                         long long, cudaStream_t);
template cudaError_t launch_attn<128, MODE_STRIDED_DENSE, EPI_DENSE_BF16, false>(const CUtensorMap&, const CUtensorMap&,
                                                                          const CUtensorMap&, const Params&,
                                                                          long long, cudaStream_t);
}  // namespace da
