// Sink + window attention over every row with the smoothed-Delta epilogue
// (appendix "Interpolation"); a translation unit of its own so it compiles in
// parallel with the others.
#include "launch_impl.cuh"

namespace da {
template cudaError_t launch_attn<64, MODE_SPARSE, EPI_FUSED_SMOOTH, false>(const CUtensorMap&, const CUtensorMap&,
                                                                    const CUtensorMap&, const Params&, long long,
                                                                    cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_FUSED_SMOOTH, false>(const CUtensorMap&, const CUtensorMap&,
                                                                     const CUtensorMap&, const Params&, long long,
                                                                     cudaStream_t);
}  // namespace da
