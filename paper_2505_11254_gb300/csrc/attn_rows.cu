// Sink + window attention with the fused Delta epilogues for row-range calls
// (delta_attn_prefill_rows with a first row above 0): items start at the
// range's first row; a translation unit of its own so it compiles in parallel.
#include "launch_impl.cuh"

namespace da {
template cudaError_t launch_attn<64, MODE_SPARSE, EPI_FUSED_INTILE, true>(const CUtensorMap&, const CUtensorMap&,
                                                                          const CUtensorMap&, const Params&,
                                                                          long long, cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_FUSED_INTILE, true>(const CUtensorMap&, const CUtensorMap&,
                                                                           const CUtensorMap&, const Params&,
                                                                           long long, cudaStream_t);
template cudaError_t launch_attn<64, MODE_SPARSE, EPI_FUSED_DELTA, true>(const CUtensorMap&, const CUtensorMap&,
                                                                         const CUtensorMap&, const Params&,
                                                                         long long, cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_FUSED_DELTA, true>(const CUtensorMap&, const CUtensorMap&,
                                                                          const CUtensorMap&, const Params&,
                                                                          long long, cudaStream_t);
}  // namespace da
