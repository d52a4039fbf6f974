// Sink + window attention over every row (MODE_SPARSE) with its epilogues.
#include "launch_impl.cuh"

namespace da {
template cudaError_t launch_attn<64, MODE_SPARSE, EPI_BF16, false>(const CUtensorMap&, const CUtensorMap&,
                                                            const CUtensorMap&, const Params&, long long,
                                                            cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_BF16, false>(const CUtensorMap&, const CUtensorMap&,
                                                             const CUtensorMap&, const Params&, long long,
                                                             cudaStream_t);
template cudaError_t launch_attn<64, MODE_SPARSE, EPI_FUSED_INTILE, false>(const CUtensorMap&, const CUtensorMap&,
                                                                    const CUtensorMap&, const Params&, long long,
                                                                    cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_FUSED_INTILE, false>(const CUtensorMap&, const CUtensorMap&,
                                                                     const CUtensorMap&, const Params&, long long,
                                                                     cudaStream_t);
template cudaError_t launch_attn<64, MODE_SPARSE, EPI_FUSED_DELTA, false>(const CUtensorMap&, const CUtensorMap&,
                                                                   const CUtensorMap&, const Params&, long long,
                                                                   cudaStream_t);
template cudaError_t launch_attn<128, MODE_SPARSE, EPI_FUSED_DELTA, false>(const CUtensorMap&, const CUtensorMap&,
                                                                    const CUtensorMap&, const Params&, long long,
                                                                    cudaStream_t);
unsigned attn_smem_bytes(int d) { return d == 64 ? Cfg<64>::SMEM : Cfg<128>::SMEM; }
}  // namespace da
