// launch_impl.cuh — the launcher template; included by the attn_*.cu units.
#pragma once
#include "attn_kernel.cuh"
#include "launch.h"

namespace da {

template <int D, int MODE, int EPI>
cudaError_t launch_attn(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv, const Params& p,
                        long long grid, cudaStream_t s) {
  auto kfn = attn_kernel<D, MODE, EPI>;
  cudaError_t e = cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<D>::SMEM);
  if (e != cudaSuccess) return e;
  if (grid <= 0) return cudaSuccess;
  kfn<<<(unsigned)grid, kThreads, Cfg<D>::SMEM, s>>>(tq, tk, tv, p);
  return cudaGetLastError();
}

}  // namespace da
