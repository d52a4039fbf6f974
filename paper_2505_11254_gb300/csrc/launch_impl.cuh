// launch_impl.cuh — the launcher template; included by the attn_*.cu units.
#pragma once
#include "attn_kernel.cuh"
#include "launch.h"

namespace da {

// Persistent launch: min(items, SMs) CTAs, each walking items with a stride
// of the grid size.
template <int D, int MODE, int EPI, bool ROWS>
cudaError_t launch_attn(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv, const Params& p,
                        long long n_items, cudaStream_t s) {
  auto kfn = attn_kernel<D, MODE, EPI, ROWS>;
  cudaError_t e = cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<D, MODE>::SMEM);
  if (e != cudaSuccess) return e;
  if (n_items <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  Params q = p;
  q.n_items = n_items;
  const long long grid = n_items < sms ? n_items : sms;
  kfn<<<(unsigned)grid, kThreads, Cfg<D, MODE>::SMEM, s>>>(tq, tk, tv, q);
  return cudaGetLastError();
}

}  // namespace da
