// launch_impl.cuh — the launcher template; included by the attn_*.cu units.
#pragma once
#include <atomic>

#include "attn_kernel.cuh"
#include "launch.h"

namespace da {

constexpr int kMaxDevices = 64;

// Persistent launch: min(items, SMs) CTAs, each walking items with a stride
// of the grid size.  The two-CTA kernel runs in clusters of two, as many as
// fit at once (a cluster's CTAs share a GPC), and an even grid; it returns
// cudaErrorNotSupported, launching nothing, where no cluster of two fits.
template <int D, int MODE, int EPI, bool ROWS, bool PAIR>
cudaError_t launch_attn(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv, const Params& p,
                        long long n_items, cudaStream_t s) {
  using C = Cfg<D, MODE, PAIR>;
  auto kfn = attn_kernel<D, MODE, EPI, ROWS, PAIR>;
  cudaError_t e = cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  if (e != cudaSuccess) return e;
  if (n_items <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  Params q = p;
  q.n_items = n_items;
  if (!PAIR) {
    const long long grid = n_items < sms ? n_items : sms;
    kfn<<<(unsigned)grid, kThreads, C::SMEM, s>>>(tq, tk, tv, q);
    return cudaGetLastError();
  }
  if (n_items % 2 != 0) return cudaErrorInvalidValue;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3((unsigned)(2 * (sms / 2)));
  // Clusters that fit at once: a property of the device and this instance,
  // asked once per device (racing first calls compute the same value; -1:
  // none fit).  When none fit the caller takes the one-CTA kernel.
  static std::atomic<int> fit[kMaxDevices];
  int clusters = dev < kMaxDevices ? fit[dev].load(std::memory_order_relaxed) : 0;
  if (clusters == 0) {
    if ((e = cudaOccupancyMaxActiveClusters(&clusters, kfn, &cfg)) != cudaSuccess) return e;
    if (clusters < 1) clusters = -1;
    if (dev < kMaxDevices) fit[dev].store(clusters, std::memory_order_relaxed);
  }
  if (clusters < 1) return cudaErrorNotSupported;
  long long grid = 2LL * clusters;
  if (grid > n_items) grid = n_items;
  cfg.gridDim = dim3((unsigned)grid);
  if ((e = cudaLaunchKernelEx(&cfg, kfn, tq, tk, tv, q)) != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace da
