// aux.cu — the standalone Delta application (Eq. 6 as a separate pass) and the
// debug kernels that dump the visibility predicate, the row -> sample map and
// the work decomposition the attention kernels use.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "launch.h"
#include "tiles.cuh"
#include "wait.cuh"

namespace da {

__device__ __forceinline__ void ld_bf16x8(const __nv_bfloat16* src, float* v) {
  uint4 u = *reinterpret_cast<const uint4*>(src);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    float2 f = __bfloat1622float2(h[e]);
    v[2 * e] = f.x;
    v[2 * e + 1] = f.y;
  }
}

__device__ __forceinline__ void st_bf16x8(__nv_bfloat16* dst, const float* v) {
  uint4 u;
  __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
  for (int e = 0; e < 4; ++e) h[e] = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
  *reinterpret_cast<uint4*>(dst) = u;
}

// One thread per (head, sample k, 8-column slice): it reads the sparse row of
// the sample first and then walks the gamma rows of the group in order, so the
// output may alias the sparse input.
//   sampled row  k*gamma: O = bf16(D_k)
//   other rows   i      : O = bf16(S_i + D_k - S_{k gamma})
__global__ void __launch_bounds__(256) delta_apply_kernel(const __nv_bfloat16* osp, const float* ss, const float* ds,
                                                          __nv_bfloat16* o, long long BH, long long N, int d,
                                                          int gamma, long long n_s) {
  const int cpr = d / 8;
  const long long total = BH * n_s * cpr;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
       idx += (long long)gridDim.x * blockDim.x) {
    const int c8 = (int)(idx % cpr);
    const long long rest = idx / cpr;
    const long long k = rest % n_s;
    const long long bh = rest / n_s;
    const long long i0 = k * gamma;
    float dk[8], sk[8];
    const float* dp = ds + (bh * n_s + k) * d + c8 * 8;
#pragma unroll
    for (int e = 0; e < 8; ++e) dk[e] = dp[e];
    if (ss != nullptr) {
      const float* sp = ss + (bh * n_s + k) * d + c8 * 8;
#pragma unroll
      for (int e = 0; e < 8; ++e) sk[e] = sp[e];
    } else {
      ld_bf16x8(osp + (bh * N + i0) * d + c8 * 8, sk);
    }
    st_bf16x8(o + (bh * N + i0) * d + c8 * 8, dk);
    const long long i_end = lmin(i0 + gamma, N);
    for (long long i = i0 + 1; i < i_end; ++i) {
      float x[8];
      ld_bf16x8(osp + (bh * N + i) * d + c8 * 8, x);
#pragma unroll
      for (int e = 0; e < 8; ++e) x[e] = x[e] + (dk[e] - sk[e]);
      st_bf16x8(o + (bh * N + i) * d + c8 * 8, x);
    }
  }
}

cudaError_t launch_delta_apply(const void* o_sparse, const float* s_sampled, const float* d_sampled, void* o, int B,
                               int Hq, long long N, int d, int gamma, cudaStream_t s) {
  const long long n_s = cdiv(N, gamma);
  const long long total = (long long)B * Hq * n_s * (d / 8);
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  long long blocks = lmin(cdiv(total, 256), (long long)sms * 16);
  if (blocks < 1) blocks = 1;
  delta_apply_kernel<<<(unsigned)blocks, 256, 0, s>>>(
      static_cast<const __nv_bfloat16*>(o_sparse), s_sampled, d_sampled, static_cast<__nv_bfloat16*>(o),
      (long long)B * Hq, N, d, gamma, n_s);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ debug
__global__ void debug_mask_kernel(long long N, int n_sink, long long window, long long i0, long long i1,
                                  unsigned char* out) {
  const long long total = (i1 - i0) * N;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
       idx += (long long)gridDim.x * blockDim.x) {
    const long long i = i0 + idx / N, j = idx % N;
    out[idx] = visible_sparse(i, j, n_sink, window) ? 1 : 0;
  }
}

cudaError_t launch_debug_mask(long long N, int n_sink, long long window, long long i0, long long i1,
                              unsigned char* out, cudaStream_t s) {
  const long long total = (i1 - i0) * N;
  const long long blocks = lmax(1, lmin(cdiv(total, 256), 4096));
  debug_mask_kernel<<<(unsigned)blocks, 256, 0, s>>>(N, n_sink, window, i0, i1, out);
  return cudaGetLastError();
}

__global__ void debug_rowmap_kernel(long long N, int gamma, long long* sample_row, unsigned char* sampled) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < N; i += (long long)gridDim.x * blockDim.x) {
    sample_row[i] = sample_of_row(i, gamma);
    sampled[i] = is_sampled_row(i, gamma) ? 1 : 0;
  }
}

cudaError_t launch_debug_rowmap(long long N, int gamma, long long* sample_row, unsigned char* sampled,
                                cudaStream_t s) {
  const long long blocks = lmax(1, lmin(cdiv(N, 256), 4096));
  debug_rowmap_kernel<<<(unsigned)blocks, 256, 0, s>>>(N, gamma, sample_row, sampled);
  return cudaGetLastError();
}

// Layout of `out`: [0..15] work header, [16 + 4*t] lane t: row, sample, head,
// valid; [16 + 512 + 2*j] key tile j: tile index, needs-mask.
template <int MODE>
__device__ void debug_work_body(const Params& p, long long index, long long* out, int max_tiles) {
  const Work w = decode_work<MODE>(p, index);
  const int t = threadIdx.x;
  if (t == 0) {
    long long h[16] = {w.b, w.h0, w.g, w.r0, w.r_last, w.n_sink_tiles, w.kt_lo, w.kt_hi,
                       w.T, w.n_chunks, w.chunk_idx, w.u0, w.unit, w.gi, w.t, p.order};
    for (int e = 0; e < 16; ++e) out[e] = h[e];
  }
  if (t < BM) {
    long long row, sample;
    int head;
    const bool ok = lane_row<MODE>(p, w, t, row, sample, head);
    out[16 + 4 * t + 0] = row;
    out[16 + 4 * t + 1] = sample;
    out[16 + 4 * t + 2] = head;
    out[16 + 4 * t + 3] = ok ? 1 : 0;
  }
  for (int j = t; j < w.T && j < max_tiles; j += blockDim.x) {
    out[16 + 4 * BM + 2 * j] = tile_index(w, j);
    out[16 + 4 * BM + 2 * j + 1] = tile_needs_mask<MODE>(p, w, j) ? 1 : 0;
  }
}

__global__ void debug_work_kernel(int mode, Params p, long long index, long long* out, int max_tiles) {
  if (mode == MODE_SPARSE)
    debug_work_body<MODE_SPARSE>(p, index, out, max_tiles);
  else if (mode == MODE_STRIDED_DENSE)
    debug_work_body<MODE_STRIDED_DENSE>(p, index, out, max_tiles);
  else
    debug_work_body<MODE_STRIDED_SPARSE>(p, index, out, max_tiles);
}

cudaError_t launch_debug_work(int mode, const Params& p, long long index, long long* out, int max_tiles,
                              cudaStream_t s) {
  debug_work_kernel<<<1, BM, 0, s>>>(mode, p, index, out, max_tiles);
  return cudaGetLastError();
}

// A wait on an mbarrier that nothing ever arrives on: the bounded wait must
// give up after limit_ns, record DA_ERR_TIMEOUT and let the kernel return.
__global__ void debug_timeout_kernel(int* status, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ volatile int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) wait_bounded(&bar, 0, &abort_flag, status, limit_ns);
}

cudaError_t launch_debug_timeout(int* status, unsigned long long limit_ns, cudaStream_t s) {
  debug_timeout_kernel<<<1, 32, 0, s>>>(status, limit_ns);
  return cudaGetLastError();
}

}  // namespace da
