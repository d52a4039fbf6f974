// rope.cu — RoPE, the positional encoding applied to Q and K before the
// attention (Sec. 2), in the rotate-half form: for c < d/2 the pair
// (x_c, x_{c+d/2}) at position pos turns by the angle pos * base^(-2c/d).
//   * rope_table_kernel: the (cos, sin) table [n_pos][d/2] in fp32, from
//     angles and sines taken in double (the angle reaches 1e6 rad at 1M
//     positions; single precision would lose it);
//   * rope_apply_kernel: rotates bf16 rows in place (K before the prefill, a
//     decode query at its position): HBM-bound, 16-byte coalesced accesses,
//     fp32 arithmetic, one rounding to bf16.
// Q is not rotated here: the attention kernels rotate each Q tile in shared
// memory before its first QK (epilogue warps, rotate_q), saving a read and a
// write of Q.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "launch.h"

namespace da {

__global__ void __launch_bounds__(256) rope_table_kernel(long long n_pos, int d, double base, float2* table) {
  const int h = d / 2;
  const long long total = n_pos * h;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const long long pos = t / h;
    const int c = (int)(t % h);
    const double a = (double)pos * pow(base, -2.0 * (double)c / (double)d);
    double sn, cs;
    sincos(a, &sn, &cs);
    table[t] = make_float2((float)cs, (float)sn);
  }
}

// One thread per (position, 8 pairs): channels c..c+7 and c+d/2..c+d/2+7 of
// every row at that position.  x holds rows/N slabs of N rows (one per
// batch and head) and slab row i is at position pos0 + i, so the thread reads
// its 64 bytes of the table once and rotates the same channels of every slab
// (a thread per row re-read the table once per slab: 2.3x the bytes of x at
// 8 KV heads).
__global__ void __launch_bounds__(256) rope_apply_kernel(__nv_bfloat16* x, long long rows, long long N, int d,
                                                         long long pos0, const float2* __restrict__ table) {
  const int h = d / 2, groups = h / 8;
  const long long total = N * groups;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const long long i = t / groups;
    const int c0 = (int)(t % groups) * 8;
    const float4* tb = reinterpret_cast<const float4*>(table + (pos0 + i) * h + c0);
    float4 cs[4];  // (cos, sin) of channels c0 + 2e and c0 + 2e + 1
#pragma unroll
    for (int e = 0; e < 4; ++e) cs[e] = tb[e];
    for (long long r = i; r < rows; r += N) {
      __nv_bfloat16* lo = x + r * d + c0;
      __nv_bfloat16* hi = lo + h;
      uint4 ul = *reinterpret_cast<const uint4*>(lo);
      uint4 uh = *reinterpret_cast<const uint4*>(hi);
      __nv_bfloat162* pl = reinterpret_cast<__nv_bfloat162*>(&ul);
      __nv_bfloat162* ph = reinterpret_cast<__nv_bfloat162*>(&uh);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 a = __bfloat1622float2(pl[e]);
        const float2 b = __bfloat1622float2(ph[e]);
        pl[e] = __floats2bfloat162_rn(a.x * cs[e].x - b.x * cs[e].y, a.y * cs[e].z - b.y * cs[e].w);
        ph[e] = __floats2bfloat162_rn(b.x * cs[e].x + a.x * cs[e].y, b.y * cs[e].z + a.y * cs[e].w);
      }
      *reinterpret_cast<uint4*>(lo) = ul;
      *reinterpret_cast<uint4*>(hi) = uh;
    }
  }
}

cudaError_t launch_rope_table(long long n_pos, int d, double base, float* table, cudaStream_t s) {
  const long long total = n_pos * (d / 2);
  const long long blocks = (total + 255) / 256 < 152LL * 16 ? (total + 255) / 256 : 152LL * 16;
  rope_table_kernel<<<(unsigned)blocks, 256, 0, s>>>(n_pos, d, base, reinterpret_cast<float2*>(table));
  return cudaGetLastError();
}

cudaError_t launch_rope_apply(void* x, long long rows, long long N, int d, long long pos0, const float* table,
                              cudaStream_t s) {
  const long long total = N * (d / 16);
  const long long blocks = (total + 255) / 256 < 152LL * 32 ? (total + 255) / 256 : 152LL * 32;
  rope_apply_kernel<<<(unsigned)blocks, 256, 0, s>>>(static_cast<__nv_bfloat16*>(x), rows, N, d, pos0,
                                                      reinterpret_cast<const float2*>(table));
  return cudaGetLastError();
}

}  // namespace da
