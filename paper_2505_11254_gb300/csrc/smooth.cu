// smooth.cu — Delta smoothing (appendix "Interpolation", Alg. 2), run between
// the Delta build and the sink+window pass.  It turns the Delta rows into
// per-sample basis vectors and a per-offset coefficient table, so that the
// sink+window epilogue adds to row i = k*gamma + r the correction
//   coef[r][0] * basis_k[0] + coef[r][1] * basis_k[1]:
//   linear interpolation  basis (Delta_k, Delta_{k+1}; the last sample repeats
//                         itself), coef (1 - r/gamma, r/gamma);
//   EMA over the rows     e_0 = Delta_0, e_i = (1 - beta) e_{i-1} + beta Delta_{floor(i/gamma)}:
//                         within a group the rows are an affine function of the
//                         value e carried in from the previous group, so basis
//                         (e_{k gamma - 1}, Delta_k) with e_{-1} := Delta_0, coef
//                         ((1-beta)^(r+1), 1 - (1-beta)^(r+1)); the carry of the
//                         next group is rho e + (1 - rho) Delta_k, rho = (1-beta)^gamma;
//   alpha-beta-gamma      Alg. 2 over the Delta vectors (position, velocity and
//   filter                acceleration; predict, take the residual, correct by
//                         alpha, beta, gamma), basis (o_k, 0), coef (1, 0).
#include <cuda_runtime.h>

#include <cmath>

#include "launch.h"
#include "tiles.cuh"

namespace da {

// The recurrences over the samples k are linear and time-invariant:
//   EMA carry   c_{k+1} = rho c_k + (1 - rho) Delta_k, c_0 = Delta_0;
//   filter      x_k = M x_{k-1} + g Delta_k (k >= 1), x_0 = (Delta_0, 0, 0),
// so the samples are split into kChunks chunks of L samples and scanned in
// three phases by a CTA of 32 columns x kChunks chunks (one thread each):
//   1. every chunk runs its recurrence from a zero state (chunk 0 from the
//      true initial state) and leaves its end state in shared memory;
//   2. one thread per column chains the chunks: the state entering chunk j+1
//      is A^L (state entering chunk j) + (chunk j's zero-start end state),
//      with A^L = rho^L or M^L precomputed on the host in double;
//   3. every chunk reruns its recurrence from its true entering state and
//      writes the basis vectors.
// Loads and stores are coalesced over the 32 columns of a warp.  The
// recurrences run in fp32 with FMAs (fp64 chains are several times slower on
// this part); the rounding stays far below the bf16 output rounding for a
// stable filter.  Linear interpolation needs no scan (phase 3 only).
constexpr int kChunks = 16;
constexpr int kCols = 32;

struct SmoothConsts {
  float rho, rhoL;     // EMA: (1 - beta)^gamma and its L-th power
  float al, be, ga;    // filter gains
  float ML[9];         // filter: M^L, row-major
  long long L;         // samples per chunk
};

__device__ __forceinline__ void abg_step(float& p, float& v, float& a, float y, const SmoothConsts& c) {
  const float pp = fmaf(0.5f, a, p + v);  // predicted position
  const float vp = v + a;                 // predicted velocity
  const float res = y - pp;
  p = fmaf(c.al, res, pp);
  v = fmaf(c.be, res, vp);
  a = fmaf(c.ga, res, a);
}

__global__ void __launch_bounds__(kCols * kChunks) delta_smooth_kernel(const float* __restrict__ delta,
                                                                      float* __restrict__ basis,
                                                                      float* __restrict__ coef, long long n_s, int d,
                                                                      int gamma, int n_coef, int kind,
                                                                      double beta, SmoothConsts sc) {
  __shared__ float st[kChunks][3][kCols];  // chunk end states, then entering states
  const int lane = threadIdx.x % kCols, j = threadIdx.x / kCols;
  if (blockIdx.x == 0) {
    for (int r = threadIdx.x; r < n_coef; r += blockDim.x) {
      double a = 1.0, b = 0.0;
      if (kind == SMOOTH_LINEAR) {
        b = (double)r / (double)gamma;
        a = 1.0 - b;
      } else if (kind == SMOOTH_EMA) {
        a = pow(1.0 - beta, (double)(r + 1));
        b = 1.0 - a;
      }
      coef[r * kSmoothJ] = (float)a;
      coef[r * kSmoothJ + 1] = (float)b;
    }
  }
  const int groups = d / kCols;
  const long long bh = blockIdx.x / groups;
  const int c = (int)(blockIdx.x % groups) * kCols + lane;
  const float* __restrict__ x = delta + bh * n_s * d + c;
  float* __restrict__ out = basis + bh * n_s * kSmoothJ * d + c;
  const long long k0 = (long long)j * sc.L, k1 = k0 + sc.L < n_s ? k0 + sc.L : n_s;

  if (kind == SMOOTH_LINEAR) {
#pragma unroll 8
    for (long long k = k0; k < k1; ++k) {
      out[(k * kSmoothJ) * d] = x[k * d];
      out[(k * kSmoothJ + 1) * d] = x[(k + 1 < n_s ? k + 1 : k) * d];
    }
    return;
  }
  // phase 1: zero-start end state of the chunk (chunk 0: from the true start)
  float s0 = 0.f, s1 = 0.f, s2 = 0.f;
  if (kind == SMOOTH_EMA) {
    if (j == 0 && k0 < k1) s0 = x[0];
#pragma unroll 8
    for (long long k = k0; k < k1; ++k) s0 = fmaf(sc.rho, s0 - x[k * d], x[k * d]);
  } else {
    long long kb = k0;
    if (j == 0 && k0 < k1) {
      s0 = x[0];
      kb = 1;
    }
#pragma unroll 8
    for (long long k = kb; k < k1; ++k) abg_step(s0, s1, s2, x[k * d], sc);
  }
  st[j][0][lane] = s0;
  st[j][1][lane] = s1;
  st[j][2][lane] = s2;
  __syncthreads();
  // phase 2: entering state of every chunk (chunk 0 starts from the initial
  // state itself, marked by its index)
  if (j == 0) {
    float e0 = st[0][0][lane], e1 = st[0][1][lane], e2 = st[0][2][lane];  // leaving chunk 0
    for (int q = 1; q < kChunks; ++q) {
      const float l0 = st[q][0][lane], l1 = st[q][1][lane], l2 = st[q][2][lane];
      st[q][0][lane] = e0;
      st[q][1][lane] = e1;
      st[q][2][lane] = e2;
      if (kind == SMOOTH_EMA) {
        e0 = fmaf(sc.rhoL, e0, l0);
      } else {
        const float n0 = fmaf(sc.ML[0], e0, fmaf(sc.ML[1], e1, fmaf(sc.ML[2], e2, l0)));
        const float n1 = fmaf(sc.ML[3], e0, fmaf(sc.ML[4], e1, fmaf(sc.ML[5], e2, l1)));
        const float n2 = fmaf(sc.ML[6], e0, fmaf(sc.ML[7], e1, fmaf(sc.ML[8], e2, l2)));
        e0 = n0;
        e1 = n1;
        e2 = n2;
      }
    }
  }
  __syncthreads();
  // phase 3: rerun from the entering state, writing the basis
  if (kind == SMOOTH_EMA) {
    float e = (j == 0) ? x[0] : st[j][0][lane];
#pragma unroll 8
    for (long long k = k0; k < k1; ++k) {
      const float y = x[k * d];
      out[(k * kSmoothJ) * d] = e;
      out[(k * kSmoothJ + 1) * d] = y;
      e = fmaf(sc.rho, e - y, y);
    }
  } else {
    float p, v, a;
    long long kb = k0;
    if (j == 0) {
      p = x[0];
      v = a = 0.f;
      if (k0 < k1) {
        out[0] = p;
        out[d] = 0.f;
      }
      kb = 1;
    } else {
      p = st[j][0][lane];
      v = st[j][1][lane];
      a = st[j][2][lane];
    }
#pragma unroll 8
    for (long long k = kb; k < k1; ++k) {
      abg_step(p, v, a, x[k * d], sc);
      out[(k * kSmoothJ) * d] = p;
      out[(k * kSmoothJ + 1) * d] = 0.f;
    }
  }
}

cudaError_t launch_delta_smooth(const float* delta, float* basis, float* coef, long long BH, long long n_s, int d,
                                int gamma, int n_coef, int kind, double c1, double c2, double c3, cudaStream_t s) {
  SmoothConsts sc{};
  sc.L = (n_s + kChunks - 1) / kChunks;
  if (kind == SMOOTH_EMA) {
    const double rho = std::pow(1.0 - c1, (double)gamma);
    sc.rho = (float)rho;
    sc.rhoL = (float)std::pow(rho, (double)sc.L);
  } else if (kind == SMOOTH_ABG) {
    sc.al = (float)c1;
    sc.be = (float)c2;
    sc.ga = (float)c3;
    // M of the filter step x_k = M x_{k-1} + g Delta_k (predict, then correct
    // with the residual Delta_k - predicted position), raised to the L-th
    // power by repeated squaring in double.
    double M[9] = {1 - c1, 1 - c1, 0.5 * (1 - c1), -c2, 1 - c2, 1 - 0.5 * c2, -c3, -c3, 1 - 0.5 * c3};
    double R[9] = {1, 0, 0, 0, 1, 0, 0, 0, 1};
    auto mul = [](const double* A, const double* B, double* C) {
      double T[9];
      for (int i = 0; i < 3; ++i)
        for (int k = 0; k < 3; ++k) T[i * 3 + k] = A[i * 3] * B[k] + A[i * 3 + 1] * B[3 + k] + A[i * 3 + 2] * B[6 + k];
      for (int i = 0; i < 9; ++i) C[i] = T[i];
    };
    for (long long e = sc.L; e > 0; e >>= 1) {
      if (e & 1) mul(R, M, R);
      mul(M, M, M);
    }
    for (int i = 0; i < 9; ++i) sc.ML[i] = (float)R[i];
  }
  const long long blocks = BH * (d / kCols);
  if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
  delta_smooth_kernel<<<(unsigned)blocks, kCols * kChunks, 0, s>>>(delta, basis, coef, n_s, d, gamma, n_coef, kind,
                                                                     c1, sc);
  return cudaGetLastError();
}

}  // namespace da
