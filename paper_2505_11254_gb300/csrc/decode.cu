// decode.cu — Eq. 2: decoding after the sparse prefill.  The query of each
// newly generated token attends densely over the whole cache [K u k_new],
// [V u v_new] of its sequence (the new key and value already appended).
//
// The step reads every cached key and value once and does 4*d FLOPs per key
// and query head, so it is bound by HBM bandwidth, not by the tensor cores
// (with one query row per head there is no tile to fill).  Design:
//   * split-K: a CTA per (batch, KV head, key range) handles the G query
//     heads of the KV group together, so each K/V byte is read once;
//   * a producer warp streams K and V chunks (contiguous rows) with
//     cp.async.bulk into a shared-memory ring completed on mbarriers: eight
//     stages of 16 keys (two per consumer warp, so a warp's next chunk loads
//     while it works on the current one) or, when a warp iteration takes 32
//     keys, four of 32; the key range is split so that one wave of CTAs fills
//     every SM;
//   * four consumer warps take whole chunks in turn.  Inside a warp, groups
//     of LPK lanes work on different keys (layout in DecLayout): a lane holds
//     a slice of the channels of q and o for every head (GP = G rounded up to
//     a power of two), forms partial dot products for its group's keys, and
//     a reduce-scatter over the group's lanes completes the scores; the online
//     softmax (running max and sum per head and group, exp2 with
//     log2(e)/sqrt(d) folded into q) then broadcasts each weight to the
//     group's lanes for P.V with packed fp32 FMAs;
//   * the (warp, group) partial states are merged in shared memory and written as
//     (unnormalised o, max, sum) per split; a second kernel, launched as a
//     programmatic dependent so that its launch overlaps this one, merges the
//     splits in a fixed order (deterministic) and writes bf16.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "launch.h"
#include "ptx.cuh"
#include "wait.cuh"

namespace da {
namespace {

constexpr int kDecWarps = 4;                        // consumer warps
constexpr int kDecThreads = (kDecWarps + 1) * 32;   // + the producer warp
constexpr int kDecQORegs = 64;  // registers per lane for its slices of q and o
constexpr int kDecMinCtas = 2;  // CTAs per SM the register allocation must allow

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ uint64_t f2_pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// Lane layout of a consumer warp for GP (padded) query heads of width D:
//   LPK lanes share one key (a group; NG = 32 / LPK groups per warp run on
//   different keys), each lane holding CPL = D / LPK channels of q and o for
//   all GP heads (2 * GP * CPL <= kDecQORegs registers, so that two CTAs fit
//   an SM's register file);
//   a group forms the partial dot products of KG keys x GP heads over its
//   channels (N = KG * GP values per lane) and reduce-scatters them over its
//   LPK lanes, leaving R = N / LPK complete scores per lane;
//   channels are dealt in 16-byte pieces, piece p of a row to lane p % LPK,
//   so the lanes of a quarter warp read one contiguous 128-byte span.
template <int D, int GP>
struct DecLayout {
  static constexpr int cl(int x, int lo, int hi) { return x < lo ? lo : (x > hi ? hi : x); }
  static constexpr int mn(int a, int b) { return a < b ? a : b; }
  static constexpr int LPK = cl(2 * GP * D / kDecQORegs, 2, 32);
  static constexpr int NG = 32 / LPK;
  static constexpr int CPL = D / LPK;
  static constexpr int R = mn(mn(4, GP), 32 / LPK);
  static constexpr int N = LPK * R;
  static constexpr int KG = N / GP;
  static constexpr int KEYS = NG * KG;           // keys per warp iteration
  static constexpr int PS = CPL < 8 ? CPL : 8;   // channels per piece
  static constexpr int T = CPL / PS;             // pieces per lane
  static_assert(KG >= 1 && N % GP == 0 && N % LPK == 0, "layout");
};

// The ring of a kernel instance: chunks of max(16, KEYS) keys, eight stages
// of 16 keys or four of 32 (64 KB at d = 128 either way, so two CTAs fit an
// SM).  Chunk i goes to stage i % STAGES and to consumer warp i % kDecWarps.
// With STAGES a multiple of kDecWarps every phase of a stage is consumed by
// the same warp in order, so a parity wait can never be satisfied by a phase
// two behind the one it wants.
template <int D, int GP>
struct DecRing {
  static constexpr int KEYS = DecLayout<D, GP>::KEYS;
  static constexpr int CHUNK = KEYS > 16 ? KEYS : 16;
  static constexpr int STAGES = CHUNK == 16 ? 8 : 4;
  static constexpr int SMEM = STAGES * 2 * CHUNK * D * 2 + 1024;
  static_assert(CHUNK % KEYS == 0, "a chunk holds whole iterations");
  static_assert(STAGES % kDecWarps == 0, "each stage must belong to one consumer warp");
};

// Channels of one row slice (T pieces of PS channels) as floats.
template <int D, int GP>
__device__ __forceinline__ void load_slice(const __nv_bfloat16* row, int sub, float* f) {
  using L = DecLayout<D, GP>;
#pragma unroll
  for (int t = 0; t < L::T; ++t) {
    const __nv_bfloat16* src = row + (sub + L::LPK * t) * L::PS;
    if constexpr (L::PS == 8) {
      const uint4 u = *reinterpret_cast<const uint4*>(src);
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        f[t * 8 + 2 * e] = __uint_as_float(w[e] << 16);
        f[t * 8 + 2 * e + 1] = __uint_as_float(w[e] & 0xffff0000u);
      }
    } else if constexpr (L::PS == 4) {
      const uint2 u = *reinterpret_cast<const uint2*>(src);
      f[t * 4 + 0] = __uint_as_float(u.x << 16);
      f[t * 4 + 1] = __uint_as_float(u.x & 0xffff0000u);
      f[t * 4 + 2] = __uint_as_float(u.y << 16);
      f[t * 4 + 3] = __uint_as_float(u.y & 0xffff0000u);
    } else {
      static_assert(L::PS == 2, "pieces of 2, 4 or 8 channels");
      const uint32_t u = *reinterpret_cast<const uint32_t*>(src);
      f[t * 2 + 0] = __uint_as_float(u << 16);
      f[t * 2 + 1] = __uint_as_float(u & 0xffff0000u);
    }
  }
}

template <int D, int GP>
__global__ void __launch_bounds__(kDecThreads, kDecMinCtas) decode_kernel(DecodeParams p) {
  using L = DecLayout<D, GP>;
  using Ring = DecRing<D, GP>;
  constexpr int CPL = L::CPL, R = L::R, LPK = L::LPK, KG = L::KG, N = L::N;
  constexpr int CHUNK = Ring::CHUNK, STAGES = Ring::STAGES;  // keys per stage, stages
  constexpr unsigned kFull = 0xffffffffu;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __nv_bfloat16* ring = reinterpret_cast<__nv_bfloat16*>(smem);  // [stage][K|V][CHUNK][D]
  __shared__ uint64_t full[STAGES], empty[STAGES];
  __shared__ volatile int abort_sh;
  constexpr int kStates = kDecWarps * L::NG;  // (warp, group) partial softmax states
  __shared__ float sm_m[kStates][GP], sm_l[kStates][GP];
  __shared__ float sm_o[kStates][GP][D];

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const long long unit = blockIdx.x;
  const int s = (int)(unit % p.n_split);
  const long long bg = unit / p.n_split;  // b * Hkv + g
  const int b = (int)(bg / p.Hkv), g = (int)(bg % p.Hkv);
  long long n = p.lens != nullptr ? p.lens[b] : p.max_keys;
  n = n < 0 ? 0 : (n > p.L ? p.L : n);
  const long long k_begin = (long long)s * p.split_keys;
  const long long k_end = (k_begin + p.split_keys < n) ? k_begin + p.split_keys : n;
  const int nc = k_end > k_begin ? (int)((k_end - k_begin + CHUNK - 1) / CHUNK) : 0;

  if (threadIdx.x == 0) {
    // let the merge grid be scheduled now; it waits for this grid's completion
    asm volatile("griddepcontrol.launch_dependents;");
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    abort_sh = 0;
    fence_mbar_init();
  }
  __syncthreads();

  const __nv_bfloat16* Kg = p.K + (bg * p.L) * D;
  const __nv_bfloat16* Vg = p.V + (bg * p.L) * D;
  if (warp == kDecWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int issued = 0;
      for (int i = 0; i < nc; ++i) {
        const int st = i % STAGES;
        if (i >= STAGES && !wait_bounded(&empty[st], ((i / STAGES) - 1) & 1, &abort_sh, p.err)) break;
        const long long k0 = k_begin + (long long)i * CHUNK;
        const long long nk = (k_end - k0 < CHUNK) ? k_end - k0 : CHUNK;
        const uint32_t bytes = (uint32_t)(nk * D * 2);
        mbar_arrive_expect_tx(&full[st], 2 * bytes);
        bulk_g2s(ring + (size_t)(st * 2) * CHUNK * D, Kg + k0 * D, bytes, &full[st]);
        bulk_g2s(ring + (size_t)(st * 2 + 1) * CHUNK * D, Vg + k0 * D, bytes, &full[st]);
        ++issued;
      }
      // The ring must be quiet before the CTA exits: wait for the latest
      // phase of every stage still in use.
      for (int i = (issued > STAGES ? issued - STAGES : 0); i < issued; ++i)
        wait_drain(&full[i % STAGES], (i / STAGES) & 1, p.err);
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const int grp = lane / LPK, sub = lane % LPK, gbase = lane & ~(LPK - 1);
  const int G = p.G;
  float qv[GP][CPL];
#pragma unroll
  for (int h = 0; h < GP; ++h) {
    if (h < G) {
      load_slice<D, GP>(p.q + ((long long)b * p.Hq + (long long)g * G + h) * D, sub, qv[h]);
#pragma unroll
      for (int c = 0; c < CPL; ++c) qv[h][c] *= p.scale_log2;
    } else {
#pragma unroll
      for (int c = 0; c < CPL; ++c) qv[h][c] = 0.f;
    }
  }
  float o[GP][CPL];
#pragma unroll
  for (int h = 0; h < GP; ++h)
#pragma unroll
    for (int c = 0; c < CPL; ++c) o[h][c] = 0.f;
  // running max / sum of heads h0 .. h0 + R - 1 of this lane's group
  float m_own[R], l_own[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    m_own[r] = -INFINITY;
    l_own[r] = 0.f;
  }
  const int kk_own = (sub * R) / GP;  // key (within the group's KG) of this lane's scores

  for (int i = warp; i < nc; i += kDecWarps) {
    const int st = i % STAGES;
    if (!__all_sync(kFull, wait_bounded(&full[st], (i / STAGES) & 1, &abort_sh, p.err))) break;
    const __nv_bfloat16* Ks = ring + (size_t)(st * 2) * CHUNK * D;
    const __nv_bfloat16* Vs = ring + (size_t)(st * 2 + 1) * CHUNK * D;
    const long long k0 = k_begin + (long long)i * CHUNK;
    const int nk = (int)((k_end - k0 < CHUNK) ? k_end - k0 : CHUNK);
    const bool partial = nk < CHUNK;  // warp-uniform
#pragma unroll 1
    for (int kb = 0; kb < nk; kb += L::KEYS) {
      const int key0 = kb + grp * KG;  // this group's first key in the chunk
      float acc[N];
#pragma unroll
      for (int kk = 0; kk < KG; ++kk) {
        float kf[CPL];
        load_slice<D, GP>(Ks + (size_t)(key0 + kk) * D, sub, kf);  // rows past nk: stale, masked below
#pragma unroll
        for (int h = 0; h < GP; ++h) {
          uint64_t a2 = f2_pack(0.f, 0.f);
#pragma unroll
          for (int c = 0; c < CPL; c += 2)
            a2 = f2_fma(f2_pack(qv[h][c], qv[h][c + 1]), f2_pack(kf[c], kf[c + 1]), a2);
          float x0, x1;
          f2_unpack(a2, x0, x1);
          acc[kk * GP + h] = x0 + x1;
        }
      }
      // reduce-scatter over the LPK lanes of the group: lane sub ends with the
      // complete scores of pairs sub * R .. sub * R + R - 1 (key x / GP, head x % GP)
      int cnt = N;
#pragma unroll
      for (int off = LPK / 2; off >= 1; off >>= 1) {
        const bool upper = (sub & off) != 0;
        const int half = cnt / 2;
#pragma unroll
        for (int e = 0; e < N / 2; ++e) {
          if (e < half) {
            const float send = upper ? acc[e] : acc[e + half];
            const float keep = upper ? acc[e + half] : acc[e];
            acc[e] = keep + __shfl_xor_sync(kFull, send, off);
          }
        }
        cnt = half;
      }
      const bool key_ok = key0 + kk_own < nk;
      float pr[R], alpha[R];
      bool grew = false;
#pragma unroll
      for (int r = 0; r < R; ++r) {
        const float sc = key_ok ? acc[r] : -INFINITY;
        float mh = sc;
#pragma unroll
        for (int off = GP / R; off < LPK; off <<= 1) mh = fmaxf(mh, __shfl_xor_sync(kFull, mh, off));
        const float m_new = fmaxf(m_own[r], mh);
        const float mu = (m_new == -INFINITY) ? 0.f : m_new;
        pr[r] = ex2(sc - mu);
        alpha[r] = ex2(m_own[r] - mu);
        float ps = pr[r];
#pragma unroll
        for (int off = GP / R; off < LPK; off <<= 1) ps += __shfl_xor_sync(kFull, ps, off);
        l_own[r] = l_own[r] * alpha[r] + ps;
        grew = grew || (m_new != m_own[r]);
        m_own[r] = m_new;
      }
      // O is rescaled only when some running max grew (alpha = 1 exactly
      // otherwise), which after the first keys is rare.
      if (__any_sync(kFull, grew)) {
#pragma unroll
        for (int h = 0; h < GP; ++h) {
          const float ah = __shfl_sync(kFull, alpha[h % R], gbase + h / R);
#pragma unroll
          for (int c = 0; c < CPL; ++c) o[h][c] *= ah;
        }
      }
#pragma unroll
      for (int kk = 0; kk < KG; ++kk) {
        float vf[CPL];
        load_slice<D, GP>(Vs + (size_t)(key0 + kk) * D, sub, vf);
        if (partial && key0 + kk >= nk) {  // stale rows of the last chunk may hold anything
#pragma unroll
          for (int c = 0; c < CPL; ++c) vf[c] = 0.f;
        }
#pragma unroll
        for (int h = 0; h < GP; ++h) {
          const int x = kk * GP + h;
          const float pk = __shfl_sync(kFull, pr[x % R], gbase + x / R);
          const uint64_t pk2 = f2_pack(pk, pk);
#pragma unroll
          for (int c = 0; c < CPL; c += 2) {
            float lo, hi;
            f2_unpack(f2_fma(pk2, f2_pack(vf[c], vf[c + 1]), f2_pack(o[h][c], o[h][c + 1])), lo, hi);
            o[h][c] = lo;
            o[h][c + 1] = hi;
          }
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[st]);
  }

  // merge the (warp, group) states, then write this split's partial
  const int state = warp * L::NG + grp;
  if (sub < GP / R) {
#pragma unroll
    for (int r = 0; r < R; ++r) {
      sm_m[state][sub * R + r] = m_own[r];
      sm_l[state][sub * R + r] = l_own[r];
    }
  }
#pragma unroll
  for (int h = 0; h < GP; ++h)
#pragma unroll
    for (int t = 0; t < L::T; ++t)
#pragma unroll
      for (int e = 0; e < L::PS; ++e) sm_o[state][h][(sub + LPK * t) * L::PS + e] = o[h][t * L::PS + e];
  asm volatile("bar.sync 1, %0;" ::"n"(kDecWarps * 32) : "memory");
  float* part = p.part + (size_t)unit * G * (D + 2);
  for (int idx = threadIdx.x; idx < G * D; idx += kDecWarps * 32) {
    const int h = idx / D, c = idx % D;
    float M = -INFINITY;
    for (int w = 0; w < kStates; ++w) M = fmaxf(M, sm_m[w][h]);
    const float Mu = (M == -INFINITY) ? 0.f : M;
    float acc = 0.f, lsum = 0.f;
    for (int w = 0; w < kStates; ++w) {
      const float f = ex2(sm_m[w][h] - Mu);
      acc = fmaf(sm_o[w][h][c], f, acc);
      lsum = fmaf(sm_l[w][h], f, lsum);
    }
    part[h * (D + 2) + c] = acc;
    if (c == 0) {
      part[h * (D + 2) + D] = M;
      part[h * (D + 2) + D + 1] = lsum;
    }
  }
}

// One CTA per (batch, query head): the split weights 2^(m_s - M) and the
// weighted sum of the split sums are formed once in shared memory; then each
// warp accumulates every column over its own residue class of splits (a lane
// holds columns lane + 32 j, so a warp reads each split's row in 128-byte
// pieces) and the warps' sums are added in warp order.  Every reduction has
// a fixed shape and order, so the result does not depend on timing.
constexpr int kMergeWarps = 8;
constexpr int kMergeThreads = kMergeWarps * 32;

__device__ __forceinline__ float block_reduce(float v, float* red, bool is_max) {
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float x = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, x) : v + x;
  }
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float r = red[0];
#pragma unroll
  for (int w = 1; w < kMergeWarps; ++w) r = is_max ? fmaxf(r, red[w]) : r + red[w];
  __syncthreads();  // red is reused by the next reduction
  return r;
}

template <int D>
__global__ void __launch_bounds__(kMergeThreads) decode_merge_kernel(const float* __restrict__ part,
                                                                     __nv_bfloat16* out, int Hq, int Hkv, int G,
                                                                     int n_split) {
  constexpr int J = D / 32;  // columns per lane
  extern __shared__ float w_sh[];  // [n_split] split weights
  __shared__ float red[kMergeWarps];
  __shared__ float acc_sh[kMergeWarps][D];
  // The partials are written by the split kernel, which may still be running
  // when this grid is scheduled (programmatic dependent launch): wait for it
  // to complete and its writes to be visible.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const long long bh = blockIdx.x;
  const long long b = bh / Hq;
  const int h = (int)(bh % Hq), g = h / G, hh = h % G;
  const float* base = part + ((size_t)(b * Hkv + g) * n_split) * G * (D + 2) + (size_t)hh * (D + 2);
  const size_t stride = (size_t)G * (D + 2);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

  float m = -INFINITY;
  for (int s = threadIdx.x; s < n_split; s += kMergeThreads) m = fmaxf(m, base[s * stride + D]);
  const float M = block_reduce(m, red, true);
  const float Mu = (M == -INFINITY) ? 0.f : M;
  float l = 0.f;
  for (int s = threadIdx.x; s < n_split; s += kMergeThreads) {
    const float f = ex2(base[s * stride + D] - Mu);
    w_sh[s] = f;
    l = fmaf(base[s * stride + D + 1], f, l);
  }
  const float lsum = block_reduce(l, red, false);  // its barriers also publish w_sh

  float a[J];
#pragma unroll
  for (int j = 0; j < J; ++j) a[j] = 0.f;
#pragma unroll 4
  for (int s = warp; s < n_split; s += kMergeWarps) {
    const float f = w_sh[s];
    const float* row = base + s * stride + lane;
#pragma unroll
    for (int j = 0; j < J; ++j) a[j] = fmaf(row[32 * j], f, a[j]);
  }
#pragma unroll
  for (int j = 0; j < J; ++j) acc_sh[warp][lane + 32 * j] = a[j];
  __syncthreads();
  if (threadIdx.x < D) {
    float acc = 0.f;
#pragma unroll
    for (int w = 0; w < kMergeWarps; ++w) acc += acc_sh[w][threadIdx.x];
    out[bh * D + threadIdx.x] = __float2bfloat16_rn(lsum > 0.f ? acc / lsum : 0.f);
  }
}

template <int D, int GP>
cudaError_t launch_decode_t(const DecodeParams& p, long long units, cudaStream_t s) {
  auto k = decode_kernel<D, GP>;
  static bool attr_set[64] = {};  // the attribute is set once per function and device
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64 || !attr_set[dev]) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, DecRing<D, GP>::SMEM);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) attr_set[dev] = true;
  }
  k<<<(unsigned)units, kDecThreads, DecRing<D, GP>::SMEM, s>>>(p);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_decode_d(const DecodeParams& p, long long units, cudaStream_t s) {
  const int G = p.G;
  if (G <= 1) return launch_decode_t<D, 1>(p, units, s);
  if (G <= 2) return launch_decode_t<D, 2>(p, units, s);
  if (G <= 4) return launch_decode_t<D, 4>(p, units, s);
  if (G <= 8) return launch_decode_t<D, 8>(p, units, s);
  return launch_decode_t<D, 16>(p, units, s);
}

}  // namespace

template <int D>
int keys_per_chunk_d(int G) {
  if (G <= 1) return DecRing<D, 1>::CHUNK;
  if (G <= 2) return DecRing<D, 2>::CHUNK;
  if (G <= 4) return DecRing<D, 4>::CHUNK;
  if (G <= 8) return DecRing<D, 8>::CHUNK;
  return DecRing<D, 16>::CHUNK;
}

int decode_keys_per_split(int d, int G) { return d == 64 ? keys_per_chunk_d<64>(G) : keys_per_chunk_d<128>(G); }

// Queried once per kernel instance (the answer is the same on every GB300;
// concurrent first calls compute the same value).
template <int D, int GP>
int ctas_per_sm_t() {
  static int cached = 0;
  if (cached > 0) return cached;
  int n = 0;
  auto k = decode_kernel<D, GP>;
  if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, DecRing<D, GP>::SMEM) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k, kDecThreads, DecRing<D, GP>::SMEM) != cudaSuccess)
    return 1;
  cached = n > 0 ? n : 1;
  return cached;
}

template <int D>
int ctas_per_sm_d(int G) {
  if (G <= 1) return ctas_per_sm_t<D, 1>();
  if (G <= 2) return ctas_per_sm_t<D, 2>();
  if (G <= 4) return ctas_per_sm_t<D, 4>();
  if (G <= 8) return ctas_per_sm_t<D, 8>();
  return ctas_per_sm_t<D, 16>();
}

int decode_ctas_per_sm(int d, int G) { return d == 64 ? ctas_per_sm_d<64>(G) : ctas_per_sm_d<128>(G); }

cudaError_t launch_decode(const DecodeParams& p, void* out, cudaStream_t s) {
  const long long units = (long long)p.B * p.Hkv * p.n_split;
  const long long rows = (long long)p.B * p.Hq;
  if (units <= 0 || units > 0x7fffffffLL || rows > 0x7fffffffLL) return cudaErrorInvalidValue;
  const size_t w_bytes = (size_t)p.n_split * sizeof(float);
  if (w_bytes > 32768) return cudaErrorInvalidValue;  // far above one wave of splits on any GPU
  cudaError_t e = p.D == 64 ? launch_decode_d<64>(p, units, s) : launch_decode_d<128>(p, units, s);
  if (e != cudaSuccess) return e;
  // The merge grid is launched as a programmatic dependent of the split
  // kernel: it is scheduled while the split kernel runs and waits on the
  // device (griddepcontrol.wait) for its partials.
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)rows);
  cfg.blockDim = dim3(kMergeThreads);
  cfg.dynamicSmemBytes = w_bytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const float* part = p.part;
  __nv_bfloat16* o = static_cast<__nv_bfloat16*>(out);
  e = p.D == 64 ? cudaLaunchKernelEx(&cfg, decode_merge_kernel<64>, part, o, p.Hq, p.Hkv, p.G, p.n_split)
                : cudaLaunchKernelEx(&cfg, decode_merge_kernel<128>, part, o, p.Hq, p.Hkv, p.G, p.n_split);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace da
