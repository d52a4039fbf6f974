// attn_kernel.cuh — the tcgen05 flash-attention kernel behind all three parts
// of the Delta Attention prefill (arXiv 2505.11254, Alg. 1):
//   MODE_SPARSE          f*(Q,K,V): StreamingLLM sink + window attention, every row
//   MODE_STRIDED_DENSE   f(~Q,K,V): dense causal attention of the rows k*gamma (Eq. 4)
//   MODE_STRIDED_SPARSE  f* at the rows k*gamma (only when gamma does not divide BM)
// and the Delta epilogues (Eq. 6) that turn them into the corrected output.
//
// One CTA owns a 128-row query tile (TMEM lanes) and walks its key tiles.
// Warp roles (192 threads):
//   warps 0-3  softmax: one query row per thread; TMEM S -> P (bf16, in TMEM);
//              lazy O rescaling; the epilogue.
//   warp 4     TMA producer: Q once, then K and V tiles through a STAGES ring.
//   warp 5     MMA issuer: S = Q K^T (smem x smem -> TMEM) and O += P V
//              (TMEM x smem -> TMEM), tcgen05.commit -> mbarriers.
// TMEM: S/P double buffer at columns [0, 2*BN), O at [2*BN, 2*BN + D).
// Every wait is bounded: a wait that exceeds WAIT_LIMIT_NS sets the CTA's
// abort flag and the device status word, every role leaves its loop, the CTA
// drains its in-flight copies and MMAs, frees TMEM and returns.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ptx.cuh"
#include "tiles.cuh"
#include "wait.cuh"

namespace da {

constexpr int kThreads = 192;
constexpr float RESCALE_THRESHOLD = 8.0f;  // log2 units; O is rescaled only past this

template <int D>
struct Cfg {
  static constexpr int STAGES = (D == 128) ? 3 : 4;
  static constexpr int CHUNKS = D / 64;                  // 64-element (128-byte) swizzle columns
  static constexpr uint32_t Q_BYTES = BM * D * 2;
  static constexpr uint32_t KV_BYTES = BN * D * 2;
  static constexpr uint32_t SMEM = Q_BYTES + 2 * STAGES * KV_BYTES + 1024;  // + alignment slack
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t COL_O = 2 * BN;
  static constexpr uint32_t IDESC_QK = idesc_bf16(BM, BN, 0, 0);
  static constexpr uint32_t IDESC_PV = idesc_bf16(BM, D, 0, 1);
};

struct Bars {
  uint64_t q_full;
  uint64_t k_full[4], v_full[4], k_empty[4], v_empty[4];
  uint64_t s_full[2], p_full[2];
  uint64_t o_done;
  uint64_t drain;
};

__device__ __forceinline__ void named_bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

template <int D>
__device__ __forceinline__ void store_row_bf16(__nv_bfloat16* dst, const float* v) {
#pragma unroll
  for (int c = 0; c < 32; c += 8) {
    uint4 u;
    u.x = pack_bf16x2(v[c + 0], v[c + 1]);
    u.y = pack_bf16x2(v[c + 2], v[c + 3]);
    u.z = pack_bf16x2(v[c + 4], v[c + 5]);
    u.w = pack_bf16x2(v[c + 6], v[c + 7]);
    *reinterpret_cast<uint4*>(dst + c) = u;
  }
}

__device__ __forceinline__ void store_f32x32(float* dst, const float* v) {
#pragma unroll
  for (int c = 0; c < 32; c += 4) *reinterpret_cast<float4*>(dst + c) = make_float4(v[c], v[c + 1], v[c + 2], v[c + 3]);
}

__device__ __forceinline__ void load_f32x32(const float* src, float* v) {
#pragma unroll
  for (int c = 0; c < 32; c += 4) {
    float4 f = *reinterpret_cast<const float4*>(src + c);
    v[c] = f.x; v[c + 1] = f.y; v[c + 2] = f.z; v[c + 3] = f.w;
  }
}

// Loads data other CTAs wrote during this kernel: bypass L1.
__device__ __forceinline__ void load_f32x32_cg(const float* src, float* v) {
#pragma unroll
  for (int c = 0; c < 32; c += 4) {
    float4 f = __ldcg(reinterpret_cast<const float4*>(src + c));
    v[c] = f.x; v[c + 1] = f.y; v[c + 2] = f.z; v[c + 3] = f.w;
  }
}

template <int D, int MODE, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const Params p) {
  using C = Cfg<D>;
  constexpr int ST = C::STAGES;
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* dsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = dsm;
  uint8_t* sK = sQ + C::Q_BYTES;
  uint8_t* sV = sK + ST * C::KV_BYTES;

  __shared__ Bars bars;
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_sh;
  __shared__ int ticket_sh;

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const Work w = decode_work<MODE>(p, blockIdx.x);
  const int T = w.T;

  if (tid == 0) {
    mbar_init(&bars.q_full, 1);
    for (int s = 0; s < ST; ++s) {
      mbar_init(&bars.k_full[s], 1);
      mbar_init(&bars.v_full[s], 1);
      mbar_init(&bars.k_empty[s], 1);
      mbar_init(&bars.v_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars.s_full[b], 1);
      mbar_init(&bars.p_full[b], 128);
    }
    mbar_init(&bars.o_done, 1);
    mbar_init(&bars.drain, 1);
    abort_sh = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&tmem_base_sh, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;

  if (warp == 4) {
    // ------------------------------------------------------------ producer
    if ((tid & 31) == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmV);
      const int qz = w.b * p.Hq + w.h0;
      const int kz = w.b * p.Hkv + w.g;
      mbar_arrive_expect_tx(&bars.q_full, C::Q_BYTES);
      for (int c = 0; c < C::CHUNKS; ++c)
        tma_load_3d(sQ + c * (BM * 128), &tmQ, &bars.q_full, c * 64, (int)w.r0, qz);
      int nk = 0, nv = 0;  // K and V tiles issued
      for (int j = 0; j < T; ++j) {
        const int s = j % ST;
        const uint32_t n = j / ST;
        const int krow = (int)(tile_index(w, j) * BN);
        if (j >= ST && !wait_bounded(&bars.k_empty[s], (n - 1) & 1, &abort_sh, p.err)) break;
        mbar_arrive_expect_tx(&bars.k_full[s], C::KV_BYTES);
        for (int c = 0; c < C::CHUNKS; ++c)
          tma_load_3d(sK + s * C::KV_BYTES + c * (BN * 128), &tmK, &bars.k_full[s], c * 64, krow, kz);
        ++nk;
        if (j >= ST && !wait_bounded(&bars.v_empty[s], (n - 1) & 1, &abort_sh, p.err)) break;
        mbar_arrive_expect_tx(&bars.v_full[s], C::KV_BYTES);
        for (int c = 0; c < C::CHUNKS; ++c)
          tma_load_3d(sV + s * C::KV_BYTES + c * (BN * 128), &tmV, &bars.v_full[s], c * 64, krow, kz);
        ++nv;
      }
      // Drain: every copy lands before the CTA exits.  Copies older than the
      // last ST per ring were consumed (their stage was reused), so only the
      // last ST can be in flight; in the normal path they have landed already.
      for (int jj = (nk > ST ? nk - ST : 0); jj < nk; ++jj) wait_drain(&bars.k_full[jj % ST], (jj / ST) & 1, p.err);
      for (int jj = (nv > ST ? nv - ST : 0); jj < nv; ++jj) wait_drain(&bars.v_full[jj % ST], (jj / ST) & 1, p.err);
      wait_drain(&bars.q_full, 0, p.err);
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------ MMA issuer
    if ((tid & 31) == 0) {
      const uint32_t q_base = smem_u32(sQ);
      const uint32_t k_base = smem_u32(sK);
      const uint32_t v_base = smem_u32(sV);
      bool ok = wait_bounded(&bars.q_full, 0, &abort_sh, p.err);
      tc_fence_after();
      for (int j = 0; ok && j <= T; ++j) {
        if (j < T) {
          const int s = j % ST;
          const uint32_t sb = (j & 1) * BN;
          if (!wait_bounded(&bars.k_full[s], (j / ST) & 1, &abort_sh, p.err)) break;
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (BM * 128) + (kk & 3) * 32;
            const uint32_t koff = (kk >> 2) * (BN * 128) + (kk & 3) * 32;
            mma_ss(tmem + sb, sdesc_sw128(q_base + off, 16, 1024),
                   sdesc_sw128(k_base + s * C::KV_BYTES + koff, 16, 1024), C::IDESC_QK, kk > 0);
          }
          mma_commit(&bars.s_full[j & 1]);
          mma_commit(&bars.k_empty[s]);
        }
        if (j >= 1) {
          const int jp = j - 1;
          const int s = jp % ST;
          const uint32_t sb = (jp & 1) * BN;
          if (!wait_bounded(&bars.p_full[jp & 1], (jp >> 1) & 1, &abort_sh, p.err)) break;
          if (!wait_bounded(&bars.v_full[s], (jp / ST) & 1, &abort_sh, p.err)) break;
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < BN / 16; ++kk) {
            mma_ts(tmem + C::COL_O, tmem + sb + kk * 8,
                   sdesc_sw128(v_base + s * C::KV_BYTES + kk * 2048, BN * 128, 1024), C::IDESC_PV,
                   (jp > 0 || kk > 0) ? 1u : 0u);
          }
          mma_commit(&bars.o_done);
          mma_commit(&bars.v_empty[s]);
        }
      }
      // Drain: all MMAs issued by this thread complete before TMEM is freed.
      mma_commit(&bars.drain);
      wait_drain(&bars.drain, 0, p.err);
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int t = tid;  // TMEM lane = query row of the tile
    const uint32_t lane_addr = static_cast<uint32_t>(warp * 32) << 16;
    long long row, sample;
    int head;
    const bool row_ok = lane_row<MODE>(p, w, t, row, sample, head);
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < T && ok; ++j) {
      const uint32_t sb = (j & 1) * BN;
      if (!__all_sync(0xffffffffu, wait_bounded(&bars.s_full[j & 1], (j >> 1) & 1, &abort_sh, p.err))) {
        ok = false;
        break;
      }
      tc_fence_after();
      float x[BN];
#pragma unroll
      for (int q = 0; q < BN / 32; ++q) {
        uint32_t r[32];
        tmem_ld32(tmem + lane_addr + sb + q * 32, r);
        tmem_ld_wait();
#pragma unroll
        for (int c = 0; c < 32; ++c) x[q * 32 + c] = __uint_as_float(r[c]) * p.scale_log2;
      }
      if (tile_needs_mask<MODE>(p, w, j)) {
        const long long k0 = tile_index(w, j) * BN;
#pragma unroll
        for (int c = 0; c < BN; ++c) {
          const long long key = k0 + c;
          const bool vis = (MODE == MODE_STRIDED_DENSE) ? visible_causal(row, key)
                                                        : visible_sparse(row, key, p.n_sink, p.window);
          if (!vis) x[c] = -INFINITY;
        }
      }
      float mt = x[0];
#pragma unroll
      for (int c = 1; c < BN; ++c) mt = fmaxf(mt, x[c]);
      float m_use = m_run;
      bool rescale = false;
      if (m_run == -INFINITY) {
        m_use = mt;
        rescale = (j > 0) && (mt != -INFINITY);  // O holds zeros; scaling by 0 keeps it so
      } else if (mt > m_run + RESCALE_THRESHOLD) {
        m_use = mt;
        rescale = true;
      }
      const float m_base = (m_use == -INFINITY) ? 0.f : m_use;
      float l_tile = 0.f;
      uint32_t pk[BN / 2];
#pragma unroll
      for (int c = 0; c < BN; c += 2) {
        const float p0 = ex2(x[c] - m_base), p1 = ex2(x[c + 1] - m_base);
        l_tile += p0 + p1;
        pk[c / 2] = pack_bf16x2(p0, p1);
      }
      // PV(j-1) must be complete before O is rescaled and before P(j)
      // overwrites the buffer that P(j-2) used (in-order MMA completion).
      if (j >= 1 && !__all_sync(0xffffffffu, wait_bounded(&bars.o_done, (j - 1) & 1, &abort_sh, p.err))) {
        ok = false;
        break;
      }
      // tcgen05.ld/st are warp-collective: the warp rescales together, rows
      // that need no rescale use the factor 1.
      if (__any_sync(0xffffffffu, rescale)) {
        const float f = !rescale ? 1.f : (m_run == -INFINITY) ? 0.f : ex2(m_run - m_use);
        l_run *= f;
        tc_fence_after();
#pragma unroll
        for (int q = 0; q < D / 32; ++q) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_addr + C::COL_O + q * 32, r);
          tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 32; ++c) r[c] = __float_as_uint(__uint_as_float(r[c]) * f);
          tmem_st32(tmem + lane_addr + C::COL_O + q * 32, r);
        }
      }
      l_run += l_tile;
      m_run = m_use;
#pragma unroll
      for (int q = 0; q < BN / 32; ++q) {
        uint32_t r[16];
#pragma unroll
        for (int c = 0; c < 16; ++c) r[c] = pk[q * 16 + c];
        tmem_st16(tmem + lane_addr + sb + q * 16, r);
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&bars.p_full[j & 1]);
    }
    if (ok && T > 0) ok = __all_sync(0xffffffffu, wait_bounded(&bars.o_done, (T - 1) & 1, &abort_sh, p.err));
    tc_fence_after();

    // ------------------------------------------------------------ epilogue
    const long long bh = (long long)w.b * p.Hq + head;
    const float inv_l = (l_run > 0.f) ? 1.f / l_run : 0.f;

    if (EPI == EPI_BF16 || EPI == EPI_FUSED_INTILE || EPI == EPI_FUSED_DELTA || EPI == EPI_DELTA_BUILD) {
      float* slot = reinterpret_cast<float*>(sK);  // K ring is idle once every MMA completed
      const bool sampled = row_ok && is_sampled_row(row, p.gamma);
      if (EPI == EPI_FUSED_INTILE) {
        fence_proxy_async_smem();  // generic writes after the ring's TMA writes
        // Pass 1: sampled rows publish their sparse output for the rows of their group.
        float* dst = slot + (t / p.gamma) * D;
#pragma unroll 1
        for (int q = 0; q < D / 32; ++q) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_addr + C::COL_O + q * 32, r);
          tmem_ld_wait();
          if (ok && sampled) {
#pragma unroll
            for (int c = 0; c < 32; ++c) dst[q * 32 + c] = __uint_as_float(r[c]) * inv_l;
          }
        }
        named_bar_sync(1, 128);
      }
#pragma unroll 1
      for (int q = 0; q < D / 32; ++q) {
        uint32_t r[32];
        tmem_ld32(tmem + lane_addr + C::COL_O + q * 32, r);
        tmem_ld_wait();
        float v[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) v[c] = __uint_as_float(r[c]) * inv_l;
        if (!ok || !row_ok) continue;
        if (EPI == EPI_BF16) {
          store_row_bf16<D>(reinterpret_cast<__nv_bfloat16*>(p.out_bf16) + (bh * p.N + row) * D + q * 32, v);
          if (p.s_sampled != nullptr && sampled) store_f32x32(p.s_sampled + (bh * p.n_s + sample) * D + q * 32, v);
        } else if (EPI == EPI_FUSED_INTILE || EPI == EPI_FUSED_DELTA) {
          float dk[32];
          load_f32x32(p.d_in + (bh * p.n_s + sample) * D + q * 32, dk);
          if (!sampled) {
            float corr[32];
            if (EPI == EPI_FUSED_INTILE) {
              const float* sk = slot + (t / p.gamma) * D + q * 32;
#pragma unroll
              for (int c = 0; c < 32; ++c) corr[c] = dk[c] - sk[c];
            } else {
              load_f32x32(p.delta_in + (bh * p.n_s + sample) * D + q * 32, corr);
            }
#pragma unroll
            for (int c = 0; c < 32; ++c) dk[c] = v[c] + corr[c];
          }
          store_row_bf16<D>(reinterpret_cast<__nv_bfloat16*>(p.out_bf16) + (bh * p.N + row) * D + q * 32, dk);
        } else {  // EPI_DELTA_BUILD: Delta_k = D_k - S_{k gamma}
          float dk[32];
          load_f32x32(p.d_in + (bh * p.n_s + sample) * D + q * 32, dk);
#pragma unroll
          for (int c = 0; c < 32; ++c) dk[c] -= v[c];
          store_f32x32(p.delta_out + (bh * p.n_s + sample) * D + q * 32, dk);
        }
      }
    } else {
      // Dense sampled rows: the whole key range in this CTA, or split-K
      // partials merged by the last CTA of the M-tile to finish.
      const size_t slot_floats = (size_t)BM * (D + 2);
      auto store_final = [&](int q, const float* v) {
        if (EPI == EPI_DENSE_F32)
          store_f32x32(p.d_out + (bh * p.n_s + sample) * D + q * 32, v);
        else
          store_row_bf16<D>(reinterpret_cast<__nv_bfloat16*>(p.out_bf16) + (bh * p.N + row) * D + q * 32, v);
      };
      if (w.n_chunks == 1) {
#pragma unroll 1
        for (int q = 0; q < D / 32; ++q) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_addr + C::COL_O + q * 32, r);
          tmem_ld_wait();
          float v[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) v[c] = __uint_as_float(r[c]) * inv_l;
          if (ok && row_ok) store_final(q, v);
        }
      } else {
        float* part = p.partials + (size_t)w.unit * slot_floats;
#pragma unroll 1
        for (int q = 0; q < D / 32; ++q) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_addr + C::COL_O + q * 32, r);
          tmem_ld_wait();
          float v[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) v[c] = __uint_as_float(r[c]);
          if (ok) store_f32x32(part + (size_t)t * D + q * 32, v);
        }
        if (ok) {
          part[(size_t)BM * D + t] = m_run;
          part[(size_t)BM * D + BM + t] = l_run;
        }
        __threadfence();
        named_bar_sync(1, 128);
        if (t == 0) {
          const int prev = abort_sh ? -1 : atomicAdd(p.tickets + w.u0, 1);
          ticket_sh = prev;
          if (prev == w.n_chunks - 1) p.tickets[w.u0] = 0;  // ready for the next call
        }
        named_bar_sync(1, 128);
        if (ticket_sh == w.n_chunks - 1 && row_ok) {
          __threadfence();
          float mstar = -INFINITY;
          for (int c = 0; c < w.n_chunks; ++c)
            mstar = fmaxf(mstar, __ldcg(p.partials + (size_t)(w.u0 + c) * slot_floats + (size_t)BM * D + t));
          float lsum = 0.f;
          for (int c = 0; c < w.n_chunks; ++c) {
            const float* pc = p.partials + (size_t)(w.u0 + c) * slot_floats;
            const float mc = __ldcg(pc + (size_t)BM * D + t);
            if (mc != -INFINITY) lsum += __ldcg(pc + (size_t)BM * D + BM + t) * ex2(mc - mstar);
          }
          const float inv = (lsum > 0.f) ? 1.f / lsum : 0.f;
#pragma unroll 1
          for (int q = 0; q < D / 32; ++q) {
            float v[32];
#pragma unroll
            for (int c = 0; c < 32; ++c) v[c] = 0.f;
            for (int c2 = 0; c2 < w.n_chunks; ++c2) {
              const float* pc = p.partials + (size_t)(w.u0 + c2) * slot_floats;
              const float mc = __ldcg(pc + (size_t)BM * D + t);
              if (mc == -INFINITY) continue;
              const float f = ex2(mc - mstar);
              float o[32];
              load_f32x32_cg(pc + (size_t)t * D + q * 32, o);
#pragma unroll
              for (int c = 0; c < 32; ++c) v[c] += o[c] * f;
            }
#pragma unroll
            for (int c = 0; c < 32; ++c) v[c] *= inv;
            store_final(q, v);
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, C::TMEM_COLS);
}

}  // namespace da
