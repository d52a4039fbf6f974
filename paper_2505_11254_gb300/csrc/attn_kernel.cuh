// attn_kernel.cuh — the tcgen05 flash-attention kernel behind all three parts
// of the Delta Attention prefill (arXiv 2505.11254, Alg. 1):
//   MODE_SPARSE          f*(Q,K,V): StreamingLLM sink + window attention, every row
//   MODE_STRIDED_DENSE   f(~Q,K,V): dense causal attention of the rows k*gamma (Eq. 4)
//   MODE_STRIDED_SPARSE  f* at the rows k*gamma (when the Delta is not fused in-tile)
// and the Delta epilogues (Eq. 6) that turn them into the corrected output.
//
// Persistent: each CTA walks work items blockIdx.x, blockIdx.x + gridDim.x, ...
// An item is a 128-row query tile (TMEM lanes) and its list of 128-key tiles.
// Warp roles (384 threads = 3 warpgroups):
//   warps 0-3  softmax: one query row per thread; S (TMEM) -> P (bf16, TMEM,
//              aliasing S); lazy O rescaling; per item the row sum l and max m.
//   warps 4-7  epilogue: rotates the next item's Q in smem ahead of time when
//              RoPE is on, then reads O out of TMEM, releases it, normalises,
//              applies the Delta correction (or, in the dense pass, writes or
//              merges the split-K partials) and writes the output.
//   warp 8     TMA producer: Q of the next item, K tiles through their ring.
//   warp 9     QK issuer: S = Q K^T once its K tile has landed and the PV
//              that last read the S buffer has completed; Q and K from smem
//              (one Q buffer at d = 128, reloaded after the item's last QK;
//              two at d = 64).
//   warp 10    PV issuer: O += P V (P from TMEM, V from smem) once the softmax
//              has written P(g).  Two issuing threads keep the tensor pipe fed:
//              neither waits on the other's inputs.
//   warp 11    V producer: V tiles through their own ring, so K loads never
//              wait for a PV to free a slot.
// Registers: launched at 168 per thread (384 x 168 = 64512); the third
// warpgroup gives back to 72 and the softmax and epilogue warpgroups grow to
// 216, so 2 x 128 x 216 + 128 x 72 = 64512 exactly.
// TMEM (512 columns, see Cfg): an S/P triple buffer and O, so QK may run
// three tiles ahead of the softmax and the chain softmax(g) -> PV(g) ->
// QK(g+3) spans three tiles.
// Every wait is bounded: past its limit a wait sets the CTA's abort flag and
// the device status word, the roles stop working (keeping every named barrier
// and warp-collective instruction uniform), drain their in-flight copies and
// MMAs, free TMEM and return.
// The sink + window pass also comes as a two-CTA form (PAIR, see Cfg): a
// cluster of two CTAs takes two query heads of one row tile, the leader's
// warps 9 and 10 issue cta_group::2 MMAs for both, and each CTA holds half of
// every K and V tile.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ptx.cuh"
#include "tiles.cuh"
#include "launch.h"
#include "wait.cuh"

namespace da {

constexpr int kThreads = 384;
constexpr int kRegsCompute = 216;  // softmax and epilogue warpgroups
constexpr int kRegsControl = 72;   // producer / MMA warpgroup
static_assert(2 * 128 * kRegsCompute + 128 * kRegsControl <= kThreads * 168, "register split above the launch total");
// O and the row sum are rescaled only when the running max grows by more than
// this many log2 units.  Until then P = 2^(s - m) can reach 2^64: bf16 and fp32
// share the 8-bit exponent, and 2^64 x 2^20 keys x |v| stays far below the
// fp32 range, so the final O / l is unchanged (it is a ratio).
constexpr float RESCALE_THRESHOLD = 64.0f;
constexpr uint32_t kFull = 0xffffffffu;

// TMEM layout (512 columns), all passes: S/P triple buffer [0,128) [128,256)
// [256,384), O [384, 384 + D).  QK reads Q and K from smem and may run three
// tiles ahead of the softmax.  (A dense-pass layout with Q in TMEM, two S/P
// buffers and no Q reads from smem measured 6-7 % slower: the third S buffer
// is worth more than the shared-memory reads it saves.)
//
// PAIR (sink + window pass, d = 128, the query heads of a KV group taken two
// at a time): a cluster of two CTAs runs the two heads' items of the same
// row tile, which visit the same key tiles.  The leader issues every MMA for
// both with cta_group::2 (M = 256): each CTA keeps its own Q, S/P and O, and
// holds only half of each K tile (keys 0-63 in the leader, 64-127 in the peer)
// and half of each V tile (columns 0-63 / 64-127).  Per tile an SM then moves
// 96 KB through shared memory (Q 32, K half 16 and V half 16 read by the
// tensor core, 32 written by TMA) instead of 160 KB.
template <int D, int MODE = MODE_SPARSE, bool PAIR = false>
struct Cfg {
  static_assert(!PAIR || (D == 128 && MODE == MODE_SPARSE), "the two-CTA form is the d = 128 sink + window pass");
  static constexpr int NQ = PAIR ? 2 : (D == 128) ? 1 : 2;  // Q buffers in smem
  static constexpr int NK = PAIR ? 5 : (D == 128) ? 3 : 4;  // K ring slots (D = 128: five fit beside Q)
  static constexpr int NV = PAIR ? 4 : (D == 128) ? 2 : 4;  // V ring slots
  static constexpr int NS = NK + NV;
  static constexpr int NSB = 3;                           // S/P buffers in TMEM
  static constexpr int CHUNKS = D / 64;          // 64-element (128-byte) swizzle columns
  static constexpr uint32_t Q_BYTES = BM * D * 2;
  static constexpr uint32_t K_BYTES = (PAIR ? BN / 2 : BN) * D * 2;  // a K slot: this CTA's keys of a tile
  static constexpr uint32_t V_BYTES = BN * (PAIR ? D / 2 : D) * 2;   // a V slot: this CTA's columns of a tile
  static constexpr uint32_t K_CHUNK = (PAIR ? BN / 2 : BN) * 128;    // bytes of one swizzle column of a K slot
  static constexpr int V_CHUNKS = PAIR ? 1 : CHUNKS;
  static constexpr uint32_t SBUF_BYTES = kSampleBufBytes;  // sampled sparse rows of the fused epilogue
  static constexpr uint32_t SMEM = NQ * Q_BYTES + NK * K_BYTES + NV * V_BYTES + SBUF_BYTES + 1024;
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t COL_S = 0;                  // + BN * buffer
  static constexpr uint32_t COL_O = 384;
  static constexpr uint32_t IDESC_QK = idesc_bf16(PAIR ? 2 * BM : BM, BN, 0, 0);
  static constexpr uint32_t IDESC_PV = idesc_bf16(PAIR ? 2 * BM : BM, D, 0, 1);
  // Arrivals that complete p_full, o_free and qt_ready: every thread of the
  // warpgroup, or in a pair one per warp of both CTAs.
  static constexpr uint32_t ARRIVALS = PAIR ? 8 : 128;
  static_assert(COL_O + D <= TMEM_COLS, "TMEM layout");
  static_assert(BN == 128, "the softmax loads S in two 64-column halves and stores P in two 32-column halves");
  static_assert(NK <= 8 && NV <= 8, "ring barriers");
  static_assert(SMEM <= 232448, "shared memory above the 227 KB per-block limit");
};

struct Bars {
  uint64_t kfull[8], kempty[8], vfull[8], vempty[8];
  uint64_t q_full[2], q_free[2];
  uint64_t qt_ready[2];
  uint64_t s_full[3], p_full[3];
  uint64_t pv_done[3], o_full, o_free;
  uint64_t l_ready[2], l_free[2];
  uint64_t drain, drain2;
};

template <int N>
__device__ __forceinline__ void regs_increase() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}
template <int N>
__device__ __forceinline__ void regs_decrease() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}

__device__ __forceinline__ void named_bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
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
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

__device__ __forceinline__ void store_bf16x32(__nv_bfloat16* dst, const float* v) {
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

// TMEM lane quarter of a warp: warps w and w+4 see lanes 32*(w%4) .. +31.
__device__ __forceinline__ uint32_t lane_base(int warp) { return static_cast<uint32_t>((warp & 3) * 32) << 16; }

template <int NCOL>
__device__ __forceinline__ void tmem_ld_row(uint32_t addr, float (&v)[NCOL]) {
#pragma unroll
  for (int q = 0; q < NCOL / 32; ++q) {
    uint32_t r[32];
    tmem_ld32(addr + q * 32, r);
#pragma unroll
    for (int c = 0; c < 32; ++c) v[q * 32 + c] = __uint_as_float(r[c]);
  }
  tmem_ld_wait();
}

// Work items of a CTA.  Static: blockIdx.x, blockIdx.x + gridDim.x, ...
// Dynamic (the split-K dense units, whose lengths differ): the producer claims
// items from a global counter, longest first, and publishes them to the other
// roles through a small shared-memory queue; the others read them in order.
constexpr int kQueue = 8;
constexpr int kQueueReaders = 11;  // V producer, QK and PV threads + 4 softmax warps + 4 epilogue warps
struct ItemQueue {
  long long item[kQueue];
  uint64_t full[kQueue], empty[kQueue];
};

// WARP_WIDE: all 32 lanes of the warp call next() together (softmax and
// epilogue warps); otherwise a single lane does (the MMA thread) and no
// warp-collective instruction may be used.
template <bool DYN, bool WARP_WIDE>
struct ItemReader {
  long long next_static;
  int n = 0;
  __device__ long long next(const Params& p, ItemQueue& q, volatile int* abort_flag) {
    if (!DYN) {
      const long long v = next_static;
      next_static += gridDim.x;
      return v < p.n_items ? v : -1;
    }
    const int slot = n % kQueue;
    long long v = -1;
    bool got = wait_bounded(&q.full[slot], (n / kQueue) & 1, abort_flag, p.err);
    if (WARP_WIDE) got = __all_sync(kFull, got);
    if (got) v = q.item[slot];
    if (WARP_WIDE) {
      __syncwarp();
      if ((threadIdx.x & 31) == 0) mbar_arrive(&q.empty[slot]);
    } else {
      mbar_arrive(&q.empty[slot]);
    }
    ++n;
    return v;
  }
};

// ROWS: the kernel of a row-range call (Params::q_row0 > 0): items start at
// row q_row0, Q and O hold rows from q_row0.  Whole-sequence launches use
// ROWS = false.
// PAIR: launched in clusters of two (see Cfg).  The items of CTA x are those
// of the one-CTA kernel (x, x + gridDim.x, ...); with G even and the grid
// even, items 2c and 2c + 1 are the two heads of one row tile, so the two
// CTAs of a cluster always work on the same row tile and key tiles.
template <int D, int MODE, int EPI, bool ROWS = false, bool PAIR = false>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const Params p) {
  using C = Cfg<D, MODE, PAIR>;
  static_assert(!PAIR || !ROWS, "row-range calls use the one-CTA kernel");
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* dsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = dsm;  // [NQ][Q_BYTES]: item i uses buffer i % NQ
  uint8_t* ring = sQ + C::NQ * C::Q_BYTES;  // K slots [0, NK), then V slots
  uint8_t* vring = ring + C::NK * C::K_BYTES;
  float* sbuf = reinterpret_cast<float*>(vring + C::NV * C::V_BYTES);

  __shared__ Bars bars;
  __shared__ uint32_t tmem_base_sh;
  __shared__ volatile int abort_sh;
  __shared__ int ticket_sh;
  __shared__ float lfin[2][BM], mfin[2][BM];
  __shared__ ItemQueue iq;
  constexpr bool DYN = (MODE == MODE_STRIDED_DENSE);

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  // Pair: this CTA's rank; the leader (rank 0) issues the MMAs and owns the
  // barriers both CTAs signal, addressed through the cluster window.
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
  const bool leader = rank == 0;
  auto at_leader = [&](uint64_t* bar) { return mapa_shared(smem_u32(bar), 0); };

  if (tid == 0) {
    for (int s = 0; s < C::NK; ++s) {
      mbar_init(&bars.kfull[s], 1);
      mbar_init(&bars.kempty[s], 1);
    }
    for (int s = 0; s < C::NV; ++s) {
      mbar_init(&bars.vfull[s], 1);
      mbar_init(&bars.vempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars.q_full[b], 1);
      mbar_init(&bars.q_free[b], 1);  // the item's last QK
      mbar_init(&bars.qt_ready[b], C::ARRIVALS);
      mbar_init(&bars.l_ready[b], 128);
      mbar_init(&bars.l_free[b], 128);
    }
    for (int b = 0; b < C::NSB; ++b) {
      mbar_init(&bars.s_full[b], 1);
      mbar_init(&bars.p_full[b], C::ARRIVALS);
      mbar_init(&bars.pv_done[b], 1);
    }
    mbar_init(&bars.o_full, 1);
    mbar_init(&bars.o_free, C::ARRIVALS);
    mbar_init(&bars.drain, 1);
    mbar_init(&bars.drain2, 1);
    for (int k = 0; k < kQueue; ++k) {
      mbar_init(&iq.full[k], 1);
      mbar_init(&iq.empty[k], kQueueReaders);
    }
    abort_sh = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    if (PAIR) {
      tmem_alloc_pair(&tmem_base_sh, C::TMEM_COLS);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(&tmem_base_sh, C::TMEM_COLS);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  if (PAIR) cluster_sync();  // both CTAs' barriers exist before either signals the other's
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;

  if (warp == 8) {
    // ================================================================ producer
    regs_decrease<kRegsControl>();
    if ((tid & 31) == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmV);
      int c = 0, nq = 0;
      bool ok = true;
      auto load_q = [&](long long item) {
        const Work wq = decode_work<MODE, ROWS>(p, item);
        // buffer qb held the Q of item nq - NQ: its last QK must have read it
        const int qb = nq % C::NQ;
        if (nq >= C::NQ && !wait_bounded(&bars.q_free[qb], ((nq / C::NQ) - 1) & 1, &abort_sh, p.err))
          return false;
        if (PAIR) {
          // Without RoPE the QK issuer waits for both CTAs' Q on the leader's
          // barrier; with RoPE each CTA's epilogue first rotates its own Q.
          const bool at_lead = p.rope == nullptr;
          if (leader || !at_lead) mbar_arrive_expect_tx(&bars.q_full[qb], at_lead ? 2 * C::Q_BYTES : C::Q_BYTES);
          const uint32_t bar = at_lead ? at_leader(&bars.q_full[qb]) : mapa_shared(smem_u32(&bars.q_full[qb]), rank);
          for (int ch = 0; ch < C::CHUNKS; ++ch)
            tma_load_3d_pair(sQ + qb * C::Q_BYTES + ch * (BM * 128), &tmQ, bar, ch * 64, (int)wq.r0,
                             wq.b * p.Hq + wq.h0);
        } else {
          mbar_arrive_expect_tx(&bars.q_full[qb], C::Q_BYTES);
          for (int ch = 0; ch < C::CHUNKS; ++ch)
            tma_load_3d(sQ + qb * C::Q_BYTES + ch * (BM * 128), &tmQ, &bars.q_full[qb], ch * 64,
                        (int)(ROWS && MODE == MODE_SPARSE ? wq.r0 - p.q_row0 : wq.r0), wq.b * p.Hq + wq.h0);
        }
        ++nq;
        return true;
      };
      // K tiles only: the V tiles have their own ring and producer (warp
      // 11), so a K load never waits for a PV to free a slot.
      auto load_k = [&](int row, int z) {
        const int s = c % C::NK;
        if (c >= C::NK && !wait_bounded(&bars.kempty[s], ((c / C::NK) - 1) & 1, &abort_sh, p.err)) return false;
        if (PAIR) {
          // this CTA's half of the tile's keys, counted on the leader's barrier
          if (leader) mbar_arrive_expect_tx(&bars.kfull[s], 2 * C::K_BYTES);
          const uint32_t bar = at_leader(&bars.kfull[s]);
          for (int ch = 0; ch < C::CHUNKS; ++ch)
            tma_load_3d_pair(ring + s * C::K_BYTES + ch * C::K_CHUNK, &tmK, bar, ch * 64, row + (int)rank * (BN / 2),
                             z);
        } else {
          mbar_arrive_expect_tx(&bars.kfull[s], C::K_BYTES);
          for (int ch = 0; ch < C::CHUNKS; ++ch)
            tma_load_3d(ring + s * C::K_BYTES + ch * C::K_CHUNK, &tmK, &bars.kfull[s], ch * 64, row, z);
        }
        ++c;
        return true;
      };
      // Claims the next item (or -1) and, when dynamic, publishes it.
      long long next_static = blockIdx.x;
      int np = 0;
      bool done = false;
      auto claim = [&]() -> long long {
        long long v = -1;
        if (!done) {
          if (DYN) {
            v = (long long)atomicAdd(p.counter, 1ull);
          } else {
            v = next_static;
            next_static += gridDim.x;
          }
          if (v >= p.n_items) v = -1;
        }
        if (DYN && !done) {
          const int slot = np % kQueue;
          if (np >= kQueue && !wait_bounded(&iq.empty[slot], ((np / kQueue) - 1) & 1, &abort_sh, p.err)) v = -1;
          iq.item[slot] = v;
          mbar_arrive(&iq.full[slot]);
          ++np;
        }
        done = done || v < 0;
        return v;
      };
      long long item = claim();
      if (item >= 0) ok = load_q(item);
      while (ok && item >= 0) {
        const Work w = decode_work<MODE, ROWS>(p, item);
        const int kz = w.b * p.Hkv + w.g;
        long long nxt = -1;
        for (int j = 0; ok && j < w.T; ++j) {
          const int krow = (int)(tile_index(w, j) * BN);
          ok = load_k(krow, kz);
          if (ok && j == 0) {
            nxt = claim();
            // with two Q buffers the next item's Q goes out at once
            if (C::NQ >= 2 && nxt >= 0) ok = load_q(nxt);
          }
        }
        // with one Q buffer it waits for this item's last QK, so it goes out
        // after this item's K/V loads (which that QK needs)
        if (C::NQ == 1 && ok && nxt >= 0) ok = load_q(nxt);
        item = nxt;
      }
      if (DYN && !done) claim();  // the readers always see the end of the sequence
      // Drain: only the last NK K loads and the last Q loads can be in flight.
      // In a pair the leader's barriers count both CTAs' copies, so the leader
      // drains for both (the peer drains its own Q only when it has a barrier
      // of its own, with RoPE).
      if (!PAIR || leader)
        for (int u = (c > C::NK ? c - C::NK : 0); u < c; ++u)
          wait_drain(&bars.kfull[u % C::NK], (u / C::NK) & 1, p.err);
      if (!PAIR || leader || p.rope != nullptr)
        for (int k = (nq > C::NQ ? nq - C::NQ : 0); k < nq; ++k)
          wait_drain(&bars.q_full[k % C::NQ], (k / C::NQ) & 1, p.err);
    }
  } else if (warp == 9) {
    // ================================================================ QK issuer
    regs_decrease<kRegsControl>();
    if ((tid & 31) == 0 && leader) {
      // Shared-memory descriptors of Q buffer 0 and ring slot 0; a buffer,
      // slot or K-step adds its byte offset / 16 to the start-address field.
      const uint64_t qdesc0 = sdesc_sw128(smem_u32(sQ), 16, 1024);
      const uint64_t kdesc0 = sdesc_sw128(smem_u32(ring), 16, 1024);
      const bool rope = p.rope != nullptr;
      uint32_t g = 0;  // tiles so far: ring slots and phases (32-bit: cheap divisions by constants)
      bool ok = true;
      ItemReader<DYN, false> items{(long long)blockIdx.x};
      int i = 0;
      for (long long item = items.next(p, iq, &abort_sh); ok && item >= 0; item = items.next(p, iq, &abort_sh), ++i) {
        const Work w = decode_work<MODE, ROWS>(p, item);
        // Q of item i: in smem buffer i % NQ (rotated in place first when RoPE is on)
        const int qb = i % C::NQ;
        uint64_t* qbar = rope ? &bars.qt_ready[qb] : &bars.q_full[qb];
        if (!wait_bounded(qbar, (uint32_t)(i / C::NQ) & 1, &abort_sh, p.err)) {
          ok = false;
          break;
        }
        const uint64_t qd = qdesc0 + ((qb * C::Q_BYTES) >> 4);
        for (int j = 0; j < w.T; ++j, ++g) {
          const int ks = (int)(g % C::NK);
          const uint32_t kph = (uint32_t)(g / C::NK) & 1;
          const int sbi = (int)(g % C::NSB);
          if (!wait_bounded(&bars.kfull[ks], kph, &abort_sh, p.err)) { ok = false; break; }
          // S buffer sbi held P(g - NSB): that PV must have read it.
          if (g >= C::NSB &&
              !wait_bounded(&bars.pv_done[sbi], (uint32_t)((g - C::NSB) / C::NSB) & 1, &abort_sh, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sb = tmem + C::COL_S + (uint32_t)sbi * BN;
          const uint64_t kd = kdesc0 + ((ks * C::K_BYTES) >> 4);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t qoff = (((kk >> 2) * (BM * 128)) + (kk & 3) * 32) >> 4;
            const uint32_t koff = (((kk >> 2) * C::K_CHUNK) + (kk & 3) * 32) >> 4;
            if (PAIR)
              mma_ss_pair(sb, qd + qoff, kd + koff, C::IDESC_QK, kk > 0 ? 1u : 0u);
            else
              mma_ss(sb, qd + qoff, kd + koff, C::IDESC_QK, kk > 0 ? 1u : 0u);
          }
          if (PAIR)
            mma_commit_pair_both(&bars.s_full[sbi]);
          else
            mma_commit(&bars.s_full[sbi]);
        }
        if (ok) {  // the item's last QK has read its Q
          if (PAIR)
            mma_commit_pair_both(&bars.q_free[qb]);
          else
            mma_commit(&bars.q_free[qb]);
        }
      }
      if (!ok)  // after an early exit, read the item queue to its end marker
        while (items.next(p, iq, &abort_sh) >= 0) {}
      if (PAIR)
        mma_commit_pair_local(&bars.drain);
      else
        mma_commit(&bars.drain);
      wait_drain(&bars.drain, 0, p.err);
    }
  } else if (warp == 10) {
    // ================================================================ PV issuer
    regs_decrease<kRegsControl>();
    if ((tid & 31) == 0 && leader) {
      const uint64_t vdesc0 = sdesc_sw128(smem_u32(vring), BN * 128, 1024);
      uint32_t g = 0;  // tiles so far: ring slots and phases (32-bit: cheap divisions by constants)
      bool ok = true;
      ItemReader<DYN, false> items{(long long)blockIdx.x};
      int i = 0;
      for (long long item = items.next(p, iq, &abort_sh); ok && item >= 0; item = items.next(p, iq, &abort_sh), ++i) {
        const Work w = decode_work<MODE, ROWS>(p, item);
        for (int j = 0; j < w.T; ++j, ++g) {
          const int vs = (int)(g % C::NV);
          const uint32_t vph = (uint32_t)(g / C::NV) & 1;
          const int sbi = (int)(g % C::NSB);
          if (!wait_bounded(&bars.p_full[sbi], (uint32_t)(g / C::NSB) & 1, &abort_sh, p.err)) {
            ok = false;
            break;
          }
          if (!wait_bounded(&bars.vfull[vs], vph, &abort_sh, p.err)) { ok = false; break; }
          // The epilogue must have read the previous item's O.
          if (j == 0 && i >= 1 && !wait_bounded(&bars.o_free, (i - 1) & 1, &abort_sh, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sb = tmem + C::COL_S + (uint32_t)sbi * BN;
          const uint64_t vd = vdesc0 + ((vs * C::V_BYTES) >> 4);
#pragma unroll
          for (int kk = 0; kk < BN / 16; ++kk) {
            const uint32_t acc = (kk > 0 || j > 0) ? 1u : 0u;
            if (PAIR)
              mma_ts_pair(tmem + C::COL_O, sb + kk * 8, vd + ((kk * 2048) >> 4), C::IDESC_PV, acc);
            else
              mma_ts(tmem + C::COL_O, sb + kk * 8, vd + ((kk * 2048) >> 4), C::IDESC_PV, acc);
          }
          if (PAIR) {
            mma_commit_pair_both(&bars.pv_done[sbi]);
            mma_commit_pair_both(&bars.vempty[vs]);
            if (j == w.T - 1) mma_commit_pair_both(&bars.o_full);
          } else {
            mma_commit(&bars.pv_done[sbi]);
            mma_commit(&bars.vempty[vs]);
            if (j == w.T - 1) mma_commit(&bars.o_full);
          }
        }
      }
      if (!ok)
        while (items.next(p, iq, &abort_sh) >= 0) {}
      if (PAIR)
        mma_commit_pair_local(&bars.drain2);
      else
        mma_commit(&bars.drain2);
      wait_drain(&bars.drain2, 0, p.err);
    }
  } else if (warp == 11) {
    // ================================================================ V producer
    regs_decrease<kRegsControl>();
    if ((tid & 31) == 0) {
      int c = 0;
      bool ok = true;
      ItemReader<DYN, false> items{(long long)blockIdx.x};
      for (long long item = items.next(p, iq, &abort_sh); ok && item >= 0; item = items.next(p, iq, &abort_sh)) {
        const Work w = decode_work<MODE, ROWS>(p, item);
        const int kz = w.b * p.Hkv + w.g;
        for (int j = 0; ok && j < w.T; ++j) {
          const int s = c % C::NV;
          if (c >= C::NV && !wait_bounded(&bars.vempty[s], ((c / C::NV) - 1) & 1, &abort_sh, p.err)) {
            ok = false;
            break;
          }
          const int krow = (int)(tile_index(w, j) * BN);
          if (PAIR) {
            // this CTA's half of the tile's value columns, counted on the leader's barrier
            if (leader) mbar_arrive_expect_tx(&bars.vfull[s], 2 * C::V_BYTES);
            tma_load_3d_pair(vring + s * C::V_BYTES, &tmV, at_leader(&bars.vfull[s]), (int)rank * (D / 2), krow, kz);
          } else {
            mbar_arrive_expect_tx(&bars.vfull[s], C::V_BYTES);
            for (int ch = 0; ch < C::V_CHUNKS; ++ch)
              tma_load_3d(vring + s * C::V_BYTES + ch * (BN * 128), &tmV, &bars.vfull[s], ch * 64, krow, kz);
          }
          ++c;
        }
      }
      if (!ok)  // after an early exit, read the item queue to its end marker
        while (items.next(p, iq, &abort_sh) >= 0) {}
      if (!PAIR || leader)
        for (int u = (c > C::NV ? c - C::NV : 0); u < c; ++u)
          wait_drain(&bars.vfull[u % C::NV], (u / C::NV) & 1, p.err);
    }
  } else if (warp < 4) {
    // ================================================================ softmax
    regs_increase<kRegsCompute>();
    const int t = tid;
    const uint32_t la = lane_base(warp);
    const float scale = p.scale_log2;
    const uint64_t scale2 = f2_pack(scale, scale);
    uint32_t g = 0;  // tiles so far (32-bit: cheap divisions by constants)
    bool ok = true;
    int i = 0;
    ItemReader<DYN, true> items{(long long)blockIdx.x};
    for (long long item = items.next(p, iq, &abort_sh); item >= 0; item = items.next(p, iq, &abort_sh), ++i) {
      const Work w = decode_work<MODE, ROWS>(p, item);
      long long row, sample;
      int head;
      lane_row<MODE>(p, w, t, row, sample, head);
      int j_plain0, j_plain1;  // tiles [j_plain0, j_plain1) need no mask
      unmasked_tiles<MODE>(p, w, j_plain0, j_plain1);
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; ok && j < w.T; ++j, ++g) {
        const int sbi = (int)(g % C::NSB);
        if (!__all_sync(kFull, wait_bounded(&bars.s_full[sbi], (uint32_t)(g / C::NSB) & 1, &abort_sh, p.err))) {
          ok = false;
          break;
        }
        // S(g) landed, so QK(g) has read its K tile.
        if (t == 0) mbar_arrive(&bars.kempty[g % C::NK]);
        tc_fence_after();
        const uint32_t sb = C::COL_S + (uint32_t)sbi * BN;
        float s[BN];
        {  // S(g): two 64-column loads (fewer, wider TMEM loads than 32-column ones measured faster)
          uint32_t r0[64], r1[64];
          tmem_ld64(tmem + la + sb, r0);
          tmem_ld64(tmem + la + sb + 64, r1);
          tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 64; ++c) {
            s[c] = __uint_as_float(r0[c]);
            s[c + 64] = __uint_as_float(r1[c]);
          }
        }
        if (j < j_plain0 || j >= j_plain1) {
          // Visible key offsets c of this tile: lo <= c <= hi (window and
          // causality), plus c < se (sinks), turned into one 32-bit word of
          // visibility bits per 32-key chunk; each key then keeps its score
          // or becomes -inf by a single bit test.  (A range test per key, with
          // or without a per-chunk warp vote, measured 5-12 % slower.)
          const long long k0 = tile_index(w, j) * BN;
          const int hi = (int)lmax(-1, lmin(BN - 1, row - k0));
          const int lo = (MODE == MODE_STRIDED_DENSE) ? 0 : (int)lmax(0, lmin(BN, row - p.window + 1 - k0));
          const int se = (MODE != MODE_STRIDED_DENSE && k0 < p.n_sink)
                             ? (int)lmin(lmin(BN, (long long)p.n_sink - k0), (long long)hi + 1)
                             : 0;
          uint32_t vis[BN / 32];
#pragma unroll
          for (int q = 0; q < BN / 32; ++q) vis[q] = visible_bits(lo, hi, se, 32 * q);
#pragma unroll
          for (int c = 0; c < BN; ++c) s[c] = ((vis[c >> 5] >> (c & 31)) & 1u) ? s[c] : -INFINITY;
        }
        float mx[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) mx[q] = s[q];
#pragma unroll
        for (int c = 4; c + 8 <= BN; c += 8) {
#pragma unroll
          for (int q = 0; q < 4; ++q) mx[q] = max3(mx[q], s[c + q], s[c + 4 + q]);
        }
        mx[0] = max3(mx[0], s[BN - 4], s[BN - 3]);
        mx[1] = max3(mx[1], s[BN - 2], s[BN - 1]);
        const float mt = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * scale;  // log2 units
        float m_use = m_run;
        bool rescale = false;
        if (m_run == -INFINITY) {
          m_use = mt;  // every earlier P of this row was 0, so O and l are exactly 0: nothing to rescale
        } else if (mt > m_run + RESCALE_THRESHOLD) {
          m_use = mt;
          rescale = true;
        }
        const float nb = (m_use == -INFINITY) ? 0.f : -m_use;
        const uint64_t nb2 = f2_pack(nb, nb);
        uint64_t acc[4] = {0, 0, 0, 0};
        uint32_t pk[BN / 2];
#pragma unroll
        for (int c = 0; c < BN; c += 2) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(s[c], s[c + 1]), scale2, nb2), x0, x1);
          const float p0 = ex2(x0), p1 = ex2(x1);
          acc[(c >> 1) & 3] = f2_add(acc[(c >> 1) & 3], f2_pack(p0, p1));
          pk[c / 2] = pack_bf16x2(p0, p1);
        }
        float a0, a1, a2, a3, a4, a5, a6, a7;
        f2_unpack(acc[0], a0, a1);
        f2_unpack(acc[1], a2, a3);
        f2_unpack(acc[2], a4, a5);
        f2_unpack(acc[3], a6, a7);
        const float l_tile = ((a0 + a1) + (a2 + a3)) + ((a4 + a5) + (a6 + a7));
        // Rescale O (rare): PV(g-1) must have landed.  QK(g-1) waited for
        // PV(g-1-NSB), and the next PV on that buffer needs this thread's
        // P(g-1+NSB), so the parity of PV(g-1) on its buffer is unambiguous.
        if (__any_sync(kFull, rescale)) {
          const int pb = (int)((g - 1) % C::NSB);
          if (!__all_sync(kFull,
                          wait_bounded(&bars.pv_done[pb], (uint32_t)((g - 1) / C::NSB) & 1, &abort_sh, p.err))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const float f = rescale ? ex2(m_run - m_use) : 1.f;
          l_run *= f;
#pragma unroll
          for (int q = 0; q < D / 32; ++q) {
            uint32_t r[32];
            tmem_ld32(tmem + la + C::COL_O + q * 32, r);
            tmem_ld_wait();
#pragma unroll
            for (int c = 0; c < 32; ++c) r[c] = __float_as_uint(__uint_as_float(r[c]) * f);
            tmem_st32(tmem + la + C::COL_O + q * 32, r);
          }
        }
        l_run += l_tile;
        m_run = m_use;
#pragma unroll
        for (int q = 0; q < BN / 64; ++q) {
          uint32_t r[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) r[c] = pk[q * 32 + c];
          tmem_st32(tmem + la + sb + q * 32, r);
        }
        tmem_st_wait();
        tc_fence_before();
        if (PAIR) {  // one arrival per warp, on the leader's barrier
          __syncwarp();
          if ((t & 31) == 0) mbar_arrive_cluster(at_leader(&bars.p_full[sbi]));
        } else {
          mbar_arrive(&bars.p_full[sbi]);
        }
      }
      if (!ok) continue;  // keep reading the item sequence to its end
      // Publish this item's row sum and max to the epilogue.
      if (i >= 2 && !__all_sync(kFull, wait_bounded(&bars.l_free[i & 1], ((i >> 1) - 1) & 1, &abort_sh, p.err))) {
        ok = false;
        continue;
      }
      lfin[i & 1][t] = l_run;
      mfin[i & 1][t] = m_run;
      mbar_arrive(&bars.l_ready[i & 1]);
    }
  } else {
    // ================================================================ epilogue
    regs_increase<kRegsCompute>();
    const int e = tid - 128;  // TMEM lane = query row of the tile
    const uint32_t la = lane_base(warp);
    bool ok = true;
    int nq = 0;
    // RoPE (Sec. 2), rotate-half, when Q comes unrotated: each row of the
    // item's Q tile turns in place in its smem buffer before its first QK.
    // Channel c turns with channel c + D/2 by the angle of the row's position;
    // word k of r holds channels 2k and 2k + 1, its partner word is k + D/4.
    // fp32, one rounding to bf16.  Without RoPE the QK reads the TMA'd tile.
    auto rotate_q = [&](int buf, long long qitem) {
      if (p.rope == nullptr) return;
      ok = ok && __all_sync(kFull, wait_sleepy(&bars.q_full[buf], (nq / C::NQ) & 1, &abort_sh, p.err));
      ++nq;
      const Work wq = decode_work<MODE, ROWS>(p, qitem);
      long long qrow, qsample;
      int qhead;
      if (ok && lane_row<MODE>(p, wq, e, qrow, qsample, qhead)) {
        uint8_t* q = sQ + buf * C::Q_BYTES;
        uint32_t r[D / 2];
#pragma unroll
        for (int ch = 0; ch < C::CHUNKS; ++ch)
#pragma unroll
          for (int pc = 0; pc < 8; ++pc) {
            const uint4 v = *reinterpret_cast<const uint4*>(q + ch * (BM * 128) + e * 128 + ((pc ^ (e & 7)) * 16));
            r[ch * 32 + pc * 4 + 0] = v.x;
            r[ch * 32 + pc * 4 + 1] = v.y;
            r[ch * 32 + pc * 4 + 2] = v.z;
            r[ch * 32 + pc * 4 + 3] = v.w;
          }
        const float4* cs = reinterpret_cast<const float4*>(p.rope + qrow * D);
#pragma unroll
        for (int k = 0; k < D / 4; ++k) {
          const float4 t = __ldg(cs + k);  // (cos, sin) of channels 2k, 2k + 1
          const float a0 = __uint_as_float(r[k] << 16), a1 = __uint_as_float(r[k] & 0xffff0000u);
          const float b0 = __uint_as_float(r[k + D / 4] << 16);
          const float b1 = __uint_as_float(r[k + D / 4] & 0xffff0000u);
          r[k] = pack_bf16x2(a0 * t.x - b0 * t.y, a1 * t.z - b1 * t.w);
          r[k + D / 4] = pack_bf16x2(b0 * t.x + a0 * t.y, b1 * t.z + a1 * t.w);
        }
#pragma unroll
        for (int ch = 0; ch < C::CHUNKS; ++ch)
#pragma unroll
          for (int pc = 0; pc < 8; ++pc)
            *reinterpret_cast<uint4*>(q + ch * (BM * 128) + e * 128 + ((pc ^ (e & 7)) * 16)) =
                make_uint4(r[ch * 32 + pc * 4 + 0], r[ch * 32 + pc * 4 + 1], r[ch * 32 + pc * 4 + 2],
                           r[ch * 32 + pc * 4 + 3]);
      }
      fence_proxy_async_smem();  // the tensor core reads the rotated tile
      if (PAIR) {  // one arrival per warp, on the leader's barrier
        __syncwarp();
        if ((e & 31) == 0) mbar_arrive_cluster(at_leader(&bars.qt_ready[buf]));
      } else {
        mbar_arrive(&bars.qt_ready[buf]);
      }
    };
    ItemReader<DYN, true> items{(long long)blockIdx.x};
    long long item = items.next(p, iq, &abort_sh);
    if (item >= 0) rotate_q(0, item);
    for (int i = 0; item >= 0; ++i) {
      const Work w = decode_work<MODE, ROWS>(p, item);
      const long long nxt = items.next(p, iq, &abort_sh);
      if (nxt >= 0) rotate_q((i + 1) % C::NQ, nxt);
      long long row, sample;
      int head;
      const bool row_ok = lane_row<MODE>(p, w, e, row, sample, head);
      ok = ok && __all_sync(kFull, wait_sleepy(&bars.l_ready[i & 1], (i >> 1) & 1, &abort_sh, p.err));
      const float l_row = lfin[i & 1][e], m_row = mfin[i & 1][e];
      mbar_arrive(&bars.l_free[i & 1]);
      // O lands about one PV after l_ready: a short wait, polled without sleeping
      // so that the next item's first PV is not held back by a sleep interval.
      ok = ok && __all_sync(kFull, wait_bounded(&bars.o_full, i & 1, &abort_sh, p.err));
      tc_fence_after();
      float o[D];
      tmem_ld_row<D>(tmem + la + C::COL_O, o);
      tc_fence_before();
      if (PAIR) {  // one arrival per warp, on the leader's barrier
        __syncwarp();
        if ((e & 31) == 0) mbar_arrive_cluster(at_leader(&bars.o_free));
      } else {
        mbar_arrive(&bars.o_free);
      }
      const long long bh = (long long)w.b * p.Hq + head;
      const float inv_l = (l_row > 0.f) ? 1.f / l_row : 0.f;


      if (EPI == EPI_BF16 || EPI == EPI_FUSED_INTILE || EPI == EPI_FUSED_DELTA || EPI == EPI_DELTA_BUILD ||
          EPI == EPI_FUSED_SMOOTH) {
#pragma unroll
        for (int c = 0; c < D; ++c) o[c] *= inv_l;
        const bool sampled = row_ok && is_sampled_row(row, p.gamma);
        if (EPI == EPI_FUSED_INTILE) {
          // Sampled rows publish their sparse output to the rows of their group.
          named_bar_sync(2, 128);  // the previous item's readers are done with sbuf
          if (ok && sampled) {
            float* dst = sbuf + (e / p.gamma) * D;
#pragma unroll
            for (int c = 0; c < D; c += 4) *reinterpret_cast<float4*>(dst + c) = make_float4(o[c], o[c + 1], o[c + 2], o[c + 3]);
          }
          named_bar_sync(2, 128);
        }
        if (ok && row_ok) {
          __nv_bfloat16* orow = reinterpret_cast<__nv_bfloat16*>(p.out_bf16) + (bh * (ROWS ? p.o_rows : p.N) + row) * D;
#pragma unroll
          for (int q = 0; q < D / 32; ++q) {
            float* v = o + q * 32;
            if (EPI == EPI_BF16) {
              store_bf16x32(orow + q * 32, v);
              if (p.s_sampled != nullptr && sampled) store_f32x32(p.s_sampled + (bh * p.n_s + sample) * D + q * 32, v);
            } else if (EPI == EPI_FUSED_SMOOTH) {
              // every row, sampled or not: S_i + the smoothed correction of offset r
              const int r = (int)(row - sample * p.gamma);
              const float c0 = __ldg(p.smooth_coef + r * kSmoothJ), c1 = __ldg(p.smooth_coef + r * kSmoothJ + 1);
              const float* bk = p.smooth_basis + (bh * p.n_s + sample) * (kSmoothJ * D) + q * 32;
              float b0[32], b1[32];
              load_f32x32(bk, b0);
              load_f32x32(bk + D, b1);
#pragma unroll
              for (int c = 0; c < 32; ++c) b0[c] = fmaf(c1, b1[c], fmaf(c0, b0[c], v[c]));
              store_bf16x32(orow + q * 32, b0);
            } else if (EPI == EPI_FUSED_INTILE || EPI == EPI_FUSED_DELTA) {
              float dk[32];
              load_f32x32(p.d_in + (bh * p.n_s + sample) * D + q * 32, dk);
              if (!sampled) {
                float corr[32];
                if (EPI == EPI_FUSED_INTILE) {
                  const float* sk = sbuf + (e / p.gamma) * D + q * 32;
#pragma unroll
                  for (int c = 0; c < 32; ++c) corr[c] = dk[c] - sk[c];
                } else {
                  load_f32x32(p.delta_in + (bh * p.n_s + sample) * D + q * 32, corr);
                }
#pragma unroll
                for (int c = 0; c < 32; ++c) dk[c] = v[c] + corr[c];
              }
              store_bf16x32(orow + q * 32, dk);
            } else {  // EPI_DELTA_BUILD: Delta_k = D_k - S_{k gamma}
              float dk[32];
              load_f32x32(p.d_in + (bh * p.n_s + sample) * D + q * 32, dk);
#pragma unroll
              for (int c = 0; c < 32; ++c) dk[c] -= v[c];
              store_f32x32(p.delta_out + (bh * p.n_s + sample) * D + q * 32, dk);
            }
          }
        }
      } else {
        // Dense sampled rows: the whole key range in this item, or split-K
        // partials merged by the last CTA of the M-tile to finish (w.unit is
        // this unit's partial slot, w.u0 the M-tile's ticket).
        const size_t slot_floats = (size_t)BM * (D + 2);
        auto store_final = [&](int q, const float* v) {
          if (EPI == EPI_DENSE_F32)
            store_f32x32(p.d_out + (bh * p.n_s + sample) * D + q * 32, v);
          else
            store_bf16x32(reinterpret_cast<__nv_bfloat16*>(p.out_bf16) + (bh * p.o_rows + row) * D + q * 32, v);
        };
        if (w.n_chunks == 1) {
          if (ok && row_ok) {
#pragma unroll
            for (int q = 0; q < D / 32; ++q) {
              float v[32];
#pragma unroll
              for (int c = 0; c < 32; ++c) v[c] = o[q * 32 + c] * inv_l;
              store_final(q, v);
            }
          }
        } else {
          float* part = p.partials + (size_t)w.unit * slot_floats;
          if (ok) {
#pragma unroll
            for (int q = 0; q < D / 32; ++q) store_f32x32(part + (size_t)e * D + q * 32, o + q * 32);
            part[(size_t)BM * D + e] = m_row;
            part[(size_t)BM * D + BM + e] = l_row;
          }
          __threadfence();
          named_bar_sync(2, 128);
          if (e == 0) {
            const int prev = (ok && !abort_sh) ? atomicAdd(p.tickets + w.u0, 1) : -1;
            ticket_sh = prev;
            if (prev == w.n_chunks - 1) p.tickets[w.u0] = 0;  // ready for the next call
          }
          named_bar_sync(2, 128);
          const bool merge = ticket_sh == w.n_chunks - 1;
          named_bar_sync(2, 128);  // ticket_sh is rewritten by the next split item
          if (merge && row_ok) {
            __threadfence();
            // Branch-free over the chunks, unrolled so that several partials'
            // loads are in flight at once.  A chunk no key of which this row
            // sees has m = -inf, l = 0 and O = 0: its weight is 0.
            float mstar = -INFINITY;
#pragma unroll 4
            for (int c = 0; c < w.n_chunks; ++c)
              mstar = fmaxf(mstar, __ldcg(p.partials + (size_t)partial_slot(p, w, c) * slot_floats + (size_t)BM * D + e));
            float lsum = 0.f;
#pragma unroll 4
            for (int c = 0; c < w.n_chunks; ++c) {
              const float* pc = p.partials + (size_t)partial_slot(p, w, c) * slot_floats;
              const float mc = __ldcg(pc + (size_t)BM * D + e);
              const float lc = __ldcg(pc + (size_t)BM * D + BM + e);
              lsum += (mc == -INFINITY) ? 0.f : lc * ex2(mc - mstar);
            }
            const float inv = (lsum > 0.f) ? 1.f / lsum : 0.f;
#pragma unroll 1
            for (int q = 0; q < D / 32; ++q) {
              float v[32];
#pragma unroll
              for (int c = 0; c < 32; ++c) v[c] = 0.f;
#pragma unroll 2
              for (int c2 = 0; c2 < w.n_chunks; ++c2) {
                const float* pc = p.partials + (size_t)partial_slot(p, w, c2) * slot_floats;
                const float mc = __ldcg(pc + (size_t)BM * D + e);
                float x[32];
                load_f32x32_cg(pc + (size_t)e * D + q * 32, x);
                const float f = (mc == -INFINITY) ? 0.f : ex2(mc - mstar);
#pragma unroll
                for (int c = 0; c < 32; ++c) v[c] = fmaf(x[c], f, v[c]);
              }
#pragma unroll
              for (int c = 0; c < 32; ++c) v[c] *= inv;
              store_final(q, v);
            }
          }
        }
      }
      item = nxt;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (PAIR) {
    // After an abort the other CTA's copies may still be landing in this
    // CTA's shared memory or counting on its barriers: give them time.
    if (abort_sh) {
      const uint64_t t0 = globaltimer_ns();
      while (globaltimer_ns() - t0 < 200000ull) __nanosleep(1000);
    }
    // Neither CTA frees its TMEM or exits while the pair's MMAs, copies or
    // arrivals may still reach it.
    cluster_sync();
  }
  tc_fence_after();
  if (warp == 0) {
    if (PAIR)
      tmem_dealloc_pair(tmem, C::TMEM_COLS);
    else
      tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

}  // namespace da
