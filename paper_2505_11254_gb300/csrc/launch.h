// launch.h — host-side declarations of the kernel launchers (instantiated in
// attn_*.cu so the kernels compile in parallel translation units).
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "tiles.cuh"

namespace da {

// ROWS: the instance for row-range calls (rows from Params::q_row0 > 0).
// PAIR: the two-CTA sink + window kernel (d = 128, G even, whole sequences);
// its K map has boxes of BN / 2 rows.
template <int D, int MODE, int EPI, bool ROWS = false, bool PAIR = false>
cudaError_t launch_attn(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv, const Params& p,
                        long long n_items, cudaStream_t s);

// Bytes of the epilogue buffer that holds the sampled sparse rows of one tile
// when the Delta is fused inside the tile.
constexpr unsigned kSampleBufBytes = 8192;

unsigned attn_smem_bytes(int d);

cudaError_t launch_delta_apply(const void* o_sparse, const float* s_sampled, const float* d_sampled, void* o, int B,
                               int Hq, long long N, int d, int gamma, cudaStream_t s);
cudaError_t launch_delta_smooth(const float* delta, float* basis, float* coef, long long BH, long long n_s, int d,
                                int gamma, int n_coef, int kind, double c1, double c2, double c3, cudaStream_t s);
// Eq. 2 decoding over the cache (decode.cu).
struct DecodeParams {
  const __nv_bfloat16* q;  // [B, Hq, D]
  const __nv_bfloat16* K;  // [B, Hkv, L, D]
  const __nv_bfloat16* V;  // [B, Hkv, L, D]
  const long long* lens;   // [B] valid keys per sequence (device), or null: max_keys each
  long long max_keys, L;
  int B, Hq, Hkv, G, D;
  int n_split;             // key ranges per (batch, KV head)
  long long split_keys;    // keys per range, a multiple of decode_keys_per_split(d, G)
  float scale_log2;        // log2(e) / sqrt(D)
  float* part;             // [B * Hkv * n_split][G][D + 2]: unnormalised o, max, sum
  int* err;                // device status word
};
int decode_keys_per_split(int d, int G);  // keys per ring chunk of the kernel instance
int decode_ctas_per_sm(int d, int G);  // resident decode CTAs per SM (occupancy)
cudaError_t launch_decode(const DecodeParams& p, void* out, cudaStream_t s);

// RoPE (rope.cu): the (cos, sin) table [n_pos][d/2] fp32 pairs, and an in-place
// rotation of bf16 rows (row r at position pos0 + r % N).
cudaError_t launch_rope_table(long long n_pos, int d, double base, float* table, cudaStream_t s);
cudaError_t launch_rope_apply(void* x, long long rows, long long N, int d, long long pos0, const float* table,
                              cudaStream_t s);

cudaError_t launch_debug_mask(long long N, int n_sink, long long window, long long i0, long long i1,
                              unsigned char* out, cudaStream_t s);
cudaError_t launch_debug_rowmap(long long N, int gamma, long long* sample_row, unsigned char* sampled,
                                cudaStream_t s);
cudaError_t launch_debug_timeout(int* status, unsigned long long limit_ns, cudaStream_t s);
cudaError_t launch_debug_work(int mode, const Params& p, long long index, long long* out, int max_tiles,
                              cudaStream_t s);

}  // namespace da
