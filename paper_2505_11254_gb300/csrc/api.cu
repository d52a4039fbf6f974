// api.cu — the C ABI of libdeltaattn.so (declared in include/delta_attn.h):
// argument validation, workspace planning, TMA descriptor encoding and the
// launch sequence of the Delta Attention prefill (arXiv 2505.11254, Alg. 1).
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <mutex>

#include <nvtx3/nvToolsExt.h>

#include "delta_attn.h"
#include "launch.h"
#include "plan.h"
#include "tiles.cuh"
#include "wait.cuh"

using namespace da;

// Per-device status word written by kernels that give up a bounded wait.
__device__ int g_da_status;

namespace {

// A named NVTX range over one call of the C ABI (the kernels it launches show
// under it in a profiler; ncu --nvtx --nvtx-include "<name>/" selects them).
// Header-only NVTX: without a tool attached a push or pop is a null check.
struct NvtxScope {
  explicit NvtxScope(const char* name) { nvtxRangePushA(name); }
  ~NvtxScope() { nvtxRangePop(); }
  NvtxScope(const NvtxScope&) = delete;
  NvtxScope& operator=(const NvtxScope&) = delete;
};

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<EncodeTiledFn>(p);
  }();
  return fn;
}

// 3-D bf16 tensor map, 128-byte swizzle, boxes of 64 x box1 x box2 elements.
// dim0 = d (contiguous), dim1 stride and dim2 stride in bytes.
bool make_map(CUtensorMap* m, const void* base, long long d, long long dim1, long long stride1, long long dim2,
              long long stride2, int box1, int box2) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)dim1, (cuuint64_t)dim2};
  cuuint64_t strides[2] = {(cuuint64_t)stride1, (cuuint64_t)stride2};
  cuuint32_t box[3] = {64, (cuuint32_t)box1, (cuuint32_t)box2};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int check_device(int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DA_ERR_CUDA;
  int major = 0, minor = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return DA_ERR_CUDA;
  if (major != 10 || minor != 3) return DA_ERR_UNSUPPORTED;
  return DA_OK;
}

int check_shape(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma) {
  if (B < 1 || Hq < 1 || Hkv < 1 || N < 1 || gamma < 1 || window < 1 || n_sink < 0) return DA_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return DA_ERR_INVALID_ARG;
  if (N > (int64_t(1) << 31) - 256) return DA_ERR_INVALID_ARG;
  if ((int64_t)B * Hq > (int64_t(1) << 30)) return DA_ERR_INVALID_ARG;
  if (d != 64 && d != 128) return DA_ERR_UNSUPPORTED;
  return DA_OK;
}

struct Plan {
  Params p;
  bool fused_intile = false;
  long long grid_sparse = 0, grid_dense = 0, grid_ssparse = 0;
  size_t off_d = 0, off_delta = 0, off_part = 0, off_ticket = 0, total = 0;
  size_t dense_part = 0, dense_ticket = 0, dense_total = 0;  // strided_dense_attn on its own
  // Dense tail block: the rows N - tail .. N - 1 as dense causal attention,
  // run as a strided-dense pass with gamma = 1 starting at row N - tail.
  long long tail = 0;
  Params pt;
  size_t off_tail_part = 0, off_tail_ticket = 0;
  // Delta smoothing: basis vectors per sample and the per-offset coefficients.
  bool smooth = false;
  size_t off_basis = 0, off_coef = 0;
  int n_coef = 0;
};

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// N: the end of the rows computed; q_row0: their first row (a row-range call
// computes rows [q_row0, N) of a longer sequence; 0 for a whole sequence).
Plan make_plan(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma, int sms,
               int64_t tail = 0, bool smooth = false, int64_t q_row0 = 0) {
  Plan pl;
  Params& p = pl.p;
  p = Params{};
  p.B = B;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.G = Hq / Hkv;
  p.N = N;
  p.n_sink = n_sink;
  p.window = window;
  p.gamma = gamma;
  p.q_row0 = q_row0;
  p.o_rows = N - q_row0;
  p.row0 = q_row0;
  p.n_s = cdiv(N - q_row0, gamma);
  p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)d));
  packing(p.G, &p.Hp, &p.R);
  p.groups_per_b = Hq / p.Hp;
  // Rows of the dense tail are recomputed densely afterwards, so the sparse
  // pass stops at the q-tile holding row N - tail - 1.
  p.qtiles = cdiv(N - tail - q_row0, BM);
  plan_split_k(p, sms, d);

  pl.grid_sparse = (long long)B * Hq * p.qtiles;
  pl.grid_dense = p.n_units;
  pl.fused_intile = gamma >= 2 && (BM % gamma) == 0 && (size_t)(BM / gamma) * d * sizeof(float) <= kSampleBufBytes;
  // Smoothing needs every Delta before any row is corrected: Delta is built
  // in its own pass, for gamma = 1 as well.
  pl.smooth = smooth;
  pl.grid_ssparse = ((gamma >= 2 && !pl.fused_intile) || smooth) ? (long long)B * p.groups_per_b * p.mtiles : 0;

  const size_t rows_bytes = (size_t)B * Hq * p.n_s * d * sizeof(float);
  const size_t part_bytes = (size_t)p.n_multi * BM * (d + 2) * sizeof(float);
  const size_t ticket_bytes = ctrl_bytes(p);
  size_t off = 0;
  if (gamma >= 2 || smooth) {
    pl.off_d = off;
    off += align256(rows_bytes);
    if (!pl.fused_intile || smooth) {
      pl.off_delta = off;
      off += align256(rows_bytes);
    }
  }
  if (smooth) {
    pl.n_coef = (int)std::min<int64_t>(gamma, N);
    pl.off_basis = off;
    off += align256(rows_bytes * kSmoothJ);
    pl.off_coef = off;
    off += align256((size_t)pl.n_coef * kSmoothJ * sizeof(float));
  }
  pl.off_part = off;
  off += align256(part_bytes);
  pl.off_ticket = off;
  off += align256(ticket_bytes);
  if (tail > 0 && (gamma >= 2 || smooth)) {
    pl.tail = tail;
    Params& t = pl.pt;
    t = p;
    t.gamma = 1;
    t.n_s = tail;
    t.row0 = N - tail;
    plan_split_k(t, sms, d);
    pl.off_tail_part = off;
    off += align256((size_t)t.n_multi * BM * (d + 2) * sizeof(float));
    pl.off_tail_ticket = off;
    off += align256(ctrl_bytes(t));
  }
  pl.total = off;
  pl.dense_part = 0;
  pl.dense_ticket = align256(part_bytes);
  pl.dense_total = align256(part_bytes) + align256(ticket_bytes);
  return pl;
}

// The device address of the status word on the current device, looked up
// once per device (with that device current) on the first call that needs it;
// later calls only read the cached address.
constexpr int kMaxStatusDevices = 64;
int* g_status_addr[kMaxStatusDevices];
cudaError_t g_status_err[kMaxStatusDevices];
std::once_flag g_status_once[kMaxStatusDevices];

int status_ptr(int** ptr) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DA_ERR_CUDA;
  if (dev < 0 || dev >= kMaxStatusDevices) return DA_ERR_UNSUPPORTED;
  std::call_once(g_status_once[dev], [dev] {
    void* a = nullptr;
    g_status_err[dev] = cudaGetSymbolAddress(&a, g_da_status);
    g_status_addr[dev] = g_status_err[dev] == cudaSuccess ? static_cast<int*>(a) : nullptr;
  });
  if (g_status_err[dev] != cudaSuccess || g_status_addr[dev] == nullptr) return DA_ERR_CUDA;
  *ptr = g_status_addr[dev];
  return DA_OK;
}

struct Maps {
  CUtensorMap q, qs, k, v;
  CUtensorMap kh;  // K in boxes of BN / 2 rows: the two-CTA sink + window kernel (pair_sparse)
};

// The sink + window pass of a whole sequence runs as the two-CTA kernel when
// the query heads of each KV group pair up (G even) at d = 128 and the window
// spans at least 4 key tiles.  Measured on GB300 against the one-CTA kernel:
// the same time per prefill at windows 512, 2048 and 8192, at a higher
// sustained clock under the power cap (it moves half the K/V bytes through
// each SM's shared memory and from L2); shorter windows were not measured.
// Results are bit-identical.  The environment variable DELTA_ATTN_PAIR
// overrides the choice: 0 always takes the one-CTA kernel, 1 the two-CTA one
// where it applies.
bool pair_sparse(int d, const Params& p) {
  if (d != 128 || p.G % 2 != 0 || p.q_row0 != 0) return false;
  const char* env = getenv("DELTA_ATTN_PAIR");
  if (env != nullptr && env[0] == '0') return false;
  if (env != nullptr && env[0] == '1') return true;
  return p.window >= 4 * BN;
}

// Sampled rows row0 + k * gamma of every (b, head): Hp heads x R samples a box.
// Q holds rows q_row0 .. N - 1 of every (b, head); sample k is row row0 + k gamma.
bool make_sample_map(CUtensorMap* m, const void* Q, const Params& p, int d) {
  const long long row_bytes = (long long)d * 2;
  const uint8_t* base = static_cast<const uint8_t*>(Q) + (p.row0 - p.q_row0) * row_bytes;
  return make_map(m, base, d, p.n_s, row_bytes * p.gamma, (long long)p.B * p.Hq, (p.N - p.q_row0) * row_bytes, p.R,
                  p.Hp);
}

// n_kv: rows K and V hold per (b, KV head), at least p.N.
bool make_maps(Maps* m, const void* Q, const void* K, const void* V, const Params& p, int d, bool need_rows,
               bool need_samples, long long n_kv) {
  const long long row_bytes = (long long)d * 2;
  const long long q_rows = p.N - p.q_row0;
  if (need_rows && !make_map(&m->q, Q, d, q_rows, row_bytes, (long long)p.B * p.Hq, q_rows * row_bytes, BM, 1))
    return false;
  if (need_samples && !make_sample_map(&m->qs, Q, p, d)) return false;
  if (!make_map(&m->k, K, d, n_kv, row_bytes, (long long)p.B * p.Hkv, n_kv * row_bytes, BN, 1)) return false;
  if (!make_map(&m->v, V, d, n_kv, row_bytes, (long long)p.B * p.Hkv, n_kv * row_bytes, BN, 1)) return false;
  if (need_rows && pair_sparse(d, p) &&
      !make_map(&m->kh, K, d, n_kv, row_bytes, (long long)p.B * p.Hkv, n_kv * row_bytes, BN / 2, 1))
    return false;
  return true;
}

template <int MODE, int EPI>
cudaError_t launch(int d, const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v, const Params& p,
                   long long grid, cudaStream_t s) {
  if (d == 64) return launch_attn<64, MODE, EPI>(q, k, v, p, grid, s);
  return launch_attn<128, MODE, EPI>(q, k, v, p, grid, s);
}

// The sink + window pass: the two-CTA kernel where pair_sparse() allows it,
// the ROWS instance for a row-range call whose range starts after row 0, the
// one-CTA whole-sequence kernel otherwise.
template <int EPI>
cudaError_t launch_sparse(int d, const Maps& m, const Params& p, long long grid, cudaStream_t s) {
  if (pair_sparse(d, p)) {
    const cudaError_t e = launch_attn<128, MODE_SPARSE, EPI, false, true>(m.q, m.kh, m.v, p, grid, s);
    if (e != cudaErrorNotSupported) return e;  // else no cluster of two fits: the one-CTA kernel below
  }
  if (p.q_row0 == 0) return launch<MODE_SPARSE, EPI>(d, m.q, m.k, m.v, p, grid, s);
  // Row ranges are Eq. 6 prefills only (delta_attn_prefill_rows).
  if constexpr (EPI == EPI_FUSED_INTILE || EPI == EPI_FUSED_DELTA) {
    if (d == 64) return launch_attn<64, MODE_SPARSE, EPI, true>(m.q, m.k, m.v, p, grid, s);
    return launch_attn<128, MODE_SPARSE, EPI, true>(m.q, m.k, m.v, p, grid, s);
  }
  return cudaErrorInvalidValue;
}

class ScopedWorkspace {
 public:
  ScopedWorkspace(void* user, size_t bytes, cudaStream_t s) : s_(s) {
    if (user != nullptr || bytes == 0) {
      ptr_ = user;
      return;
    }
    if (cudaMallocAsync(&ptr_, bytes, s) != cudaSuccess) ptr_ = nullptr;
    owned_ = ptr_ != nullptr;
    failed_ = !owned_;
  }
  ~ScopedWorkspace() {
    if (owned_) cudaFreeAsync(ptr_, s_);
  }
  bool failed() const { return failed_; }
  uint8_t* get() const { return static_cast<uint8_t*>(ptr_); }

 private:
  void* ptr_ = nullptr;
  cudaStream_t s_;
  bool owned_ = false, failed_ = false;
};

struct SmoothArgs {
  int kind = DA_SMOOTH_NONE;
  double c1 = 0, c2 = 0, c3 = 0;
};

int check_smooth(const SmoothArgs& sm, int mode) {
  if (sm.kind < DA_SMOOTH_NONE || sm.kind > DA_SMOOTH_ABG) return DA_ERR_INVALID_ARG;
  if (sm.kind != DA_SMOOTH_NONE && mode != DA_MODE_DELTA) return DA_ERR_INVALID_ARG;
  if (!std::isfinite(sm.c1) || !std::isfinite(sm.c2) || !std::isfinite(sm.c3)) return DA_ERR_INVALID_ARG;
  if (sm.kind == DA_SMOOTH_EMA && !(sm.c1 >= 0.0 && sm.c1 <= 1.0)) return DA_ERR_INVALID_ARG;
  return DA_OK;
}

// Split of the decode's key range: one wave of resident CTAs (the occupancy
// of the kernel instance) over all (batch, KV head) pairs, each range a whole
// number of ring chunks.
struct DecodePlan {
  int n_split = 1;
  long long split_keys = 0;
  size_t bytes = 0;
};

int check_decode(int B, int Hq, int Hkv, int64_t L, int64_t max_keys, int d) {
  if (B < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || max_keys < 1 || L < max_keys) return DA_ERR_INVALID_ARG;
  if ((int64_t)B * Hq > (int64_t(1) << 30) || L > (int64_t(1) << 40)) return DA_ERR_INVALID_ARG;
  if (d != 64 && d != 128) return DA_ERR_UNSUPPORTED;
  if (Hq / Hkv > 16) return DA_ERR_UNSUPPORTED;
  return DA_OK;
}

DecodePlan make_decode_plan(int B, int Hq, int Hkv, int64_t max_keys, int d, int sms) {
  DecodePlan dp;
  const long long chunk = decode_keys_per_split(d, Hq / Hkv);
  const long long chunks = cdiv(max_keys, chunk);
  const long long pairs = (long long)B * Hkv;
  // at most one wave: a second, partial wave would run alone at the end
  long long n = ((long long)decode_ctas_per_sm(d, Hq / Hkv) * std::max(sms, 1)) / pairs;
  n = std::max<long long>(1, std::min(n, chunks));
  dp.split_keys = cdiv(chunks, n) * chunk;
  dp.n_split = (int)cdiv(max_keys, dp.split_keys);
  dp.bytes = align256((size_t)pairs * dp.n_split * (Hq / Hkv) * (d + 2) * sizeof(float));
  return dp;
}

int check_variant(int mode, int64_t tail, int64_t N) {
  if (mode != DA_MODE_DELTA && mode != DA_MODE_RECOMPUTE) return DA_ERR_INVALID_ARG;
  if (tail < 0 || tail > N) return DA_ERR_INVALID_ARG;
  return DA_OK;
}

// Kernel launches of one prefill call, in order.
int prefill_kernels(const Plan& pl, int gamma, int mode) {
  const int tail = pl.tail > 0 ? 1 : 0;
  if (pl.smooth) return 4 + tail;
  if (gamma == 1) return 1;
  if (mode == DA_MODE_RECOMPUTE) return 2 + tail;
  return (pl.fused_intile ? 2 : 3) + tail;
}

}  // namespace

extern "C" {

const char* delta_attn_status_string(int status) {
  switch (status) {
    case DA_OK: return "ok";
    case DA_ERR_INVALID_ARG: return "invalid argument";
    case DA_ERR_UNSUPPORTED: return "unsupported head dimension or device (needs d in {64,128} and sm_103)";
    case DA_ERR_MISALIGNED: return "pointer not 16-byte aligned";
    case DA_ERR_WORKSPACE: return "workspace too small";
    case DA_ERR_CUDA: return "CUDA error";
    case DA_ERR_TIMEOUT: return "kernel gave up a bounded wait";
    default: return "unknown status";
  }
}

int delta_attn_workspace_size(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                              size_t* bytes) {
  if (!bytes) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, n_sink, window, gamma);
  if (rc) return rc;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  *bytes = make_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, sms).total;
  return DA_OK;
}

int delta_attn_workspace_size_ex(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                                 int mode, int64_t tail_dense, size_t* bytes) {
  if (!bytes) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, n_sink, window, gamma);
  if (rc) return rc;
  if ((rc = check_variant(mode, tail_dense, N))) return rc;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  *bytes = make_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, sms, tail_dense).total;
  return DA_OK;
}

int delta_attn_workspace_size_smoothed(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window,
                                       int gamma, int smooth, int64_t tail_dense, size_t* bytes) {
  if (!bytes) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, n_sink, window, gamma);
  if (rc) return rc;
  if ((rc = check_variant(DA_MODE_DELTA, tail_dense, N))) return rc;
  if (smooth < DA_SMOOTH_NONE || smooth > DA_SMOOTH_ABG) return DA_ERR_INVALID_ARG;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  *bytes = make_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, sms, tail_dense, smooth != DA_SMOOTH_NONE).total;
  return DA_OK;
}

int strided_dense_workspace_size(int B, int Hq, int Hkv, int64_t N, int d, int gamma, size_t* bytes) {
  if (!bytes) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, 0, 1, gamma);
  if (rc) return rc;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  *bytes = make_plan(B, Hq, Hkv, N, d, 0, 1, gamma, sms).dense_total;
  return DA_OK;
}

int delta_attn_plan_info(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                         int64_t* info) {
  if (!info) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, n_sink, window, gamma);
  if (rc) return rc;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  Plan pl = make_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, sms);
  info[0] = gamma == 1 ? 0 : pl.grid_sparse;
  info[1] = pl.grid_dense;
  info[2] = pl.grid_ssparse;
  info[3] = pl.p.chunk;
  info[4] = pl.p.n_multi;
  info[5] = pl.p.Hp;
  info[6] = pl.p.R;
  info[7] = pl.fused_intile ? 1 : 0;
  info[8] = gamma == 1 ? 1 : (pl.fused_intile ? 2 : 3);
  info[9] = sms;
  return DA_OK;
}

// rope: a (cos, sin) table [>= N][d/2][2] when Q and K come unrotated; K is
// then rotated in place before the first kernel and every Q tile on its way
// into tensor memory.
// A row range of a longer sequence (delta_attn_prefill_rows): rows
// [q_row0, N) with K and V of n_kv rows; {0, 0} for a whole sequence.
struct RowRange {
  int64_t q_row0 = 0, n_kv = 0;
};

static int check_rows(int64_t N_kv, int gamma, int64_t row_begin, int64_t n_rows) {
  if (row_begin < 0 || n_rows < 1 || gamma < 1 || row_begin > N_kv - n_rows) return DA_ERR_INVALID_ARG;
  if (row_begin % BM != 0 || row_begin % gamma != 0) return DA_ERR_INVALID_ARG;
  return DA_OK;
}

static int prefill_impl(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv, int64_t N,
                        int d, int n_sink, int64_t window, int gamma, int mode, int64_t tail, const SmoothArgs& sm,
                        void* workspace, size_t ws_bytes, void* stream, void* const* events, int n_events,
                        const float* rope = nullptr, RowRange rr = RowRange{}) {
  if (!Q || !K || !V || !O) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, n_sink, window, gamma);
  if (rc) return rc;
  if ((rc = check_variant(mode, tail, N))) return rc;
  if ((rc = check_smooth(sm, mode))) return rc;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O) || !aligned16(workspace) ||
      !aligned16(rope))
    return DA_ERR_MISALIGNED;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  const bool smooth = sm.kind != DA_SMOOTH_NONE;
  Plan pl = make_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, sms, tail, smooth, rr.q_row0);
  // A row range: the passes that index O by absolute row, and the per-sample
  // buffers by absolute sample, get base pointers moved back by the range's
  // first row (sample), so the kernels' indexing is that of a whole sequence.
  // Only rows and samples inside the range are ever addressed through them.
  const long long s_off = rr.q_row0 / gamma;
  void* const O_abs = static_cast<uint8_t*>(O) - rr.q_row0 * (long long)d * 2;
  auto abs_samples = [&](float* f) { return f - s_off * d; };
  const int n_kernels = prefill_kernels(pl, gamma, mode);
  if (n_events != 0 && (events == nullptr || n_events != n_kernels + 1)) return DA_ERR_INVALID_ARG;
  if (workspace != nullptr && ws_bytes < pl.total) return DA_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Params p = pl.p;
  if ((rc = status_ptr(&p.err))) return rc;
  Maps m;
  if (!make_maps(&m, Q, K, V, p, d, gamma >= 2 || smooth, true, rr.n_kv > 0 ? rr.n_kv : N))
    return DA_ERR_INVALID_ARG;
  CUtensorMap q_tail;
  if (pl.tail > 0 && !make_sample_map(&q_tail, Q, pl.pt, d)) return DA_ERR_INVALID_ARG;

  ScopedWorkspace ws(workspace, pl.total, s);
  if (ws.failed()) return DA_ERR_CUDA;
  if (rope != nullptr) {
    if (launch_rope_apply(const_cast<void*>(K), (long long)B * Hkv * N, N, d, 0, rope, s) != cudaSuccess)
      return DA_ERR_CUDA;
    p.rope = rope;
  }
  uint8_t* base = ws.get();
  p.partials = reinterpret_cast<float*>(base + pl.off_part);
  p.counter = reinterpret_cast<unsigned long long*>(base + pl.off_ticket);
  p.tickets = reinterpret_cast<int*>(base + pl.off_ticket + 4 * sizeof(unsigned long long));
  if (cudaMemsetAsync(p.counter, 0, ctrl_bytes(p), s) != cudaSuccess) return DA_ERR_CUDA;
  Params pt = pl.pt;
  if (pl.tail > 0) {
    pt.err = p.err;
    pt.rope = p.rope;
    pt.partials = reinterpret_cast<float*>(base + pl.off_tail_part);
    pt.counter = reinterpret_cast<unsigned long long*>(base + pl.off_tail_ticket);
    pt.tickets = reinterpret_cast<int*>(base + pl.off_tail_ticket + 4 * sizeof(unsigned long long));
    pt.out_bf16 = O;
    if (cudaMemsetAsync(pt.counter, 0, ctrl_bytes(pt), s) != cudaSuccess) return DA_ERR_CUDA;
  }

  int ev = 0;
  auto mark = [&]() -> bool {
    return n_events == 0 || cudaEventRecord(static_cast<cudaEvent_t>(events[ev++]), s) == cudaSuccess;
  };
  // Appendix "Implementation Details": the final block of rows is replaced
  // by dense rows, after every pass that writes rows of O.
  auto run_tail = [&]() -> int {
    if (pl.tail == 0) return DA_OK;
    cudaError_t e = launch<MODE_STRIDED_DENSE, EPI_DENSE_BF16>(d, q_tail, m.k, m.v, pt, pt.n_units, s);
    return (e == cudaSuccess && mark()) ? DA_OK : DA_ERR_CUDA;
  };
  if (!mark()) return DA_ERR_CUDA;
  cudaError_t e;
  if (smooth) {
    // Appendix "Interpolation": D, then every Delta_k, then the smoothing
    // pass, then the sink+window pass adding the smoothed correction to
    // every row (sampled rows included).
    float* dbuf = reinterpret_cast<float*>(base + pl.off_d);
    float* delta = reinterpret_cast<float*>(base + pl.off_delta);
    float* basis = reinterpret_cast<float*>(base + pl.off_basis);
    float* coef = reinterpret_cast<float*>(base + pl.off_coef);
    p.d_out = dbuf;
    e = launch<MODE_STRIDED_DENSE, EPI_DENSE_F32>(d, m.qs, m.k, m.v, p, pl.grid_dense, s);
    if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
    p.d_out = nullptr;
    p.d_in = dbuf;
    p.delta_out = delta;
    e = launch<MODE_STRIDED_SPARSE, EPI_DELTA_BUILD>(d, m.qs, m.k, m.v, p, pl.grid_ssparse, s);
    if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
    p.delta_out = nullptr;
    e = launch_delta_smooth(delta, basis, coef, (long long)B * Hq, p.n_s, d, gamma, pl.n_coef, sm.kind, sm.c1, sm.c2,
                            sm.c3, s);
    if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
    p.out_bf16 = O_abs;
    p.smooth_basis = basis - s_off * kSmoothJ * d;  // kSmoothJ vectors per sample
    p.smooth_coef = coef;
    e = launch_sparse<EPI_FUSED_SMOOTH>(d, m, p, pl.grid_sparse, s);
    if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
    return run_tail();
  }
  if (gamma == 1) {
    // Every row is a sampled row: the output is dense causal attention.
    p.out_bf16 = O_abs;
    e = launch<MODE_STRIDED_DENSE, EPI_DENSE_BF16>(d, m.qs, m.k, m.v, p, pl.grid_dense, s);
    return (e == cudaSuccess && mark()) ? DA_OK : DA_ERR_CUDA;
  }
  if (mode == DA_MODE_RECOMPUTE) {
    // Eq. 5: sparse rows everywhere, then the sampled rows overwritten by
    // their dense rows; no correction reaches the other rows.
    p.out_bf16 = O_abs;
    e = launch_sparse<EPI_BF16>(d, m, p, pl.grid_sparse, s);
    if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
    e = launch<MODE_STRIDED_DENSE, EPI_DENSE_BF16>(d, m.qs, m.k, m.v, p, pl.grid_dense, s);
    if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
    return run_tail();
  }
  float* dbuf = reinterpret_cast<float*>(base + pl.off_d);
  p.d_out = dbuf;
  e = launch<MODE_STRIDED_DENSE, EPI_DENSE_F32>(d, m.qs, m.k, m.v, p, pl.grid_dense, s);
  if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
  p.d_out = nullptr;
  p.out_bf16 = O_abs;
  if (pl.fused_intile) {
    p.d_in = abs_samples(dbuf);
    e = launch_sparse<EPI_FUSED_INTILE>(d, m, p, pl.grid_sparse, s);
  } else {
    float* delta = reinterpret_cast<float*>(base + pl.off_delta);
    p.d_in = dbuf;  // the strided sparse pass indexes its own samples
    p.delta_out = delta;
    e = launch<MODE_STRIDED_SPARSE, EPI_DELTA_BUILD>(d, m.qs, m.k, m.v, p, pl.grid_ssparse, s);
    if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
    p.delta_out = nullptr;
    p.d_in = abs_samples(dbuf);
    p.delta_in = abs_samples(delta);
    e = launch_sparse<EPI_FUSED_DELTA>(d, m, p, pl.grid_sparse, s);
  }
  if (e != cudaSuccess || !mark()) return DA_ERR_CUDA;
  return run_tail();
}

int delta_attn_prefill(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv, int64_t N,
                       int d, int n_sink, int64_t window, int gamma, void* workspace, size_t ws_bytes,
                       void* stream) {
  NvtxScope nvtx_scope("delta_attn_prefill");
  return prefill_impl(Q, K, V, O, B, Hq, Hkv, N, d, n_sink, window, gamma, DA_MODE_DELTA, 0, SmoothArgs{},
                      workspace, ws_bytes, stream, nullptr, 0);
}

int delta_attn_prefill_ex(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv, int64_t N,
                          int d, int n_sink, int64_t window, int gamma, int mode, int64_t tail_dense,
                          void* workspace, size_t ws_bytes, void* stream) {
  NvtxScope nvtx_scope("delta_attn_prefill_ex");
  return prefill_impl(Q, K, V, O, B, Hq, Hkv, N, d, n_sink, window, gamma, mode, tail_dense, SmoothArgs{},
                      workspace, ws_bytes, stream, nullptr, 0);
}

int delta_attn_prefill_smoothed(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv,
                                int64_t N, int d, int n_sink, int64_t window, int gamma, int smooth, double c1,
                                double c2, double c3, int64_t tail_dense, void* workspace, size_t ws_bytes,
                                void* stream) {
  NvtxScope nvtx_scope("delta_attn_prefill_smoothed");
  SmoothArgs sm;
  sm.kind = smooth;
  sm.c1 = c1;
  sm.c2 = c2;
  sm.c3 = c3;
  return prefill_impl(Q, K, V, O, B, Hq, Hkv, N, d, n_sink, window, gamma, DA_MODE_DELTA, tail_dense, sm, workspace,
                      ws_bytes, stream, nullptr, 0);
}

int delta_attn_prefill_events(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv,
                              int64_t N, int d, int n_sink, int64_t window, int gamma, void* workspace,
                              size_t ws_bytes, void* stream, void* const* events, int n_events) {
  NvtxScope nvtx_scope("delta_attn_prefill_events");
  return prefill_impl(Q, K, V, O, B, Hq, Hkv, N, d, n_sink, window, gamma, DA_MODE_DELTA, 0, SmoothArgs{},
                      workspace, ws_bytes, stream, events,
                      n_events);
}

int sparse_window_attn(const void* Q, const void* K, const void* V, void* O_sparse, float* S_sampled, int B,
                       int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma, void* stream) {
  NvtxScope nvtx_scope("sparse_window_attn");
  if (!Q || !K || !V || !O_sparse) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, n_sink, window, gamma);
  if (rc) return rc;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O_sparse) || !aligned16(S_sampled))
    return DA_ERR_MISALIGNED;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  Plan pl = make_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, sms);
  Params p = pl.p;
  if ((rc = status_ptr(&p.err))) return rc;
  Maps m;
  if (!make_maps(&m, Q, K, V, p, d, true, false, N)) return DA_ERR_INVALID_ARG;
  p.out_bf16 = O_sparse;
  p.s_sampled = S_sampled;
  cudaError_t e = launch_sparse<EPI_BF16>(d, m, p, pl.grid_sparse, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? DA_OK : DA_ERR_CUDA;
}

int strided_dense_attn(const void* Q, const void* K, const void* V, float* D_sampled, int B, int Hq, int Hkv,
                       int64_t N, int d, int gamma, void* workspace, size_t ws_bytes, void* stream) {
  NvtxScope nvtx_scope("strided_dense_attn");
  if (!Q || !K || !V || !D_sampled) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, 0, 1, gamma);
  if (rc) return rc;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(D_sampled) || !aligned16(workspace))
    return DA_ERR_MISALIGNED;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  Plan pl = make_plan(B, Hq, Hkv, N, d, 0, 1, gamma, sms);
  if (workspace != nullptr && ws_bytes < pl.dense_total) return DA_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Params p = pl.p;
  if ((rc = status_ptr(&p.err))) return rc;
  Maps m;
  if (!make_maps(&m, Q, K, V, p, d, false, true, N)) return DA_ERR_INVALID_ARG;
  ScopedWorkspace ws(workspace, pl.dense_total, s);
  if (ws.failed()) return DA_ERR_CUDA;
  p.partials = reinterpret_cast<float*>(ws.get() + pl.dense_part);
  p.counter = reinterpret_cast<unsigned long long*>(ws.get() + pl.dense_ticket);
  p.tickets = reinterpret_cast<int*>(ws.get() + pl.dense_ticket + 4 * sizeof(unsigned long long));
  if (cudaMemsetAsync(p.counter, 0, 4 * sizeof(unsigned long long) + p.n_multi * sizeof(int), s) != cudaSuccess)
    return DA_ERR_CUDA;
  p.d_out = D_sampled;
  cudaError_t e = launch<MODE_STRIDED_DENSE, EPI_DENSE_F32>(d, m.qs, m.k, m.v, p, pl.grid_dense, s);
  return e == cudaSuccess ? DA_OK : DA_ERR_CUDA;
}

int delta_apply(const void* O_sparse, const float* S_sampled, const float* D_sampled, void* O, int B, int Hq,
                int64_t N, int d, int gamma, void* stream) {
  NvtxScope nvtx_scope("delta_apply");
  if (!O_sparse || !D_sampled || !O) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hq, N, d, 0, 1, gamma);
  if (rc) return rc;
  if (!aligned16(O_sparse) || !aligned16(S_sampled) || !aligned16(D_sampled) || !aligned16(O))
    return DA_ERR_MISALIGNED;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  cudaError_t e = launch_delta_apply(O_sparse, S_sampled, D_sampled, O, B, Hq, N, d, gamma,
                                     static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? DA_OK : DA_ERR_CUDA;
}

int delta_attn_decode_workspace_size(int B, int Hq, int Hkv, int64_t max_keys, int d, size_t* bytes) {
  if (!bytes) return DA_ERR_INVALID_ARG;
  int rc = check_decode(B, Hq, Hkv, max_keys, max_keys, d);
  if (rc) return rc;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  *bytes = make_decode_plan(B, Hq, Hkv, max_keys, d, sms).bytes;
  return DA_OK;
}

int delta_attn_decode(const void* q, const void* K, const void* V, const int64_t* lens, void* O, int B, int Hq,
                      int Hkv, int64_t L, int64_t max_keys, int d, void* workspace, size_t ws_bytes, void* stream) {
  NvtxScope nvtx_scope("delta_attn_decode");
  if (!q || !K || !V || !O) return DA_ERR_INVALID_ARG;
  int rc = check_decode(B, Hq, Hkv, L, max_keys, d);
  if (rc) return rc;
  if (!aligned16(q) || !aligned16(K) || !aligned16(V) || !aligned16(O) || !aligned16(workspace))
    return DA_ERR_MISALIGNED;
  if ((reinterpret_cast<uintptr_t>(lens) & 7u) != 0) return DA_ERR_MISALIGNED;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  const DecodePlan dp = make_decode_plan(B, Hq, Hkv, max_keys, d, sms);
  if (workspace != nullptr && ws_bytes < dp.bytes) return DA_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DecodeParams p{};
  if ((rc = status_ptr(&p.err))) return rc;
  ScopedWorkspace ws(workspace, dp.bytes, s);
  if (ws.failed()) return DA_ERR_CUDA;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.K = static_cast<const __nv_bfloat16*>(K);
  p.V = static_cast<const __nv_bfloat16*>(V);
  p.lens = reinterpret_cast<const long long*>(lens);
  p.max_keys = max_keys;
  p.L = L;
  p.B = B;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.G = Hq / Hkv;
  p.D = d;
  p.n_split = dp.n_split;
  p.split_keys = dp.split_keys;
  p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)d));
  p.part = reinterpret_cast<float*>(ws.get());
  return launch_decode(p, O, s) == cudaSuccess ? DA_OK : DA_ERR_CUDA;
}

int delta_attn_rope_table(int64_t n_pos, int d, double base, float* table, void* stream) {
  NvtxScope nvtx_scope("delta_attn_rope_table");
  if (!table || n_pos < 1 || n_pos > (int64_t(1) << 34) || !(base > 0.0) || !std::isfinite(base))
    return DA_ERR_INVALID_ARG;
  if (d != 64 && d != 128) return DA_ERR_UNSUPPORTED;
  if (!aligned16(table)) return DA_ERR_MISALIGNED;
  return launch_rope_table(n_pos, d, base, table, static_cast<cudaStream_t>(stream)) == cudaSuccess ? DA_OK
                                                                                                  : DA_ERR_CUDA;
}

int delta_attn_rope_apply(void* X, int B, int H, int64_t N, int d, int64_t pos0, const float* table,
                          int64_t table_rows, void* stream) {
  NvtxScope nvtx_scope("delta_attn_rope_apply");
  if (!X || !table || B < 1 || H < 1 || N < 1 || pos0 < 0 || (int64_t)B * H > (int64_t(1) << 30))
    return DA_ERR_INVALID_ARG;
  if (d != 64 && d != 128) return DA_ERR_UNSUPPORTED;
  if (pos0 + N > table_rows) return DA_ERR_INVALID_ARG;  // the table must cover every position
  if (!aligned16(X) || !aligned16(table)) return DA_ERR_MISALIGNED;
  return launch_rope_apply(X, (long long)B * H * N, N, d, pos0, table, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? DA_OK
             : DA_ERR_CUDA;
}

int delta_attn_prefill_rope(const void* Q, void* K, const void* V, void* O, int B, int Hq, int Hkv, int64_t N, int d,
                            int n_sink, int64_t window, int gamma, const float* table, int64_t table_rows,
                            void* workspace, size_t ws_bytes, void* stream) {
  NvtxScope nvtx_scope("delta_attn_prefill_rope");
  if (!table || table_rows < N) return DA_ERR_INVALID_ARG;
  return prefill_impl(Q, K, V, O, B, Hq, Hkv, N, d, n_sink, window, gamma, DA_MODE_DELTA, 0, SmoothArgs{},
                      workspace, ws_bytes, stream, nullptr, 0, table);
}

int delta_attn_workspace_size_rows(int B, int Hq, int Hkv, int64_t N_kv, int d, int n_sink, int64_t window,
                                   int gamma, int64_t row_begin, int64_t n_rows, size_t* bytes) {
  if (!bytes) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N_kv, d, n_sink, window, gamma);
  if (rc) return rc;
  if ((rc = check_rows(N_kv, gamma, row_begin, n_rows))) return rc;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  *bytes = make_plan(B, Hq, Hkv, row_begin + n_rows, d, n_sink, window, gamma, sms, 0, false, row_begin).total;
  return DA_OK;
}

int delta_attn_prefill_rows(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv,
                            int64_t N_kv, int d, int n_sink, int64_t window, int gamma, int64_t row_begin,
                            int64_t n_rows, void* workspace, size_t ws_bytes, void* stream) {
  NvtxScope nvtx_scope("delta_attn_prefill_rows");
  int rc = check_shape(B, Hq, Hkv, N_kv, d, n_sink, window, gamma);
  if (rc) return rc;
  if ((rc = check_rows(N_kv, gamma, row_begin, n_rows))) return rc;
  return prefill_impl(Q, K, V, O, B, Hq, Hkv, row_begin + n_rows, d, n_sink, window, gamma, DA_MODE_DELTA, 0,
                      SmoothArgs{}, workspace, ws_bytes, stream, nullptr, 0, nullptr, RowRange{row_begin, N_kv});
}

int delta_attn_check(void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return DA_ERR_CUDA;
  int v = 0;
  if (cudaMemcpyFromSymbolAsync(&v, g_da_status, sizeof(int), 0, cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return DA_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return DA_ERR_CUDA;
  if (v != 0) {
    const int zero = 0;
    if (cudaMemcpyToSymbolAsync(g_da_status, &zero, sizeof(int), 0, cudaMemcpyHostToDevice, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
      return DA_ERR_CUDA;
  }
  return v;
}

int delta_attn_debug_mask(int64_t N, int n_sink, int64_t window, int64_t i0, int64_t i1, uint8_t* out,
                          void* stream) {
  if (!out || N < 1 || window < 1 || n_sink < 0 || i0 < 0 || i1 <= i0 || i1 > N) return DA_ERR_INVALID_ARG;
  return launch_debug_mask(N, n_sink, window, i0, i1, out, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? DA_OK
             : DA_ERR_CUDA;
}

int delta_attn_debug_rowmap(int64_t N, int gamma, int64_t* sample_row, uint8_t* is_sampled, void* stream) {
  if (!sample_row || !is_sampled || N < 1 || gamma < 1) return DA_ERR_INVALID_ARG;
  return launch_debug_rowmap(N, gamma, reinterpret_cast<long long*>(sample_row), is_sampled,
                             static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? DA_OK
             : DA_ERR_CUDA;
}

int delta_attn_debug_work(int mode, int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window,
                          int gamma, int64_t index, int64_t* out, int max_tiles, void* stream) {
  if (!out || max_tiles < 0 || mode < 0 || mode > 2) return DA_ERR_INVALID_ARG;
  int rc = check_shape(B, Hq, Hkv, N, d, n_sink, window, gamma);
  if (rc) return rc;
  int sms = 0;
  if ((rc = check_device(&sms))) return rc;
  Plan pl = make_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, sms);
  const long long count = mode == 0 ? pl.grid_sparse : mode == 1 ? pl.grid_dense
                                                                 : (long long)B * pl.p.groups_per_b * pl.p.mtiles;
  if (index < 0 || index >= count) return DA_ERR_INVALID_ARG;
  return launch_debug_work(mode, pl.p, index, reinterpret_cast<long long*>(out), max_tiles,
                           static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? DA_OK
             : DA_ERR_CUDA;
}

int delta_attn_debug_timeout(int64_t limit_ns, void* stream) {
  if (limit_ns <= 0 || limit_ns > (int64_t)WAIT_LIMIT_NS) return DA_ERR_INVALID_ARG;
  int* status = nullptr;
  int rc = status_ptr(&status);
  if (rc) return rc;
  return launch_debug_timeout(status, (unsigned long long)limit_ns, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? DA_OK
             : DA_ERR_CUDA;
}

}  // extern "C"
