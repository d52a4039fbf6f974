// host_pipeline.cu — delta_attn_prefill_host: the prefill on host buffers,
// with the copies in and out overlapped with the attention kernels.
//
// The attention of one (batch, KV head) group — its G query heads and one
// K/V head — is independent of every other group, so the problem is cut into
// B * Hkv chunks and pipelined over three streams:
//   copy-in stream   Q, K, V of chunk c       (host -> device staging buffer c % 2)
//   caller's stream  the prefill of chunk c   (delta_attn_prefill, B = 1, Hq = G, Hkv = 1)
//   copy-out stream  O of chunk c             (staging buffer c % 2 -> host)
// with events between them: chunk c's copy-in waits until the prefill of chunk
// c - 2 has read the staging buffer, and its prefill waits until the copy-out
// of chunk c - 2 has emptied the output buffer.  Each chunk is contiguous in
// every tensor, so one cudaMemcpyAsync per tensor and chunk moves it.  Host
// buffers should be page-locked (cudaHostAlloc, or torch pin_memory), or the
// copies stop being asynchronous.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "delta_attn.h"

namespace {

constexpr int kMaxDevices = 64;
constexpr int kStages = 2;  // staging buffers

struct CopyStreams {
  cudaStream_t in = nullptr, out = nullptr;
};
CopyStreams g_streams[kMaxDevices];
std::once_flag g_streams_once[kMaxDevices];
cudaError_t g_streams_err[kMaxDevices];

// The two copy streams of the current device, created once per device (they
// live until the process exits, like the library's other per-device state).
int copy_streams(CopyStreams* out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DA_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return DA_ERR_UNSUPPORTED;
  std::call_once(g_streams_once[dev], [dev] {
    cudaError_t e = cudaStreamCreateWithFlags(&g_streams[dev].in, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&g_streams[dev].out, cudaStreamNonBlocking);
    g_streams_err[dev] = e;
  });
  if (g_streams_err[dev] != cudaSuccess) return DA_ERR_CUDA;
  *out = g_streams[dev];
  return DA_OK;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct HostPlan {
  int G = 1;
  size_t q_bytes = 0, kv_bytes = 0;  // one chunk's Q (and O), and its K (and V)
  size_t off_q = 0, off_k = 0, off_v = 0, off_o = 0, stage = 0;
  size_t chunk_ws = 0, off_ws = 0, total = 0;
};

int make_host_plan(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                   HostPlan* hp) {
  if (B < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0) return DA_ERR_INVALID_ARG;
  HostPlan p;
  p.G = Hq / Hkv;
  int rc = delta_attn_workspace_size(1, p.G, 1, N, d, n_sink, window, gamma, &p.chunk_ws);
  if (rc != DA_OK) return rc;
  p.q_bytes = (size_t)p.G * (size_t)N * (size_t)d * 2;
  p.kv_bytes = (size_t)N * (size_t)d * 2;
  p.off_q = 0;
  p.off_k = align256(p.q_bytes);
  p.off_v = p.off_k + align256(p.kv_bytes);
  p.off_o = p.off_v + align256(p.kv_bytes);
  p.stage = p.off_o + align256(p.q_bytes);
  p.off_ws = kStages * p.stage;
  p.total = p.off_ws + align256(p.chunk_ws);
  *hp = p;
  return DA_OK;
}

}  // namespace

extern "C" {

int delta_attn_host_workspace_size(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                                   size_t* bytes) {
  if (!bytes) return DA_ERR_INVALID_ARG;
  HostPlan hp;
  int rc = make_host_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, &hp);
  if (rc != DA_OK) return rc;
  *bytes = hp.total;
  return DA_OK;
}

int delta_attn_prefill_host(const void* Qh, const void* Kh, const void* Vh, void* Oh, int B, int Hq, int Hkv,
                            int64_t N, int d, int n_sink, int64_t window, int gamma, void* workspace,
                            size_t ws_bytes, void* stream) {
  nvtxRangePushA("delta_attn_prefill_host");
  struct Pop {
    ~Pop() { nvtxRangePop(); }
  } nvtx_pop;
  if (!Qh || !Kh || !Vh || !Oh) return DA_ERR_INVALID_ARG;
  HostPlan hp;
  int rc = make_host_plan(B, Hq, Hkv, N, d, n_sink, window, gamma, &hp);
  if (rc != DA_OK) return rc;
  if (workspace != nullptr && ws_bytes < hp.total) return DA_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return DA_ERR_MISALIGNED;
  CopyStreams cs;
  if ((rc = copy_streams(&cs)) != DA_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  const long long chunks = (long long)B * Hkv;
  std::vector<cudaEvent_t> ev;  // entry, then per chunk: copied in, computed, copied out
  auto cleanup = [&]() {
    for (cudaEvent_t e : ev) cudaEventDestroy(e);
  };
  auto new_event = [&](cudaEvent_t* e) -> bool {
    if (cudaEventCreateWithFlags(e, cudaEventDisableTiming) != cudaSuccess) return false;
    ev.push_back(*e);
    return true;
  };
  uint8_t* base = static_cast<uint8_t*>(workspace);
  bool owned = false;
  if (base == nullptr) {
    if (cudaMallocAsync(reinterpret_cast<void**>(&base), hp.total, s) != cudaSuccess) return DA_ERR_CUDA;
    owned = true;
  }
  // On a failure part of the pipeline may already be queued: the caller's
  // stream waits for both copy streams before the workspace is released.
  auto fail = [&](int code) {
    cudaEvent_t a, b;
    if (cudaEventCreateWithFlags(&a, cudaEventDisableTiming) == cudaSuccess) {
      if (cudaEventRecord(a, cs.in) == cudaSuccess) cudaStreamWaitEvent(s, a, 0);
      cudaEventDestroy(a);
    }
    if (cudaEventCreateWithFlags(&b, cudaEventDisableTiming) == cudaSuccess) {
      if (cudaEventRecord(b, cs.out) == cudaSuccess) cudaStreamWaitEvent(s, b, 0);
      cudaEventDestroy(b);
    }
    cleanup();
    if (owned) cudaFreeAsync(base, s);
    return code;
  };

  cudaEvent_t entry;
  if (!new_event(&entry) || cudaEventRecord(entry, s) != cudaSuccess ||
      cudaStreamWaitEvent(cs.in, entry, 0) != cudaSuccess || cudaStreamWaitEvent(cs.out, entry, 0) != cudaSuccess)
    return fail(DA_ERR_CUDA);
  std::vector<cudaEvent_t> in_done(chunks), comp_done(chunks), out_done(chunks);
  const uint8_t* q8 = static_cast<const uint8_t*>(Qh);
  const uint8_t* k8 = static_cast<const uint8_t*>(Kh);
  const uint8_t* v8 = static_cast<const uint8_t*>(Vh);
  uint8_t* o8 = static_cast<uint8_t*>(Oh);
  for (long long c = 0; c < chunks; ++c) {
    uint8_t* st = base + (size_t)(c % kStages) * hp.stage;
    if (!new_event(&in_done[c]) || !new_event(&comp_done[c]) || !new_event(&out_done[c])) return fail(DA_ERR_CUDA);
    // copy in (chunk c = (b, g): G consecutive query heads, one K and V head)
    if (c >= kStages && cudaStreamWaitEvent(cs.in, comp_done[c - kStages], 0) != cudaSuccess)
      return fail(DA_ERR_CUDA);
    if (cudaMemcpyAsync(st + hp.off_q, q8 + (size_t)c * hp.q_bytes, hp.q_bytes, cudaMemcpyHostToDevice, cs.in) !=
            cudaSuccess ||
        cudaMemcpyAsync(st + hp.off_k, k8 + (size_t)c * hp.kv_bytes, hp.kv_bytes, cudaMemcpyHostToDevice,
                        cs.in) != cudaSuccess ||
        cudaMemcpyAsync(st + hp.off_v, v8 + (size_t)c * hp.kv_bytes, hp.kv_bytes, cudaMemcpyHostToDevice,
                        cs.in) != cudaSuccess ||
        cudaEventRecord(in_done[c], cs.in) != cudaSuccess)
      return fail(DA_ERR_CUDA);
    // compute on the caller's stream
    if (cudaStreamWaitEvent(s, in_done[c], 0) != cudaSuccess ||
        (c >= kStages && cudaStreamWaitEvent(s, out_done[c - kStages], 0) != cudaSuccess))
      return fail(DA_ERR_CUDA);
    rc = delta_attn_prefill(st + hp.off_q, st + hp.off_k, st + hp.off_v, st + hp.off_o, 1, hp.G, 1, N, d, n_sink,
                            window, gamma, base + hp.off_ws, hp.chunk_ws, s);
    if (rc != DA_OK) return fail(rc);
    if (cudaEventRecord(comp_done[c], s) != cudaSuccess) return fail(DA_ERR_CUDA);
    // copy out
    if (cudaStreamWaitEvent(cs.out, comp_done[c], 0) != cudaSuccess ||
        cudaMemcpyAsync(o8 + (size_t)c * hp.q_bytes, st + hp.off_o, hp.q_bytes, cudaMemcpyDeviceToHost, cs.out) !=
            cudaSuccess ||
        cudaEventRecord(out_done[c], cs.out) != cudaSuccess)
      return fail(DA_ERR_CUDA);
  }
  // the caller's stream resumes once the last output has landed (the copy-out
  // stream keeps the chunks in order)
  if (cudaStreamWaitEvent(s, out_done[chunks - 1], 0) != cudaSuccess) return fail(DA_ERR_CUDA);
  if (owned && cudaFreeAsync(base, s) != cudaSuccess) {
    cleanup();
    return DA_ERR_CUDA;
  }
  cleanup();  // events are released once their pending work has completed
  return DA_OK;
}

}  // extern "C"
