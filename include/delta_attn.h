/*
 * delta_attn.h — C ABI of libdeltaattn.so: the Delta Attention prefill
 * (Willette, Lee, Hwang, "Delta Attention: Fast and Accurate Sparse Attention
 * Inference by Delta Correction", arXiv 2505.11254) on NVIDIA GB300 (sm_103a).
 *
 * What is computed (0-based rows; tau = 1/sqrt(d)):
 *   Eq. 1   dense causal attention  D_i = sum_{j<=i} softmax_j(tau q_i.k_j) v_j
 *   f*      StreamingLLM sparse attention over
 *           W(i) = { j <= i : j < n_sink  or  j > i - window },
 *           S_i = sum_{j in W(i)} softmax_W(tau q_i.k_j) v_j   (normalised over W(i) only)
 *   Eq. 4   sampled query rows k*gamma, k = 0 .. n_s-1, n_s = ceil(N / gamma)
 *   Alg. 1  Delta_k = D_{k gamma} - S_{k gamma}
 *   Eq. 6   O_i = S_i + Delta_{floor(i/gamma)}
 *           (on a sampled row this equals D_{k gamma}; the library writes D there)
 * GQA: query head h reads KV head floor(h / (Hq/Hkv)).
 *
 * Layouts (all row-major, contiguous, device memory, 16-byte aligned):
 *   Q, O, O_sparse     [B, Hq,  N, d]   bf16
 *   K, V               [B, Hkv, N, d]   bf16
 *   D_sampled, S_sampled [B, Hq, n_s, d] fp32 (row k holds sample row k*gamma)
 * Supported: d in {64, 128}; Hq % Hkv == 0; N, gamma, window >= 1; n_sink >= 0;
 * N <= 2^31 - 256; a device of compute capability 10.3 (GB300).
 *
 * Ownership and execution: the caller owns every buffer.  All calls are
 * asynchronous on `stream` (a cudaStream_t; NULL is the legacy default stream)
 * and never synchronise the device, except delta_attn_check().  Arguments are
 * validated on the host before anything is launched; invalid arguments return
 * an error and launch nothing.  Launch failures return DA_ERR_CUDA.  A kernel
 * that gives up a bounded wait (it never should) records DA_ERR_TIMEOUT in a
 * per-device status word that delta_attn_check() reports; the word's device
 * address is looked up once per device, on the first launching call made with
 * that device current.  Results are deterministic: fixed merge order, no
 * floating-point atomics.
 *
 * Kernel choice: the sink + window pass of a whole sequence at d = 128 with
 * an even Hq / Hkv and window >= 512 runs as a two-CTA kernel (thread-block
 * clusters of two, one per pair of query heads of a KV group); other shapes
 * run the one-CTA kernel.  Both give the same bits.  The environment variable
 * DELTA_ATTN_PAIR, read at each call, overrides the choice: "0" always takes
 * the one-CTA kernel, "1" the two-CTA kernel wherever the shape allows it.
 */
#ifndef DELTA_ATTN_H
#define DELTA_ATTN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DA_OK = 0,
    DA_ERR_INVALID_ARG = -1,  /* bad sizes, NULL pointer, Hq % Hkv != 0 ... */
    DA_ERR_UNSUPPORTED = -2,  /* head dim or device not supported            */
    DA_ERR_MISALIGNED = -3,   /* a pointer is not 16-byte aligned            */
    DA_ERR_WORKSPACE = -4,    /* workspace smaller than required             */
    DA_ERR_CUDA = -5,         /* a CUDA runtime call or launch failed        */
    DA_ERR_TIMEOUT = -6       /* a kernel gave up a bounded wait             */
} da_status;

/* Workspace bytes delta_attn_prefill() needs for this shape on the current
 * device (fp32 dense sampled rows, Delta rows when gamma does not divide 128,
 * split-K partials and their tickets).  Writes *bytes; returns a da_status. */
int delta_attn_workspace_size(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                              size_t* bytes);

/* The full prefill (Alg. 1 with Eq. 6): writes O.  Runs the strided dense
 * kernel (D at the sampled rows), then the sink+window kernel whose epilogue
 * adds Delta and writes bf16 O once.  gamma = 1 makes every row a dense row
 * (plain causal attention).  `workspace` (device, >= the size above) may be
 * NULL, in which case the library allocates it stream-ordered
 * (cudaMallocAsync / cudaFreeAsync on `stream`). */
int delta_attn_prefill(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv, int64_t N,
                       int d, int n_sink, int64_t window, int gamma, void* workspace, size_t ws_bytes,
                       void* stream);

/* delta_attn_prefill() with timing marks: records the caller's CUDA events
 * (cudaEvent_t, created by the caller) on `stream` before the first kernel and
 * after each kernel of the prefill, so events[i+1] - events[i] is the duration
 * of kernel i.  n_events must equal the kernel count + 1 (plan_info()[8] + 1).
 * The kernels are the strided dense kernel, [the strided sparse kernel when
 * gamma does not divide 128,] and the sink+window kernel with the Delta
 * epilogue; with gamma = 1 only the dense kernel runs. */
int delta_attn_prefill_events(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv,
                              int64_t N, int d, int n_sink, int64_t window, int gamma, void* workspace,
                              size_t ws_bytes, void* stream, void* const* events, int n_events);

/* Output variants of delta_attn_prefill_ex(). */
typedef enum {
    DA_MODE_DELTA = 0,     /* Eq. 6: every row i gets Delta of sample floor(i/gamma)   */
    DA_MODE_RECOMPUTE = 1  /* Eq. 5: only the sampled rows k*gamma become dense rows;
                              every other row keeps its sink+window output            */
} da_mode;

/* Workspace bytes delta_attn_prefill_ex() needs for this shape, mode and dense
 * tail (the sizes of delta_attn_workspace_size() plus the tail's split-K
 * partials and tickets).  Writes *bytes; returns a da_status. */
int delta_attn_workspace_size_ex(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                                 int mode, int64_t tail_dense, size_t* bytes);

/* The prefill with the paper's two ablation forms.
 *   mode: DA_MODE_DELTA (Eq. 6; the same result as delta_attn_prefill()) or
 *         DA_MODE_RECOMPUTE (Eq. 5, the "recompute" form of Sec. 3: the
 *         sink+window output for every row, the dense row at each sampled row
 *         k*gamma, and no correction of the rows between samples).
 *   tail_dense: 0 <= tail_dense <= N.  The last tail_dense rows
 *         (N - tail_dense .. N - 1) are dense causal attention rows (appendix
 *         "Implementation Details": a final block of queries recomputed
 *         densely); the rows before it are unchanged by the tail.  The paper
 *         does not give the block's size, so the caller chooses it; 0 means
 *         no tail.
 * Kernels, in stream order: the sampled-row and sparse passes of the chosen
 * mode (Delta: strided dense, [strided sparse,] sink+window with the Delta
 * epilogue; recompute: sink+window, then the dense sampled rows written over
 * O), then, when tail_dense > 0, a dense pass over the tail rows written over
 * O.  The sparse pass stops at the 128-row tile holding row N - tail_dense - 1.
 * gamma = 1 ignores both options (every row is dense).  Layouts, workspace
 * and error behaviour as delta_attn_prefill(); an unknown mode or a
 * tail_dense outside [0, N] returns DA_ERR_INVALID_ARG. */
int delta_attn_prefill_ex(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv, int64_t N,
                          int d, int n_sink, int64_t window, int gamma, int mode, int64_t tail_dense,
                          void* workspace, size_t ws_bytes, void* stream);

/* Delta smoothing forms of delta_attn_prefill_smoothed() (appendix
 * "Interpolation"). */
typedef enum {
    DA_SMOOTH_NONE = 0,    /* Eq. 6 as is                                          */
    DA_SMOOTH_LINEAR = 1,  /* row i = k*gamma + r gets (1 - r/gamma) Delta_k +
                              (r/gamma) Delta_{k+1}; the last group keeps Delta_k    */
    DA_SMOOTH_EMA = 2,     /* c1 = beta in [0, 1]: over the rows, e_0 = Delta_0,
                              e_i = (1 - beta) e_{i-1} + beta Delta_{floor(i/gamma)}   */
    DA_SMOOTH_ABG = 3      /* c1, c2, c3 = the alpha, beta, gamma of Alg. 2's filter,
                              run over the Delta vectors; row i gets the filter's
                              output for its sample floor(i/gamma)                  */
} da_smooth;

/* Workspace bytes delta_attn_prefill_smoothed() needs: fp32 D and Delta rows,
 * two fp32 basis vectors per sample, min(gamma, N) x 2 coefficients, split-K
 * partials and tickets, and the dense tail's.  Returns a da_status. */
int delta_attn_workspace_size_smoothed(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window,
                                       int gamma, int smooth, int64_t tail_dense, size_t* bytes);

/* The Eq. 6 prefill with the Delta corrections smoothed before they are added
 * (appendix "Interpolation", Alg. 2).  Every row, sampled rows included, is
 * written as bf16(S_i + corrected Delta); with DA_SMOOTH_NONE this is
 * delta_attn_prefill_ex() in DA_MODE_DELTA.  Kernels, in stream order: the
 * strided dense kernel (fp32 D), the strided sparse kernel (fp32 Delta_k =
 * D_k - S_{k gamma}), the smoothing pass (one thread per head and column,
 * sequential over the samples: the EMA carry between groups and the filter
 * state), the sink+window kernel whose epilogue adds the smoothed correction,
 * and the dense tail pass when tail_dense > 0.  c1..c3 must be finite; an EMA
 * beta outside [0, 1] or an unknown form returns DA_ERR_INVALID_ARG.  The
 * filter's stability is the caller's choice of coefficients.  Layouts,
 * workspace, tail and errors as delta_attn_prefill_ex(). */
int delta_attn_prefill_smoothed(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv,
                                int64_t N, int d, int n_sink, int64_t window, int gamma, int smooth, double c1,
                                double c2, double c3, int64_t tail_dense, void* workspace, size_t ws_bytes,
                                void* stream);

/* f*(Q,K,V) of Alg. 1 alone: StreamingLLM sink + window attention of every
 * row, written as bf16 to O_sparse.  When S_sampled is not NULL the fp32
 * sparse rows at the sampled rows k*gamma are also written (the operand
 * delta_apply() subtracts). */
int sparse_window_attn(const void* Q, const void* K, const void* V, void* O_sparse, float* S_sampled, int B,
                       int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma, void* stream);

/* Workspace bytes strided_dense_attn() needs (split-K partials, tickets). */
int strided_dense_workspace_size(int B, int Hq, int Hkv, int64_t N, int d, int gamma, size_t* bytes);

/* f(~Q,K,V) of Alg. 1 alone: dense causal attention of the sampled rows
 * k*gamma (Eq. 4), fp32, into D_sampled [B,Hq,n_s,d].  The key range is split
 * across CTAs where that balances the GPU; partials are merged in a fixed
 * order.  `workspace` may be NULL (stream-ordered allocation). */
int strided_dense_attn(const void* Q, const void* K, const void* V, float* D_sampled, int B, int Hq, int Hkv,
                       int64_t N, int d, int gamma, void* workspace, size_t ws_bytes, void* stream);

/* strided_dense_attn() for callers that cannot allocate device memory (their
 * memory is owned by another allocator or budgeted up front, or their hot path
 * must not allocate).  The paper has no counterpart: this is an integration
 * variant.  Same arguments and results as strided_dense_attn() without the
 * workspace: the split-K scratch lives in a fixed 16 MiB device array inside
 * the library, held by every GPU that loads it until the process exits.  A
 * shape whose scratch (strided_dense_workspace_size()) exceeds 16 MiB returns
 * DA_ERR_WORKSPACE.  No call allocates: the first call on a device looks up
 * the array's device address and the library's device status word (so make
 * that first call before any stream capture); every call then zeroes the
 * scratch's tickets and counter on `stream` and launches the kernel.  All calls share the one array, so calls
 * whose work overlaps on the GPU (different streams, or several host threads)
 * race and must be serialised by the caller. */
int strided_dense_attn_noalloc(const void* Q, const void* K, const void* V, float* D_sampled, int B, int Hq,
                               int Hkv, int64_t N, int d, int gamma, void* stream);

/* Eq. 6 as a separate pass: O_i = bf16(S_i + D_k - S_{k gamma}) for rows that
 * are not sampled and O_{k gamma} = bf16(D_k), with S_i read from the bf16
 * O_sparse and S_{k gamma} from S_sampled (fp32) or, when S_sampled is NULL,
 * from O_sparse's sampled row.  O may alias O_sparse. */
int delta_apply(const void* O_sparse, const float* S_sampled, const float* D_sampled, void* O, int B, int Hq,
                int64_t N, int d, int gamma, void* stream);

/* Workspace bytes delta_attn_decode() needs: one fp32 partial (o, max, sum)
 * per query head and key range.  Returns a da_status. */
int delta_attn_decode_workspace_size(int B, int Hq, int Hkv, int64_t max_keys, int d, size_t* bytes);

/* Eq. 2: decoding after the prefill.  The query of one newly generated token
 * per sequence attends densely over that sequence's cache, whose last valid
 * entry is the new token's own key and value:
 *   O[b,h,:] = softmax_j(q[b,h,:] . K[b,g,j,:] / sqrt(d)) V[b,g,j,:],
 *   j = 0 .. lens[b] - 1, g = floor(h / (Hq/Hkv)).
 *   q, O: [B, Hq, d] bf16; K, V: [B, Hkv, L, d] bf16 caches of capacity L
 *   (rows past a sequence's length are never read); device pointers, 16-byte
 *   aligned.  lens: device int64 [B], each in [1, L] (values outside are
 *   clamped to [0, L]; a sequence with 0 keys gets a zero row), or NULL for
 *   max_keys keys everywhere; 1 <= max_keys <= L bounds every lens[b] and
 *   sizes the split.  Hq / Hkv <= 16, d in {64, 128}.
 * Bound by HBM bandwidth (each cached byte is read once per step): CUDA-core
 * kernel, split-K over key ranges with a second kernel merging them in a
 * fixed order.  workspace may be NULL (stream-ordered allocation on `stream`).
 * Returns a da_status; asynchronous on `stream`. */
int delta_attn_decode(const void* q, const void* K, const void* V, const int64_t* lens, void* O, int B, int Hq,
                      int Hkv, int64_t L, int64_t max_keys, int d, void* workspace, size_t ws_bytes, void* stream);

/* RoPE (Sec. 2: positional encodings on Q and K before the attention), in the
 * rotate-half form: for c < d/2 the pair (x_c, x_{c+d/2}) of a row at
 * position pos is rotated by the angle pos * base^(-2c/d).
 *
 * delta_attn_rope_table: writes the (cos, sin) table for positions
 * 0 .. n_pos-1, table [n_pos][d/2][2] fp32 (device, 16-byte aligned,
 * n_pos * d * 4 bytes), angles and sines taken in double.  Built once per
 * (n_pos, d, base) and shared by every layer and call. */
int delta_attn_rope_table(int64_t n_pos, int d, double base, float* table, void* stream);

/* Rotates X [B, H, N, d] bf16 (device, 16-byte aligned) in place, row n at
 * position pos0 + n (a new token's query or key at its position, or a whole
 * K before the prefill); fp32 arithmetic, one rounding to bf16 (RNE).  The
 * table (table_rows positions) must cover pos0 + N - 1. */
int delta_attn_rope_apply(void* X, int B, int H, int64_t N, int d, int64_t pos0, const float* table,
                          int64_t table_rows, void* stream);

/* delta_attn_prefill() for unrotated Q and K, with RoPE fused: K is rotated
 * in place first (on return it holds RoPE(K), the form the cache keeps for
 * decoding), and each Q tile is rotated by the attention kernels while it is
 * copied into tensor memory (Q itself is not modified), so no rotated copy of
 * Q is written or read.  Positions are the row indices 0 .. N-1; the table
 * must cover them (table_rows >= N).  Everything else as delta_attn_prefill(). */
int delta_attn_prefill_rope(const void* Q, void* K, const void* V, void* O, int B, int Hq, int Hkv, int64_t N, int d,
                            int n_sink, int64_t window, int gamma, const float* table, int64_t table_rows,
                            void* workspace, size_t ws_bytes, void* stream);

/* Rows row_begin .. row_begin + n_rows - 1 of delta_attn_prefill() over a
 * sequence of N_kv tokens: one rank's share of a sequence split by rows
 * (context parallelism).  Alg. 1 and Eq. 6 evaluate each row from its own
 * query and the keys up to it, so the rows of a range need the whole Q and O
 * of the range only, and K, V up to its last row (the sink keys, the window
 * before the first row and, for the sampled rows' dense attention, every
 * earlier key).
 *   Q, O: [B, Hq, n_rows, d] bf16, row i of the sequence at index i - row_begin;
 *   K, V: [B, Hkv, N_kv, d] bf16, rows from 0 (rows past row_begin + n_rows are
 *         not read); row_begin a multiple of 128 and of gamma (the range starts
 *         a row tile and a sample group), n_rows >= 1, row_begin + n_rows <= N_kv.
 * The result rows equal those of the whole-sequence call up to the order of
 * the dense rows' split-K merge.  workspace as delta_attn_prefill(), sized by
 * delta_attn_workspace_size_rows().  Returns a da_status; asynchronous on
 * `stream`. */
int delta_attn_workspace_size_rows(int B, int Hq, int Hkv, int64_t N_kv, int d, int n_sink, int64_t window,
                                   int gamma, int64_t row_begin, int64_t n_rows, size_t* bytes);
int delta_attn_prefill_rows(const void* Q, const void* K, const void* V, void* O, int B, int Hq, int Hkv,
                            int64_t N_kv, int d, int n_sink, int64_t window, int gamma, int64_t row_begin,
                            int64_t n_rows, void* workspace, size_t ws_bytes, void* stream);

/* Workspace bytes delta_attn_prefill_host() needs: two device staging buffers
 * of one (batch, KV head) chunk (its G query heads of Q and O, one K and V
 * head) and the workspace of a chunk's prefill.  Returns a da_status. */
int delta_attn_host_workspace_size(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                                   size_t* bytes);

/* delta_attn_prefill() on HOST buffers: Qh, Kh, Vh, Oh with the layouts of
 * delta_attn_prefill() in host memory (page-locked for asynchronous copies).
 * The B * Hkv (batch, KV head) chunks are independent, so their copies in,
 * prefills and copies out are pipelined over three streams (two internal copy
 * streams, created once per device, and `stream` for the kernels), with two
 * device staging buffers in the workspace (device, 256-byte aligned, or NULL
 * for stream-ordered allocation on `stream`).  Asynchronous: Oh is complete
 * when `stream` reaches the end of the call.  Each chunk's prefill is
 * delta_attn_prefill() with B = 1, Hq = G, Hkv = 1 (the split-K plan of the
 * dense rows follows the chunk's size, so the result may differ from one
 * whole-problem call in the last bits of fp32 rounding order). */
int delta_attn_prefill_host(const void* Qh, const void* Kh, const void* Vh, void* Oh, int B, int Hq, int Hkv,
                            int64_t N, int d, int n_sink, int64_t window, int gamma, void* workspace,
                            size_t ws_bytes, void* stream);

/* Synchronises `stream`, returns and clears the device status word
 * (DA_OK, DA_ERR_TIMEOUT), or DA_ERR_CUDA if the stream reports an error. */
int delta_attn_check(void* stream);

/* Static description of a status code. */
const char* delta_attn_status_string(int status);

/* ---- Introspection for tests (same code paths the kernels use). ---- */

/* Host: how the prefill is decomposed.  info[0..9] = CTAs of the sink+window
 * kernel, CTAs of the strided dense kernel, CTAs of the strided sparse kernel
 * (0 unless used), key tiles per split-K unit, split units, heads packed per
 * sampled-row tile, samples per head in it, 1 if Delta is fused inside the
 * row tile (gamma divides 128 and 128/gamma sampled rows fit the epilogue
 * buffer: gamma >= 8 at d = 128, gamma >= 4 at d = 64), kernels one prefill
 * launches, SM count.  CTA counts are work items; the kernels are persistent
 * with min(items, SMs) CTAs. */
int delta_attn_plan_info(int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window, int gamma,
                         int64_t* info);

/* Device: out[(i - i0) * N + j] = 1 if key j is in W(i), else 0, for
 * i in [i0, i1) — the predicate the sparse kernels apply. out: uint8 device. */
int delta_attn_debug_mask(int64_t N, int n_sink, int64_t window, int64_t i0, int64_t i1, uint8_t* out,
                          void* stream);

/* Device: sample_row[i] = floor(i/gamma)*gamma and is_sampled[i] = (i % gamma == 0)
 * for i in [0, N), as the epilogues compute them. */
int delta_attn_debug_rowmap(int64_t N, int gamma, int64_t* sample_row, uint8_t* is_sampled, void* stream);

/* Device: the work item `index` of kernel `mode` (0 sink+window rows,
 * 1 strided dense, 2 strided sparse) as the kernel decodes it.  out (int64,
 * device) holds 16 + 4*128 + 2*max_tiles entries: a header (b, first head,
 * kv head, first row or sample, last row or sample, sink tiles, first and last
 * band tile, tiles, chunks, chunk index, merge ticket, partial slot, (b, head
 * group) index, M-tile index, split-K order: 0 longest-first, 1 key-range
 * levels), then per TMEM lane (row, sample, head, valid), then per key tile
 * (tile index, needs mask). */
int delta_attn_debug_work(int mode, int B, int Hq, int Hkv, int64_t N, int d, int n_sink, int64_t window,
                          int gamma, int64_t index, int64_t* out, int max_tiles, void* stream);

/* Device: exercises the bounded-wait failure path without faulting the GPU.
 * Launches one warp that waits on an mbarrier nothing arrives on; after
 * limit_ns (0 < limit_ns <= 1e9) the wait gives up and records DA_ERR_TIMEOUT,
 * which the next delta_attn_check() returns (and clears). */
int delta_attn_debug_timeout(int64_t limit_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DELTA_ATTN_H */
