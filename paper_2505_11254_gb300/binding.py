"""ctypes binding of libdeltaattn.so (C ABI in include/delta_attn.h).

Argument marshalling only: every step of the prefill runs in the library's
CUDA kernels.  Tensors are torch CUDA tensors (device memory); streams are
torch CUDA streams (default: the current stream).  There is no CPU fallback:
``load()`` raises if the library cannot be built or loaded.
"""
import ctypes
import os

import torch

from . import build as _build
from .flops import n_samples

DA_OK = 0
DA_ERR_INVALID_ARG = -1
DA_ERR_UNSUPPORTED = -2
DA_ERR_MISALIGNED = -3
DA_ERR_WORKSPACE = -4
DA_ERR_CUDA = -5
DA_ERR_TIMEOUT = -6

DA_MODE_DELTA = 0
DA_MODE_RECOMPUTE = 1
_MODES = {"delta": DA_MODE_DELTA, "recompute": DA_MODE_RECOMPUTE}
_SMOOTH = {"none": 0, "linear": 1, "ema": 2, "abg": 3}

_lib = None

_i = ctypes.c_int
_i64 = ctypes.c_int64
_p = ctypes.c_void_p
_sz = ctypes.c_size_t

_SIGNATURES = {
    "delta_attn_workspace_size": ([_i, _i, _i, _i64, _i, _i, _i64, _i, ctypes.POINTER(_sz)], _i),
    "delta_attn_prefill": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _i64, _i, _p, _sz, _p], _i),
    "delta_attn_workspace_size_ex": ([_i, _i, _i, _i64, _i, _i, _i64, _i, _i, _i64, ctypes.POINTER(_sz)], _i),
    "delta_attn_prefill_ex": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _i64, _i, _i, _i64, _p, _sz, _p], _i),
    "delta_attn_workspace_size_smoothed": ([_i, _i, _i, _i64, _i, _i, _i64, _i, _i, _i64, ctypes.POINTER(_sz)], _i),
    "delta_attn_prefill_smoothed": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _i64, _i, _i, ctypes.c_double,
                                     ctypes.c_double, ctypes.c_double, _i64, _p, _sz, _p], _i),
    "delta_attn_prefill_events": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _i64, _i, _p, _sz, _p,
                                   ctypes.POINTER(_p), _i], _i),
    "sparse_window_attn": ([_p, _p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _i64, _i, _p], _i),
    "strided_dense_workspace_size": ([_i, _i, _i, _i64, _i, _i, ctypes.POINTER(_sz)], _i),
    "strided_dense_attn": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _p, _sz, _p], _i),
    "strided_dense_attn_noalloc": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _p], _i),
    "delta_apply": ([_p, _p, _p, _p, _i, _i, _i64, _i, _i, _p], _i),
    "delta_attn_decode_workspace_size": ([_i, _i, _i, _i64, _i, ctypes.POINTER(_sz)], _i),
    "delta_attn_decode": ([_p, _p, _p, _p, _p, _i, _i, _i, _i64, _i64, _i, _p, _sz, _p], _i),
    "delta_attn_rope_table": ([_i64, _i, ctypes.c_double, _p, _p], _i),
    "delta_attn_rope_apply": ([_p, _i, _i, _i64, _i, _i64, _p, _i64, _p], _i),
    "delta_attn_prefill_rope": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _i64, _i, _p, _i64, _p, _sz, _p], _i),
    "delta_attn_workspace_size_rows": ([_i, _i, _i, _i64, _i, _i, _i64, _i, _i64, _i64, ctypes.POINTER(_sz)], _i),
    "delta_attn_prefill_rows": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _i64, _i, _i64, _i64, _p, _sz, _p], _i),
    "delta_attn_host_workspace_size": ([_i, _i, _i, _i64, _i, _i, _i64, _i, ctypes.POINTER(_sz)], _i),
    "delta_attn_prefill_host": ([_p, _p, _p, _p, _i, _i, _i, _i64, _i, _i, _i64, _i, _p, _sz, _p], _i),
    "delta_attn_check": ([_p], _i),
    "delta_attn_status_string": ([_i], ctypes.c_char_p),
    "delta_attn_plan_info": ([_i, _i, _i, _i64, _i, _i, _i64, _i, ctypes.POINTER(_i64)], _i),
    "delta_attn_debug_mask": ([_i64, _i, _i64, _i64, _i64, _p, _p], _i),
    "delta_attn_debug_rowmap": ([_i64, _i, _p, _p, _p], _i),
    "delta_attn_debug_work": ([_i, _i, _i, _i, _i64, _i, _i, _i64, _i, _i64, _p, _i, _p], _i),
    "delta_attn_debug_timeout": ([_i64, _p], _i),
}


class DeltaAttnError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__("%s failed: %s (%d)" % (where, status_string(status), status))


def library_path() -> str:
    return _build.LIB


def load(build_if_needed: bool = True):
    """Load (building first if stale) the CUDA library; raises on failure."""
    global _lib
    if _lib is None:
        path = _build.build() if build_if_needed else _build.LIB
        if not os.path.exists(path):
            raise RuntimeError("libdeltaattn.so is missing (%s); build it with __graft_entry__.build()" % path)
        lib = ctypes.CDLL(path)
        for name, (args, res) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _lib = lib
    return _lib


def status_string(status: int) -> str:
    return load().delta_attn_status_string(status).decode()


def _check(rc, where):
    if rc != DA_OK:
        raise DeltaAttnError(rc, where)


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _dptr(t):
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


def _qkv_shape(q, k, v):
    for name, t in (("q", q), ("k", k), ("v", v)):
        if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous() or t.dim() != 4:
            raise ValueError("%s must be a contiguous 4-D bf16 CUDA tensor" % name)
    B, Hq, N, d = q.shape
    if k.shape != v.shape or k.shape[0] != B or k.shape[2] != N or k.shape[3] != d:
        raise ValueError("q [B,Hq,N,d], k/v [B,Hkv,N,d]")
    return B, Hq, k.shape[1], N, d


def workspace_size(B, Hq, Hkv, N, d, n_sink, window, gamma, mode="delta", tail_dense=0, smooth="none") -> int:
    out = _sz(0)
    if smooth != "none":
        if mode != "delta":
            raise ValueError("smoothing applies to the Eq. 6 output")
        _check(load().delta_attn_workspace_size_smoothed(B, Hq, Hkv, N, d, n_sink, window, gamma, _SMOOTH[smooth],
                                                         tail_dense, ctypes.byref(out)),
               "delta_attn_workspace_size_smoothed")
    elif mode == "delta" and tail_dense == 0:
        _check(load().delta_attn_workspace_size(B, Hq, Hkv, N, d, n_sink, window, gamma, ctypes.byref(out)),
               "delta_attn_workspace_size")
    else:
        _check(load().delta_attn_workspace_size_ex(B, Hq, Hkv, N, d, n_sink, window, gamma, _MODES[mode],
                                                   tail_dense, ctypes.byref(out)), "delta_attn_workspace_size_ex")
    return out.value


def strided_dense_workspace_size(B, Hq, Hkv, N, d, gamma) -> int:
    out = _sz(0)
    _check(load().strided_dense_workspace_size(B, Hq, Hkv, N, d, gamma, ctypes.byref(out)),
           "strided_dense_workspace_size")
    return out.value


def workspace_size_rows(B, Hq, Hkv, N_kv, d, n_sink, window, gamma, row_begin, n_rows) -> int:
    out = _sz(0)
    _check(load().delta_attn_workspace_size_rows(B, Hq, Hkv, N_kv, d, n_sink, window, gamma, row_begin, n_rows,
                                                 ctypes.byref(out)), "delta_attn_workspace_size_rows")
    return out.value


def delta_attn_prefill_rows(q_rows, k, v, n_sink, window, gamma, row_begin, out=None, workspace=None, stream=None):
    """Rows row_begin .. row_begin + n_rows - 1 of the prefill of a sequence
    of N_kv tokens (one rank's share under context parallelism): ``q_rows``
    [B,Hq,n_rows,d] holds those rows of Q, ``k``/``v`` [B,Hkv,N_kv,d] the keys
    and values from row 0.  Returns bf16 [B,Hq,n_rows,d]."""
    for name, t in (("q_rows", q_rows), ("k", k), ("v", v)):
        if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous() or t.dim() != 4:
            raise ValueError("%s must be a contiguous 4-D bf16 CUDA tensor" % name)
    B, Hq, n_rows, d = q_rows.shape
    if k.shape != v.shape or k.shape[0] != B or k.shape[3] != d:
        raise ValueError("q_rows [B,Hq,n_rows,d], k/v [B,Hkv,N_kv,d]")
    Hkv, N_kv = k.shape[1], k.shape[2]
    if out is None:
        out = torch.empty_like(q_rows)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().delta_attn_prefill_rows(_dptr(q_rows), _dptr(k), _dptr(v), _dptr(out), B, Hq, Hkv, N_kv, d, n_sink,
                                          window, gamma, row_begin, n_rows, _dptr(workspace), ws_bytes,
                                          _stream(stream)), "delta_attn_prefill_rows")
    return out


def alloc_workspace(nbytes, device):
    return torch.empty(max(int(nbytes), 16), dtype=torch.uint8, device=device)


def delta_attn_prefill(q, k, v, n_sink, window, gamma, out=None, workspace=None, stream=None, mode="delta",
                       tail_dense=0, smooth="none", smooth_params=()):
    """Delta Attention prefill (Alg. 1 / Eq. 6) -> bf16 [B,Hq,N,d].

    ``mode="recompute"`` gives the Eq. 5 form and ``tail_dense=t`` makes the
    last t rows dense (both through delta_attn_prefill_ex); ``smooth`` =
    "linear", "ema" (params (beta,)) or "abg" (params (alpha, beta, gamma))
    smooths the corrections (delta_attn_prefill_smoothed)."""
    B, Hq, Hkv, N, d = _qkv_shape(q, k, v)
    if out is None:
        out = torch.empty_like(q)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    if smooth != "none":
        if mode != "delta":
            raise ValueError("smoothing applies to the Eq. 6 output")
        c1, c2, c3 = (tuple(float(x) for x in smooth_params) + (0.0, 0.0, 0.0))[:3]
        _check(load().delta_attn_prefill_smoothed(_dptr(q), _dptr(k), _dptr(v), _dptr(out), B, Hq, Hkv, N, d, n_sink,
                                                  window, gamma, _SMOOTH[smooth], c1, c2, c3, tail_dense,
                                                  _dptr(workspace), ws_bytes, _stream(stream)),
               "delta_attn_prefill_smoothed")
    elif mode == "delta" and tail_dense == 0:
        _check(load().delta_attn_prefill(_dptr(q), _dptr(k), _dptr(v), _dptr(out), B, Hq, Hkv, N, d, n_sink,
                                         window, gamma, _dptr(workspace), ws_bytes, _stream(stream)),
               "delta_attn_prefill")
    else:
        _check(load().delta_attn_prefill_ex(_dptr(q), _dptr(k), _dptr(v), _dptr(out), B, Hq, Hkv, N, d, n_sink,
                                            window, gamma, _MODES[mode], tail_dense, _dptr(workspace), ws_bytes,
                                            _stream(stream)), "delta_attn_prefill_ex")
    return out


def delta_attn_prefill_events(q, k, v, n_sink, window, gamma, events, out=None, workspace=None, stream=None):
    """The prefill with timing marks: ``events`` (torch.cuda.Event, already
    recorded once so they exist) are recorded before the first and after each
    kernel of the prefill on the launching stream."""
    B, Hq, Hkv, N, d = _qkv_shape(q, k, v)
    if out is None:
        out = torch.empty_like(q)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    arr = (_p * len(events))(*[ctypes.c_void_p(e.cuda_event) for e in events])
    _check(load().delta_attn_prefill_events(_dptr(q), _dptr(k), _dptr(v), _dptr(out), B, Hq, Hkv, N, d, n_sink,
                                            window, gamma, _dptr(workspace), ws_bytes, _stream(stream), arr,
                                            len(events)), "delta_attn_prefill_events")
    return out


def decode_workspace_size(B, Hq, Hkv, max_keys, d) -> int:
    out = _sz(0)
    _check(load().delta_attn_decode_workspace_size(B, Hq, Hkv, max_keys, d, ctypes.byref(out)),
           "delta_attn_decode_workspace_size")
    return out.value


def decode(q, k_cache, v_cache, lens=None, max_keys=None, out=None, workspace=None, stream=None):
    """Eq. 2 decoding: ``q`` [B,Hq,d] bf16 (one new token per sequence),
    ``k_cache``/``v_cache`` [B,Hkv,L,d] bf16 holding the new token's key and
    value at index lens[b]-1; ``lens`` int64 CUDA tensor [B] or None (all
    ``max_keys``, default L).  Returns bf16 [B,Hq,d]."""
    if q.dim() != 3 or k_cache.dim() != 4 or v_cache.shape != k_cache.shape:
        raise ValueError("q [B,Hq,d], caches [B,Hkv,L,d]")
    for t in (q, k_cache, v_cache):
        if not t.is_cuda or t.dtype != torch.bfloat16 or not t.is_contiguous():
            raise ValueError("q and the caches must be contiguous bf16 CUDA tensors")
    B, Hq, d = q.shape
    Hkv, L = k_cache.shape[1], k_cache.shape[2]
    if max_keys is None:
        max_keys = L
    if lens is not None and (lens.dtype != torch.int64 or not lens.is_cuda or lens.numel() != B):
        raise ValueError("lens: int64 CUDA tensor [B]")
    if out is None:
        out = torch.empty_like(q)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().delta_attn_decode(_dptr(q), _dptr(k_cache), _dptr(v_cache), _dptr(lens), _dptr(out), B, Hq, Hkv,
                                    L, max_keys, d, _dptr(workspace), ws_bytes, _stream(stream)), "delta_attn_decode")
    return out


def rope_table(n_pos, d, base, device="cuda", stream=None):
    """RoPE (cos, sin) table fp32 [n_pos, d/2, 2] for positions 0..n_pos-1."""
    t = torch.empty((n_pos, d // 2, 2), dtype=torch.float32, device=device)
    _check(load().delta_attn_rope_table(n_pos, d, float(base), _dptr(t), _stream(stream)), "delta_attn_rope_table")
    return t


def rope_apply(x, table, pos0=0, stream=None):
    """Rotates x [B,H,N,d] bf16 in place (row n at position pos0 + n)."""
    if x.dim() != 4 or x.dtype != torch.bfloat16 or not x.is_cuda or not x.is_contiguous():
        raise ValueError("x: contiguous bf16 CUDA tensor [B,H,N,d]")
    B, H, N, d = x.shape
    _check(load().delta_attn_rope_apply(_dptr(x), B, H, N, d, pos0, _dptr(table), table.shape[0], _stream(stream)),
           "delta_attn_rope_apply")
    return x


def delta_attn_prefill_rope(q, k, v, n_sink, window, gamma, table, out=None, workspace=None, stream=None):
    """The prefill for unrotated q and k with RoPE fused (k rotated in place)."""
    B, Hq, Hkv, N, d = _qkv_shape(q, k, v)
    if out is None:
        out = torch.empty_like(q)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().delta_attn_prefill_rope(_dptr(q), _dptr(k), _dptr(v), _dptr(out), B, Hq, Hkv, N, d, n_sink,
                                          window, gamma, _dptr(table), table.shape[0], _dptr(workspace), ws_bytes,
                                          _stream(stream)), "delta_attn_prefill_rope")
    return out


def host_workspace_size(B, Hq, Hkv, N, d, n_sink, window, gamma) -> int:
    out = _sz(0)
    _check(load().delta_attn_host_workspace_size(B, Hq, Hkv, N, d, n_sink, window, gamma, ctypes.byref(out)),
           "delta_attn_host_workspace_size")
    return out.value


def delta_attn_prefill_host(qh, kh, vh, n_sink, window, gamma, out=None, workspace=None, stream=None):
    """The prefill on host tensors (bf16, contiguous, page-locked): copies in,
    kernels and copies out pipelined per (batch, KV head) chunk.  Returns the
    host output tensor; it is complete once the stream reaches this point."""
    for name, t in (("q", qh), ("k", kh), ("v", vh)):
        if t.dtype != torch.bfloat16 or t.is_cuda or not t.is_contiguous() or t.dim() != 4:
            raise ValueError("%s: contiguous bf16 host tensor [B,H,N,d]" % name)
    B, Hq, N, d = qh.shape
    Hkv = kh.shape[1]
    if out is None:
        out = torch.empty(qh.shape, dtype=torch.bfloat16, pin_memory=True)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().delta_attn_prefill_host(_dptr(qh), _dptr(kh), _dptr(vh), _dptr(out), B, Hq, Hkv, N, d, n_sink,
                                          window, gamma, _dptr(workspace), ws_bytes, _stream(stream)),
           "delta_attn_prefill_host")
    return out


def sparse_window_attn(q, k, v, n_sink, window, gamma, out=None, s_sampled=None, stream=None):
    """StreamingLLM sink + window attention of every row -> bf16; optionally the
    fp32 sparse rows at the sampled rows into ``s_sampled`` [B,Hq,n_s,d]."""
    B, Hq, Hkv, N, d = _qkv_shape(q, k, v)
    if out is None:
        out = torch.empty_like(q)
    _check(load().sparse_window_attn(_dptr(q), _dptr(k), _dptr(v), _dptr(out), _dptr(s_sampled), B, Hq, Hkv, N, d,
                                     n_sink, window, gamma, _stream(stream)), "sparse_window_attn")
    return out


def strided_dense_attn(q, k, v, gamma, out=None, workspace=None, stream=None):
    """Dense causal attention of the rows k*gamma -> fp32 [B,Hq,n_s,d]."""
    B, Hq, Hkv, N, d = _qkv_shape(q, k, v)
    if out is None:
        out = torch.empty((B, Hq, n_samples(N, gamma), d), dtype=torch.float32, device=q.device)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().strided_dense_attn(_dptr(q), _dptr(k), _dptr(v), _dptr(out), B, Hq, Hkv, N, d, gamma,
                                     _dptr(workspace), ws_bytes, _stream(stream)), "strided_dense_attn")
    return out


def strided_dense_attn_noalloc(q, k, v, gamma, out=None, stream=None):
    """strided_dense_attn without a workspace: the library's fixed device
    scratch is used (for callers that cannot allocate)."""
    B, Hq, Hkv, N, d = _qkv_shape(q, k, v)
    if out is None:
        out = torch.empty((B, Hq, n_samples(N, gamma), d), dtype=torch.float32, device=q.device)
    _check(load().strided_dense_attn_noalloc(_dptr(q), _dptr(k), _dptr(v), _dptr(out), B, Hq, Hkv, N, d, gamma,
                                             _stream(stream)), "strided_dense_attn_noalloc")
    return out


def delta_apply(o_sparse, s_sampled, d_sampled, gamma, out=None, stream=None):
    """Eq. 6 as a separate pass; ``out`` may be ``o_sparse`` (in place)."""
    B, Hq, N, d = o_sparse.shape
    if out is None:
        out = torch.empty_like(o_sparse)
    _check(load().delta_apply(_dptr(o_sparse), _dptr(s_sampled), _dptr(d_sampled), _dptr(out), B, Hq, N, d, gamma,
                              _stream(stream)), "delta_apply")
    return out


def check(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device status word."""
    return load().delta_attn_check(_stream(stream))


def plan_info(B, Hq, Hkv, N, d, n_sink, window, gamma) -> dict:
    info = (_i64 * 10)()
    _check(load().delta_attn_plan_info(B, Hq, Hkv, N, d, n_sink, window, gamma, info), "delta_attn_plan_info")
    keys = ("ctas_sparse", "ctas_dense", "ctas_strided_sparse", "chunk", "split_units", "heads_per_tile",
            "samples_per_head", "fused_in_tile", "kernels", "sms")
    return dict(zip(keys, list(info)))


def debug_mask(N, n_sink, window, i0, i1, device="cuda"):
    out = torch.empty((i1 - i0) * N, dtype=torch.uint8, device=device)
    _check(load().delta_attn_debug_mask(N, n_sink, window, i0, i1, _dptr(out), _stream(None)),
           "delta_attn_debug_mask")
    return out.view(i1 - i0, N)


def debug_rowmap(N, gamma, device="cuda"):
    rows = torch.empty(N, dtype=torch.int64, device=device)
    sampled = torch.empty(N, dtype=torch.uint8, device=device)
    _check(load().delta_attn_debug_rowmap(N, gamma, _dptr(rows), _dptr(sampled), _stream(None)),
           "delta_attn_debug_rowmap")
    return rows, sampled


def debug_work(mode, B, Hq, Hkv, N, d, n_sink, window, gamma, index, max_tiles=4096, device="cuda"):
    out = torch.zeros(16 + 4 * 128 + 2 * max_tiles, dtype=torch.int64, device=device)
    _check(load().delta_attn_debug_work(mode, B, Hq, Hkv, N, d, n_sink, window, gamma, index, _dptr(out),
                                        max_tiles, _stream(None)), "delta_attn_debug_work")
    o = out.cpu().tolist()
    hdr = o[:16]
    T = hdr[8]
    return {
        "b": hdr[0], "h0": hdr[1], "g": hdr[2], "r0": hdr[3], "r_last": hdr[4], "n_sink_tiles": hdr[5],
        "kt_lo": hdr[6], "kt_hi": hdr[7], "T": T, "n_chunks": hdr[9], "chunk_idx": hdr[10], "ticket": hdr[11],
        "slot": hdr[12], "group": hdr[13], "mtile": hdr[14], "order": hdr[15],
        "lanes": [tuple(o[16 + 4 * t: 20 + 4 * t]) for t in range(128)],
        "tiles": [tuple(o[16 + 512 + 2 * j: 18 + 512 + 2 * j]) for j in range(min(T, max_tiles))],
    }


def debug_timeout(limit_ns, stream=None):
    _check(load().delta_attn_debug_timeout(limit_ns, _stream(stream)), "delta_attn_debug_timeout")
