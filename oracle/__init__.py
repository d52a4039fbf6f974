"""fp64 CPU oracle for the Delta Attention prefill — TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It shares no code with the CUDA path.

Two independent statements of the method live here:

* ``delta_oracle.c`` (wrapped below): direct per-row evaluation of Eq. 1
  (causal softmax attention), the StreamingLLM sink + window set, Eq. 4
  (sampled rows k*gamma), Alg. 1 / Eq. 6 (Delta correction), Eq. 5
  ("recompute"), the appendix dense tail block and the appendix Delta
  smoothing (linear interpolation, EMA, Alg. 2's alpha-beta-gamma filter)
  Eq. 2 decoding over the cache and RoPE on Q and K, all in double precision.
* ``brute.py``: whole-matrix numpy evaluation (explicit N x N score matrix,
  -inf masks, matrix softmax, ``np.repeat`` of Delta) for small N.

Inputs are bf16 bit patterns (numpy ``uint16``), shape ``[B, H, N, d]``.
Every function takes ``lib=`` to run another build of the C oracle (the
tests use this to show that the pins reject deliberately broken variants).
"""
import ctypes
import os

import numpy as np

from . import build as _build

_libs = {}


def _load(path=None):
    path = path or _build.build()
    if path not in _libs:
        lib = ctypes.CDLL(path)
        u16p = ctypes.POINTER(ctypes.c_uint16)
        dp = ctypes.POINTER(ctypes.c_double)
        i64 = ctypes.c_int64
        ci = ctypes.c_int
        lib.oracle_delta_attn_box.argtypes = [u16p, u16p, u16p, ci, ci, ci, i64, ci, ci, i64, ci,
                                              ci, ci, ci, ci, i64, i64, ci, i64,
                                              dp, dp, dp, dp, ci]
        lib.oracle_delta_attn_box.restype = ci
        lib.oracle_rows.argtypes = [u16p, u16p, u16p, ci, ci, ci, i64, ci, ci, i64, ci,
                                    ctypes.POINTER(ctypes.c_int64), i64, dp, dp, dp, dp, dp, ci]
        lib.oracle_rows.restype = ci
        lib.oracle_lemma1.argtypes = [u16p, u16p, u16p, ci, ci, ci, i64, ci, ci, i64, ci,
                                      ci, ci, i64, dp, dp, dp]
        lib.oracle_lemma1.restype = ci
        lib.oracle_smooth_seq.argtypes = [ci, ctypes.c_double, ctypes.c_double, ctypes.c_double, dp, i64, ci, i64,
                                          ci, i64, i64, dp]
        lib.oracle_smooth_seq.restype = ci
        lib.oracle_delta_attn_smoothed.argtypes = [u16p, u16p, u16p, ci, ci, ci, i64, ci, ci, i64, ci,
                                                   ci, ci, ci, ci, i64, i64, ci, ctypes.c_double, ctypes.c_double,
                                                   ctypes.c_double, i64, dp, dp, ci]
        lib.oracle_delta_attn_smoothed.restype = ci
        lib.oracle_decode.argtypes = [u16p, u16p, u16p, ci, ci, ci, i64, ci, ctypes.POINTER(ctypes.c_int64), dp, dp,
                                      ci]
        lib.oracle_decode.restype = ci
        lib.oracle_rope_f64.argtypes = [u16p, i64, i64, ci, i64, ctypes.c_double, dp]
        lib.oracle_rope_f64.restype = ci
        lib.oracle_rope_bf16.argtypes = [u16p, i64, i64, ci, i64, ctypes.c_double, u16p]
        lib.oracle_rope_bf16.restype = ci
        _libs[path] = lib
    return _libs[path]


def library_path() -> str:
    return _build.LIB


def _u16(a):
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError("oracle inputs are bf16 bit patterns (numpy uint16)")
    return a


def _ptr(a, t):
    return a.ctypes.data_as(ctypes.POINTER(t))


def _shape(Q, K, V):
    if Q.ndim != 4 or K.ndim != 4 or V.shape != K.shape:
        raise ValueError("Q [B,Hq,N,d], K,V [B,Hkv,N,d]")
    B, Hq, N, d = Q.shape
    if K.shape[0] != B or K.shape[2] != N or K.shape[3] != d:
        raise ValueError("shape mismatch")
    return B, Hq, K.shape[1], N, d


def bf16_bits_to_f64(a) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    a = np.asarray(a, dtype=np.uint16)
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


SMOOTH_KINDS = {"none": 0, "linear": 1, "ema": 2, "abg": 3}


def smooth_seq(kind, params, delta, n_s, gamma, rows, lib=None):
    """Smoothed Delta corrections of rows [r0, r1) of one (batch, head)
    (appendix "Interpolation"): ``delta`` [n_k, d] float64 holds Delta_0..;
    ``params`` = (c1, c2, c3): EMA beta, or the filter's alpha, beta, gamma."""
    delta = np.ascontiguousarray(delta, dtype=np.float64)
    n_k, d = delta.shape
    r0, r1 = rows
    out = np.empty((r1 - r0, d), np.float64)
    c1, c2, c3 = (tuple(params) + (0.0, 0.0, 0.0))[:3]
    rc = _load(lib).oracle_smooth_seq(SMOOTH_KINDS[kind], c1, c2, c3, _ptr(delta, ctypes.c_double), n_k, d, n_s,
                                      gamma, r0, r1, _ptr(out, ctypes.c_double))
    if rc != 0:
        raise ValueError("oracle_smooth_seq failed (invalid arguments)")
    return out


def delta_attn(Q, K, V, n_sink, window, gamma, *, batches=None, heads=None, rows=None,
               mode="delta", tail_dense=0, smooth="none", smooth_params=(), nthreads=0, lib=None):
    """Delta Attention (Alg. 1 / Eq. 6) over a box of batches, q-heads and rows.

    Returns a dict with float64 arrays ``A`` (corrected output A^V),
    ``S`` (sparse output A*V), ``D`` (dense output ~AV of the samples covering
    the rows, first sample floor(r0/gamma)) and ``max_dev`` (max |sum p - 1|
    over every softmax vector evaluated).
    ``mode``: "delta" (Eq. 6) or "recompute" (Eq. 5).
    ``smooth``: "none", "linear", "ema" or "abg" with ``smooth_params``
    (appendix "Interpolation"; Eq. 6 mode only).  With smoothing only ``A``
    and ``max_dev`` are returned.
    """
    Q, K, V = _u16(Q), _u16(K), _u16(V)
    B, Hq, Hkv, N, d = _shape(Q, K, V)
    b0, b1 = batches if batches is not None else (0, B)
    h0, h1 = heads if heads is not None else (0, Hq)
    r0, r1 = rows if rows is not None else (0, N)
    if smooth != "none":
        if mode != "delta":
            raise ValueError("smoothing applies to the Eq. 6 output")
        A = np.empty((b1 - b0, h1 - h0, r1 - r0, d), np.float64)
        dev = ctypes.c_double(0.0)
        c1, c2, c3 = (tuple(smooth_params) + (0.0, 0.0, 0.0))[:3]
        rc = _load(lib).oracle_delta_attn_smoothed(
            _ptr(Q, ctypes.c_uint16), _ptr(K, ctypes.c_uint16), _ptr(V, ctypes.c_uint16),
            B, Hq, Hkv, N, d, n_sink, window, gamma, b0, b1, h0, h1, r0, r1,
            SMOOTH_KINDS[smooth], c1, c2, c3, tail_dense, _ptr(A, ctypes.c_double), ctypes.byref(dev), nthreads)
        if rc != 0:
            raise ValueError("oracle_delta_attn_smoothed failed (invalid arguments)")
        return {"A": A, "max_dev": dev.value}
    k0, k1 = r0 // gamma, (r1 - 1) // gamma + 1
    nb, nh, nr, nk = b1 - b0, h1 - h0, r1 - r0, k1 - k0
    S = np.empty((nb, nh, nr, d), np.float64)
    D = np.empty((nb, nh, nk, d), np.float64)
    A = np.empty((nb, nh, nr, d), np.float64)
    dev = ctypes.c_double(0.0)
    dp = ctypes.c_double
    rc = _load(lib).oracle_delta_attn_box(
        _ptr(Q, ctypes.c_uint16), _ptr(K, ctypes.c_uint16), _ptr(V, ctypes.c_uint16),
        B, Hq, Hkv, N, d, n_sink, window, gamma,
        b0, b1, h0, h1, r0, r1, {"delta": 0, "recompute": 1}[mode], tail_dense,
        _ptr(S, dp), _ptr(D, dp), _ptr(A, dp), ctypes.byref(dev), nthreads)
    if rc != 0:
        raise ValueError("oracle_delta_attn_box failed (invalid arguments)")
    return {"A": A, "S": S, "D": D, "max_dev": dev.value}


def decode(q, K, V, n_keys, nthreads=0, lib=None):
    """Eq. 2 decoding: ``q`` [B,Hq,d] bf16 bits (one new token per sequence),
    ``K``/``V`` caches [B,Hkv,L,d] bf16 bits holding the new token's key and
    value at index n_keys[b]-1; ``n_keys`` [B] int.  Returns (out [B,Hq,d]
    float64, max |sum p - 1|)."""
    q, K, V = _u16(q), _u16(K), _u16(V)
    if q.ndim != 3 or K.ndim != 4 or V.shape != K.shape or q.shape[0] != K.shape[0] or q.shape[2] != K.shape[3]:
        raise ValueError("q [B,Hq,d], K,V [B,Hkv,L,d]")
    B, Hq, d = q.shape
    Hkv, L = K.shape[1], K.shape[2]
    nk = np.ascontiguousarray(np.asarray(n_keys, dtype=np.int64).reshape(B))
    out = np.empty((B, Hq, d), np.float64)
    dev = ctypes.c_double(0.0)
    rc = _load(lib).oracle_decode(_ptr(q, ctypes.c_uint16), _ptr(K, ctypes.c_uint16), _ptr(V, ctypes.c_uint16),
                                  B, Hq, Hkv, L, d, _ptr(nk, ctypes.c_int64), _ptr(out, ctypes.c_double),
                                  ctypes.byref(dev), nthreads)
    if rc != 0:
        raise ValueError("oracle_decode failed (invalid arguments)")
    return out, dev.value


def rope(X, base, pos0=0, rounded=True, lib=None):
    """RoPE (rotate-half, angle pos * base^(-2c/d)) of X [..., N, d] bf16 bits,
    row n at position pos0 + n.  rounded=True returns bf16 bits (RNE),
    otherwise the float64 rotation."""
    X = _u16(X)
    N, d = X.shape[-2], X.shape[-1]
    rows_total = X.size // d
    if rounded:
        out = np.empty(X.shape, np.uint16)
        rc = _load(lib).oracle_rope_bf16(_ptr(X, ctypes.c_uint16), rows_total, N, d, pos0, base,
                                         _ptr(out, ctypes.c_uint16))
    else:
        out = np.empty(X.shape, np.float64)
        rc = _load(lib).oracle_rope_f64(_ptr(X, ctypes.c_uint16), rows_total, N, d, pos0, base,
                                        _ptr(out, ctypes.c_double))
    if rc != 0:
        raise ValueError("oracle rope failed (invalid arguments)")
    return out


def rows(Q, K, V, n_sink, window, gamma, bhi, nthreads=0, lib=None):
    """Per-row evaluation for (b, h, i) triples: returns dict of [n, d] arrays
    ``S`` (sparse row i), ``D_sample``/``S_sample`` (dense/sparse row of the
    sample floor(i/gamma)*gamma) and ``A`` (Eq. 6 output row i)."""
    Q, K, V = _u16(Q), _u16(K), _u16(V)
    B, Hq, Hkv, N, d = _shape(Q, K, V)
    bhi = np.ascontiguousarray(np.asarray(bhi, dtype=np.int64).reshape(-1, 3))
    n = bhi.shape[0]
    out = {k: np.empty((n, d), np.float64) for k in ("S", "D_sample", "S_sample", "A")}
    dev = ctypes.c_double(0.0)
    dp = ctypes.c_double
    rc = _load(lib).oracle_rows(
        _ptr(Q, ctypes.c_uint16), _ptr(K, ctypes.c_uint16), _ptr(V, ctypes.c_uint16),
        B, Hq, Hkv, N, d, n_sink, window, gamma,
        _ptr(bhi, ctypes.c_int64), n,
        _ptr(out["S"], dp), _ptr(out["D_sample"], dp), _ptr(out["S_sample"], dp),
        _ptr(out["A"], dp), ctypes.byref(dev), nthreads)
    if rc != 0:
        raise ValueError("oracle_rows failed (invalid arguments)")
    out["max_dev"] = dev.value
    return out


def lemma1(Q, K, V, n_sink, window, gamma, b, h, k, lib=None):
    """Lemma 1 terms for sample k of (b, h): (lhs[d], rhs[d], H/(H+T))."""
    Q, K, V = _u16(Q), _u16(K), _u16(V)
    B, Hq, Hkv, N, d = _shape(Q, K, V)
    lhs = np.empty(d, np.float64)
    rhs = np.empty(d, np.float64)
    frac = ctypes.c_double(0.0)
    dp = ctypes.c_double
    rc = _load(lib).oracle_lemma1(
        _ptr(Q, ctypes.c_uint16), _ptr(K, ctypes.c_uint16), _ptr(V, ctypes.c_uint16),
        B, Hq, Hkv, N, d, n_sink, window, gamma, b, h, k,
        _ptr(lhs, dp), _ptr(rhs, dp), ctypes.byref(frac))
    if rc != 0:
        raise ValueError("oracle_lemma1 failed (invalid arguments)")
    return lhs, rhs, frac.value
