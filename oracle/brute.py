"""Whole-matrix numpy statement of Delta Attention for small N (test
infrastructure only).

Independent of ``delta_oracle.c``: it builds the explicit N x N score matrix,
masks it with -inf, applies a matrix softmax and follows Alg. 1 literally
(``np.repeat`` of the Delta rows).  Nothing here is shared with the C oracle
or with the CUDA path.  Intended for N <= 64 or so.
"""
import numpy as np


def _masked_softmax(scores: np.ndarray, keep: np.ndarray) -> np.ndarray:
    z = np.where(keep, scores, -np.inf)
    z = z - z.max(axis=-1, keepdims=True)
    e = np.exp(z)
    return e / e.sum(axis=-1, keepdims=True)


def smooth(kind, params, delta, N, gamma):
    """Smoothed corrections for all N rows from the Delta rows [n_s, d]
    (appendix "Interpolation"), each in a form unlike the C oracle's loop:
    linear interpolation with ``np.interp`` through (k gamma, Delta_k), held
    constant after the last sample; the EMA as one lower-triangular weight
    matrix (row 0 keeps y_0, then weights beta (1-beta)^(i-j)); the
    alpha-beta-gamma filter of Alg. 2 as the linear state-space recursion
    x_k = M x_{k-1} + g Delta_k on the state (position, velocity,
    acceleration) over the Delta rows, its outputs then repeated gamma times."""
    n_s, d = delta.shape
    y = np.repeat(delta, gamma, axis=0)[:N]
    if kind == "none":
        return y
    if kind == "linear":
        xs = np.arange(n_s) * gamma
        rows = np.arange(N)
        return np.stack([np.interp(rows, xs, delta[:, e]) for e in range(d)], axis=1)
    if kind == "ema":
        beta = params[0]
        i = np.arange(N)[:, None]
        j = np.arange(N)[None, :]
        W = np.where(j <= i, beta * (1.0 - beta) ** np.maximum(i - j, 0), 0.0)
        W[:, 0] = (1.0 - beta) ** np.arange(N)
        return W @ y
    al, be, ga = params
    # predict p+v+a/2, v+a; residual r = y - predicted p; p += al r, v += be r, a += ga r
    M = np.array([[1.0 - al, 1.0 - al, 0.5 * (1.0 - al)],
                  [-be, 1.0 - be, 1.0 - 0.5 * be],
                  [-ga, -ga, 1.0 - 0.5 * ga]])
    g = np.array([al, be, ga])
    out = np.empty_like(delta)
    x = np.stack([delta[0], np.zeros(d), np.zeros(d)])     # [3, d]
    out[0] = delta[0]
    for k in range(1, n_s):
        x = M @ x + np.outer(g, delta[k])
        out[k] = x[0]
    return np.repeat(out, gamma, axis=0)[:N]


def lemma1_terms(Qf, Kf, Vf, n_sink, window, gamma, b, h, k):
    """Both sides of Lemma 1 for the sampled row i = k gamma of (b, h), from
    the explicit score row: a = causal softmax, a* = sparse softmax, the
    omitted set C(i) minus W(i).  H/(H+T) is the total causal-softmax weight of
    the omitted keys; returns (lhs[d], rhs[d], H/(H+T))."""
    N, d = Qf.shape[2], Qf.shape[3]
    G = Qf.shape[1] // Kf.shape[1]
    i = k * gamma
    Kh, Vh = Kf[b, h // G], Vf[b, h // G]
    col = np.arange(N)
    causal = col <= i
    sparse = causal & ((col > i - window) | (col < n_sink))
    omitted = causal & ~sparse
    scores = (Kh @ Qf[b, h, i]) / np.sqrt(d)
    a = _masked_softmax(scores[None, :], causal[None, :])[0]
    a_star = _masked_softmax(scores[None, :], sparse[None, :])[0]
    delta = a @ Vh - a_star @ Vh
    head = np.where(omitted, a, 0.0) @ Vh
    frac = a[omitted].sum()
    return np.abs(delta - head), frac * np.abs(Vh[sparse]).max(axis=0), frac


def delta_attn(Qf, Kf, Vf, n_sink, window, gamma, mode="delta", tail_dense=0, smooth_kind="none",
               smooth_params=()):
    """Qf [B,Hq,N,d], Kf/Vf [B,Hkv,N,d] float64.  Returns (A_hat, S, D_full).

    Eq. 1 attention matrix sigma(QK^T/sqrt(d)) with the causal mask; the
    StreamingLLM sparse matrix A* keeps the first n_sink columns and a band of
    `window` columns ending on the diagonal; Alg. 1: Delta at the rows
    delta = {i : i mod gamma = 0}, A^V = A*V + repeat(Delta, gamma).
    """
    B, Hq, N, d = Qf.shape
    G = Hq // Kf.shape[1]
    row = np.arange(N)[:, None]
    col = np.arange(N)[None, :]
    causal = col <= row
    band = col > row - window           # the `window` most recent keys, diagonal included
    sinks = col < n_sink
    sparse = causal & (band | sinks)
    A_hat = np.empty((B, Hq, N, d))
    S_all = np.empty((B, Hq, N, d))
    D_all = np.empty((B, Hq, N, d))
    for b in range(B):
        for h in range(Hq):
            Kh, Vh = Kf[b, h // G], Vf[b, h // G]
            scores = Qf[b, h] @ Kh.T / np.sqrt(d)
            AV = _masked_softmax(scores, causal) @ Vh        # quadratic attention, every row
            AsV = _masked_softmax(scores, sparse) @ Vh       # sparse attention, every row
            delta = AV[::gamma] - AsV[::gamma]               # rows i with i mod gamma == 0
            if mode == "delta":
                corr = smooth(smooth_kind, smooth_params, delta, N, gamma)
            else:                                            # Eq. 5: only the sampled rows move
                corr = np.zeros_like(AsV)
                corr[::gamma] = delta
            out = AsV + corr
            if tail_dense > 0:
                out[N - tail_dense:] = AV[N - tail_dense:]
            A_hat[b, h], S_all[b, h], D_all[b, h] = out, AsV, AV
    return A_hat, S_all, D_all
