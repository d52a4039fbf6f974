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


def delta_attn(Qf, Kf, Vf, n_sink, window, gamma, mode="delta", tail_dense=0):
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
                corr = np.repeat(delta, gamma, axis=0)[:N]
            else:                                            # Eq. 5: only the sampled rows move
                corr = np.zeros_like(AsV)
                corr[::gamma] = delta
            out = AsV + corr
            if tail_dense > 0:
                out[N - tail_dense:] = AV[N - tail_dense:]
            A_hat[b, h], S_all[b, h], D_all[b, h] = out, AsV, AV
    return A_hat, S_all, D_all
