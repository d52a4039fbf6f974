"""Work accounting for the Delta Attention prefill (host logic, no GPU).

Useful work counts only the unmasked (query, key) pairs that the method's
definition evaluates:

* sparse part (StreamingLLM f*, every row i): |W(i)| keys, with
  W(i) = {j <= i : j < n_sink or j >= i - window + 1};
* dense part (Alg. 1's f on the strided queries of Eq. 4): row k*gamma sees
  k*gamma + 1 keys.

Each pair costs 2d FLOPs for q.k and 2d for p*v, i.e. 4d per pair per head.
The appendix "Approx Window Size Calculation" amortises the same count as
w + C/(2 gamma) keys per row (3072 at C = 2^17, w = 2048, gamma = 64).
"""
import numpy as np


def n_samples(N: int, gamma: int) -> int:
    """Number of sampled rows {0, gamma, 2 gamma, ...} below N (Eq. 4)."""
    return (N + gamma - 1) // gamma


def sparse_pairs_per_head(N: int, n_sink: int, window: int) -> int:
    """sum_i |W(i)| for i in [0, N)."""
    i = np.arange(N, dtype=np.int64)
    start = np.maximum(0, i - window + 1)          # first key of the band
    band = i - start + 1
    sinks_outside = np.minimum(n_sink, start)      # sinks not already in the band
    return int((band + sinks_outside).sum())


def dense_pairs_per_head(N: int, gamma: int) -> int:
    """sum_k (k gamma + 1) over the sampled rows."""
    ns = n_samples(N, gamma)
    return gamma * ns * (ns - 1) // 2 + ns


def causal_pairs_per_head(N: int) -> int:
    """Dense causal attention (gamma = 1): N (N + 1) / 2 pairs."""
    return N * (N + 1) // 2


def tail_pairs_per_head(N: int, tail: int) -> int:
    """Dense rows N - tail .. N - 1 of the tail block: sum of (i + 1)."""
    t = max(0, min(tail, N))
    return causal_pairs_per_head(N) - causal_pairs_per_head(N - t)


def useful_flops(B, Hq, N, d, n_sink, window, gamma) -> int:
    pairs = sparse_pairs_per_head(N, n_sink, window) + dense_pairs_per_head(N, gamma)
    return 4 * d * B * Hq * pairs


def dense_flops(B, Hq, N, d) -> int:
    return 4 * d * B * Hq * causal_pairs_per_head(N)


def approx_window_size(C: int, window: int, gamma: int) -> float:
    """The appendix's amortised keys per row: w + C / (2 gamma)."""
    return window + C / (2.0 * gamma)


def hbm_bytes(B, Hq, Hkv, N, d, gamma) -> int:
    """Compulsory HBM traffic of one prefill: read Q, K, V once, write O once
    (bf16), plus the fp32 dense rows of the samples written and read back."""
    ns = n_samples(N, gamma)
    return 2 * d * N * (2 * B * Hq + 2 * B * Hkv) + 2 * 4 * B * Hq * ns * d
