"""Work accounting (host logic) against brute-force counts and the paper's
worked example (tests/golden/approx_window_size.txt)."""
import os

import pytest

from paper_2505_11254_gb300 import flops

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "approx_window_size.txt")


def _golden():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if line and not line.startswith("#"):
            rows.append(dict(kv.split("=") for kv in line.split()))
    return rows


def _brute_pairs(N, n_sink, window, gamma):
    sparse = sum(1 for i in range(N) for j in range(i + 1) if j < n_sink or j > i - window)
    dense = sum(i + 1 for i in range(0, N, gamma))
    return sparse, dense


@pytest.mark.parametrize("N,n_sink,window,gamma", [
    (1, 0, 1, 1), (1, 4, 256, 16), (37, 4, 7, 5), (64, 0, 1, 64), (100, 10, 3, 7),
    (129, 4, 64, 16), (300, 200, 50, 33), (257, 4, 1000, 1)])
def test_pair_counts_match_brute_force(N, n_sink, window, gamma):
    s, d = _brute_pairs(N, n_sink, window, gamma)
    assert flops.sparse_pairs_per_head(N, n_sink, window) == s
    assert flops.dense_pairs_per_head(N, gamma) == d
    assert flops.n_samples(N, gamma) == len(range(0, N, gamma))


def test_worked_example_approx_window_size():
    g = _golden()[0]
    C, w, gamma = int(g["C"]), int(g["window"]), int(g["gamma"])
    assert flops.approx_window_size(C, w, gamma) == float(g["approx_keys_per_row"])
    # the exact count per row (sinks, the first-window triangle and the +1
    # terms included) is within 1% of the paper's amortised figure
    exact = (flops.sparse_pairs_per_head(C, 4, w) + flops.dense_pairs_per_head(C, gamma)) / C
    assert abs(exact - 3072) / 3072 < 0.01


def test_sampling_fraction():
    g = _golden()[1]
    gamma = int(g["gamma"])
    frac = flops.n_samples(1 << 20, gamma) / (1 << 20)
    assert abs(100 * frac - float(g["extra_percent"])) < 0.1
    assert abs(100 * (1 - frac) - float(g["sparsity_percent"])) < 0.1


def test_dense_flops_gamma1():
    # gamma = 1 makes every row a dense causal row
    assert flops.dense_pairs_per_head(1000, 1) == flops.causal_pairs_per_head(1000)


def test_tail_pairs_brute_force():
    for N, t in ((1, 1), (10, 3), (300, 44), (517, 0), (64, 64), (64, 100)):
        assert flops.tail_pairs_per_head(N, t) == sum(i + 1 for i in range(max(0, N - t), N))
