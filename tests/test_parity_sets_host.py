"""Host logic of the full-size parity sets: the sampled-row sets hold the
rows they claim (Eq. 4: rows k*gamma below N)."""
from test_gpu_workloads import EARLY_ROWS, sampled_rows


def test_all_sampled_rows():
    assert sampled_rows(640, 64) == list(range(0, 640, 64))
    assert sampled_rows(641, 64) == list(range(0, 641, 64))  # the partial last group has its sample
    assert sampled_rows(1, 7) == [0]


def test_spread_and_last_samples():
    N, g = 1 << 20, 64
    n_s = N // g
    s = sampled_rows(N, g, spread=192, last=64)
    assert s[0] == 0
    assert s[-64:] == [k * g for k in range(n_s - 64, n_s)]  # the longest dense rows
    assert len(s) >= 255 and s == sorted(set(s)) and all(r % g == 0 and r < N for r in s)


def test_early_rows_are_sink_rows():
    assert min(EARLY_ROWS) >= 1 and max(EARLY_ROWS) < 32
