"""Full-size seeded workloads through delta_attn_prefill (the launch
configuration bench.py times), checked element by element against the fp64
oracle on sets of output rows, each set with its own max-abs and mean-abs:

  groups   every row of the first two gamma-groups and of the last group
           (Eq. 6 rows around their samples; the last group of a long
           sequence holds the longest dense row)
  sampled  the sampled rows k*gamma (Eq. 4): every one at 32K, 131K and in the
           B=4 sweep; at 1M 192 evenly spaced samples plus the last 64, whose
           dense rows (about 1M keys each) are the longest split-K merges
  random   seeded uniformly random rows (1024 per pair; 128 per pair and
           point in the B=4 sweep)
  early    rows 1, 2, 3, 5, 9, 17: dominated by the sink keys (scaled x8 at
           131K)

for four (b, h) pairs on distinct KV heads (and distinct sequences for B=4);
the small 2048-token configuration is compared on every element.
Tolerance: max-abs 2e-2, mean-abs 2e-3 per set.  With DA_PARITY_RECORD set to
a file name, every set's figures are appended to it as JSON lines.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.inputs import (LLAMA8B_N1M, LLAMA8B_N131K, LLAMA8B_N32K, SWEEP_B4_N64K, SWEEP_GAMMAS,
                                           SWEEP_WINDOWS, TINY_N2048, generate, to_bits)
from gpu_helpers import MAX_ABS, MEAN_ABS

pytestmark = pytest.mark.gpu

EARLY_ROWS = (1, 2, 3, 5, 9, 17)


def sampled_rows(N, gamma, spread=None, last=0):
    """Sampled rows k*gamma: all of them, or `spread` evenly spaced samples
    plus the last `last` samples."""
    n_s = (N + gamma - 1) // gamma
    if spread is None:
        ks = np.arange(n_s)
    else:
        ks = np.unique(np.concatenate([np.linspace(0, n_s - 1 - last, spread).astype(np.int64),
                                       np.arange(max(0, n_s - last), n_s)]))
    return [int(k) * gamma for k in ks]


def _record(entry):
    path = os.environ.get("DA_PARITY_RECORD")
    if path:
        with open(path, "a") as f:
            f.write(json.dumps(entry) + "\n")


def _assert_set(w, name, got, ref, stats):
    err = np.abs(got - ref)
    assert np.all(np.isfinite(got)), (w.name, name, "non-finite output")
    mx, mn = float(err.max()), float(err.mean())
    stats[name] = {"rows": int(err.size // w.d), "max_abs": mx, "mean_abs": mn}
    assert mx <= MAX_ABS and mn <= MEAN_ABS, (w.name, name, mx, mn)


def _check(w, q, k, v, out, bh_pairs, n_random, seed=0, spread=None, last=0):
    """Compare `out` with the oracle on the four sets of every (b, h) pair;
    returns the per-set figures."""
    Qb, Kb, Vb = to_bits(q), to_bits(k), to_bits(v)
    g, N = w.gamma, w.N
    rng = np.random.default_rng(seed)
    samples = sampled_rows(N, g, spread, last)
    stats = {}
    per_set = {"groups": ([], []), "sampled": ([], []), "random": ([], []), "early": ([], [])}
    for (b, h) in bh_pairs:
        # groups 0 and 1 and the last group, through the box form of the oracle
        # (one dense row per group)
        for (r0, r1) in ((0, min(2 * g, N)), (((N - 1) // g) * g, N)):
            ref = oracle.delta_attn(Qb, Kb, Vb, w.n_sink, w.window, g, batches=(b, b + 1), heads=(h, h + 1),
                                    rows=(r0, r1))["A"][0, 0]
            per_set["groups"][0].append(out[b, h, r0:r1].double().cpu().numpy())
            per_set["groups"][1].append(ref)
        # single rows through the per-row form
        for name, rows in (("sampled", samples), ("random", [int(i) for i in rng.integers(0, N, n_random)]),
                           ("early", [i for i in EARLY_ROWS if i < N])):
            bhi = [(b, h, i) for i in rows]
            ref = oracle.rows(Qb, Kb, Vb, w.n_sink, w.window, g, bhi)["A"]
            idx = torch.tensor(rows, dtype=torch.long, device=out.device)
            per_set[name][0].append(out[b, h].index_select(0, idx).double().cpu().numpy())
            per_set[name][1].append(ref)
    for name, (got, ref) in per_set.items():
        _assert_set(w, name, np.concatenate(got), np.concatenate(ref), stats)
    _record({"workload": w.name, "window": w.window, "gamma": w.gamma, "pairs": [list(p) for p in bh_pairs],
             "sets": stats})
    return stats


def _prefill(w, q, k, v):
    ws = binding.alloc_workspace(binding.workspace_size(w.B, w.Hq, w.Hkv, w.N, w.d, w.n_sink, w.window, w.gamma),
                                 q.device)
    out = binding.delta_attn_prefill(q, k, v, w.n_sink, w.window, w.gamma, workspace=ws)
    assert binding.check() == binding.DA_OK
    return out


def test_tiny_all_elements():
    """The small configuration (B=1, 4 heads, d=64, N=2048, window 256,
    gamma 16): every element of the output."""
    w = TINY_N2048
    q, k, v = generate(w, device="cuda")
    out = _prefill(w, q, k, v)
    ref = oracle.delta_attn(to_bits(q), to_bits(k), to_bits(v), w.n_sink, w.window, w.gamma)["A"]
    stats = {}
    _assert_set(w, "all", out.double().cpu().numpy(), ref, stats)
    _record({"workload": w.name, "window": w.window, "gamma": w.gamma, "pairs": "all", "sets": stats})


def test_llama8b_n32k():
    w = LLAMA8B_N32K
    q, k, v = generate(w, device="cuda")
    out = _prefill(w, q, k, v)
    _check(w, q, k, v, out, [(0, 0), (0, 9), (0, 18), (0, 31)], n_random=1024)


def test_llama8b_n131k_sinks():
    w = LLAMA8B_N131K
    q, k, v = generate(w, device="cuda")
    out = _prefill(w, q, k, v)
    _check(w, q, k, v, out, [(0, 0), (0, 13), (0, 22), (0, 31)], n_random=1024)


def test_llama8b_n1m():
    w = LLAMA8B_N1M
    q, k, v = generate(w, device="cuda")
    out = _prefill(w, q, k, v)
    _check(w, q, k, v, out, [(0, 5), (0, 14), (0, 23), (0, 30)], n_random=1024, spread=192, last=64)


@pytest.mark.parametrize("window", SWEEP_WINDOWS)
def test_b4_n64k_sweep(window):
    w0 = SWEEP_B4_N64K.with_(window=window)
    q, k, v = generate(w0, device="cuda")
    for gamma in SWEEP_GAMMAS:
        w = w0.with_(gamma=gamma)
        out = _prefill(w, q, k, v)
        _check(w, q, k, v, out, [(0, 3), (1, 12), (2, 21), (3, 30)], n_random=128, seed=gamma)
        del out
