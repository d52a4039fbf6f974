"""Full-size seeded workloads through delta_attn_prefill (the launch
configuration bench.py times), checked against the fp64 oracle on sampled
outputs: the first two gamma-groups and the last group of rows (contiguous
blocks, one dense row per group), seeded random rows, the sink-dominated first
rows, for query heads on distinct KV heads (and distinct sequences for B=4).
Tolerance: max-abs 2e-2, mean-abs 2e-3 per checked set."""
import numpy as np
import pytest
import torch

import oracle
from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.inputs import (LLAMA8B_N1M, LLAMA8B_N131K, LLAMA8B_N32K, SWEEP_B4_N64K, SWEEP_GAMMAS,
                                           SWEEP_WINDOWS, generate, to_bits)
from gpu_helpers import MAX_ABS, MEAN_ABS

pytestmark = pytest.mark.gpu


def _check(w, q, k, v, out, bh_pairs, n_random, seed=0):
    Qb, Kb, Vb = to_bits(q), to_bits(k), to_bits(v)
    o = out.float()
    g, N = w.gamma, w.N
    errs = []
    for (b, h) in bh_pairs:
        blocks = [(0, min(2 * g, N)), (((N - 1) // g) * g, N)]
        for (r0, r1) in blocks:
            ref = oracle.delta_attn(Qb, Kb, Vb, w.n_sink, w.window, g, batches=(b, b + 1), heads=(h, h + 1),
                                    rows=(r0, r1))["A"][0, 0]
            got = o[b, h, r0:r1].double().cpu().numpy()
            errs.append(np.abs(got - ref))
    rng = np.random.default_rng(seed)
    rows = []
    for (b, h) in bh_pairs:
        for i in rng.integers(0, N, n_random):
            rows.append((b, h, int(i)))
        for i in (1, 2, 3, 5, 9):  # sink-dominated early rows
            rows.append((b, h, i))
    ref = oracle.rows(Qb, Kb, Vb, w.n_sink, w.window, g, rows)["A"]
    got = torch.stack([o[b, h, i] for (b, h, i) in rows]).double().cpu().numpy()
    errs.append(np.abs(got - ref))
    err = np.concatenate([e.reshape(-1) for e in errs])
    assert np.all(np.isfinite(err))
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (w.name, err.max(), err.mean())
    return err.max(), err.mean()


def _prefill(w, q, k, v):
    ws = binding.alloc_workspace(binding.workspace_size(w.B, w.Hq, w.Hkv, w.N, w.d, w.n_sink, w.window, w.gamma),
                                 q.device)
    out = binding.delta_attn_prefill(q, k, v, w.n_sink, w.window, w.gamma, workspace=ws)
    assert binding.check() == binding.DA_OK
    return out


def test_llama8b_n32k():
    w = LLAMA8B_N32K
    q, k, v = generate(w, device="cuda")
    out = _prefill(w, q, k, v)
    _check(w, q, k, v, out, [(0, 0), (0, 9), (0, 18), (0, 31)], n_random=48)


def test_llama8b_n131k_sinks():
    w = LLAMA8B_N131K
    q, k, v = generate(w, device="cuda")
    out = _prefill(w, q, k, v)
    _check(w, q, k, v, out, [(0, 0), (0, 13), (0, 22), (0, 31)], n_random=32)


def test_llama8b_n1m():
    w = LLAMA8B_N1M
    q, k, v = generate(w, device="cuda")
    out = _prefill(w, q, k, v)
    _check(w, q, k, v, out, [(0, 5), (0, 30)], n_random=8)


@pytest.mark.parametrize("window", SWEEP_WINDOWS)
def test_b4_n64k_sweep(window):
    w0 = SWEEP_B4_N64K.with_(window=window)
    q, k, v = generate(w0, device="cuda")
    for gamma in SWEEP_GAMMAS:
        w = w0.with_(gamma=gamma)
        out = _prefill(w, q, k, v)
        _check(w, q, k, v, out, [(0, 3), (1, 12), (2, 21), (3, 30)], n_random=6, seed=gamma)
        del out
