"""Delta smoothing (appendix "Interpolation", Alg. 2) through
delta_attn_prefill_smoothed, against the fp64 oracle element by element:
linear interpolation, the EMA over the rows and the alpha-beta-gamma filter
over the Delta vectors, over gamma that divides 128 and gamma that does not,
gamma = 1, gamma > 128, GQA, d = 64 and 128, ragged N, N = 1 and the dense tail;
then the full-size 131K workload on sampled rows.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.inputs import LLAMA8B_N131K, generate, to_bits
from gpu_helpers import MAX_ABS, MEAN_ABS, assert_close, oracle_full, rand_qkv

pytestmark = pytest.mark.gpu

ABG_PAPER = (0.2, 0.05, 0.0035)  # one of the paper's filter settings

# (B, Hq, Hkv, N, d, n_sink, window, gamma, smooth, params, tail_dense)
CASES = [
    (1, 2, 1, 300, 128, 4, 64, 16, "linear", (), 0),
    (2, 8, 2, 517, 128, 4, 100, 64, "ema", (0.5,), 0),
    (1, 4, 2, 333, 64, 8, 7, 3, "abg", ABG_PAPER, 0),
    (1, 4, 1, 1536, 128, 4, 300, 48, "ema", (0.95,), 100),
    (1, 2, 2, 400, 128, 0, 50, 5, "linear", (), 7),
    (1, 2, 1, 500, 128, 4, 64, 1, "ema", (0.75,), 0),         # gamma = 1
    (1, 4, 4, 520, 64, 4, 64, 4, "abg", (0.1, 5e-3, 1.66e-4), 0),
    (1, 2, 1, 700, 128, 4, 2048, 200, "linear", (), 0),       # window >= N: every Delta is 0
    (1, 2, 2, 1, 128, 4, 16, 4, "abg", (0.5, 0.4, 0.1), 0),   # N = 1
    (1, 8, 2, 1100, 128, 4, 96, 32, "abg", (0.05, 1.25e-4, 2.08e-5), 0),
]


def _ids(c):
    return "B%d_H%d-%d_N%d_d%d_s%d_w%d_g%d_%s_t%d" % (c[:9] + (c[10],))


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_smoothed_prefill_matches_oracle(case):
    B, Hq, Hkv, N, d, s, w, gamma, kind, par, tail = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case[:8]) + 19)
    ref = oracle_full(q, k, v, s, w, gamma, smooth=kind, smooth_params=par, tail_dense=tail)
    ws = binding.alloc_workspace(binding.workspace_size(B, Hq, Hkv, N, d, s, w, gamma, tail_dense=tail, smooth=kind),
                                 "cuda")
    out = binding.delta_attn_prefill(q, k, v, s, w, gamma, workspace=ws, tail_dense=tail, smooth=kind,
                                     smooth_params=par)
    assert binding.check() == binding.DA_OK
    assert_close(out, ref["A"], "smoothed prefill (%s)" % kind)


def test_smooth_none_is_plain_delta():
    """DA_SMOOTH_NONE through the smoothing entry point is the Eq. 6 prefill."""
    q, k, v = rand_qkv(1, 4, 2, 700, 128, seed=5)
    ref = binding.delta_attn_prefill(q, k, v, 4, 100, 16)
    out = torch.empty_like(q)
    rc = binding.load().delta_attn_prefill_smoothed(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), 1, 4, 2,
                                                    700, 128, 4, 100, 16, 0, 0.0, 0.0, 0.0, 0, None, 0, None)
    assert rc == binding.DA_OK
    torch.cuda.synchronize()
    assert torch.equal(out, ref)


def test_invalid_smoothing_arguments():
    q, k, v = rand_qkv(1, 2, 2, 64, 128, seed=3)
    lib = binding.load()
    for kind, c1 in ((4, 0.0), (-1, 0.0), (2, 1.5), (2, -0.1), (1, float("nan"))):
        rc = lib.delta_attn_prefill_smoothed(q.data_ptr(), k.data_ptr(), v.data_ptr(), q.data_ptr(), 1, 2, 2, 64,
                                             128, 4, 16, 4, kind, c1, 0.0, 0.0, 0, None, 0, None)
        assert rc == binding.DA_ERR_INVALID_ARG, (kind, c1, rc)


@pytest.mark.parametrize("kind,par", [("ema", (0.5,)), ("abg", ABG_PAPER), ("linear", ())])
def test_llama8b_n131k_smoothed(kind, par):
    """Full-size workload (N = 131072, scaled sink keys, gamma 64): rows at the
    start, a block in the middle and the last rows for two query heads on
    distinct KV heads, against the oracle (which runs the smoothing from row 0)."""
    W = LLAMA8B_N131K
    q, k, v = generate(W, device="cuda")
    ws = binding.alloc_workspace(binding.workspace_size(W.B, W.Hq, W.Hkv, W.N, W.d, W.n_sink, W.window, W.gamma,
                                                        smooth=kind), "cuda")
    out = binding.delta_attn_prefill(q, k, v, W.n_sink, W.window, W.gamma, workspace=ws, smooth=kind,
                                     smooth_params=par)
    assert binding.check() == binding.DA_OK
    Qb, Kb, Vb = to_bits(q), to_bits(k), to_bits(v)
    o = out.float()
    N = W.N
    errs = []
    for h, blocks in ((3, ((0, 2 * W.gamma), (N - 96, N))), (26, ((N // 2 - 40, N // 2 + 90),))):
        for (r0, r1) in blocks:
            ref = oracle.delta_attn(Qb, Kb, Vb, W.n_sink, W.window, W.gamma, heads=(h, h + 1), rows=(r0, r1),
                                    smooth=kind, smooth_params=par)["A"][0, 0]
            errs.append(np.abs(o[0, h, r0:r1].double().cpu().numpy() - ref).reshape(-1))
    err = np.concatenate(errs)
    assert np.all(np.isfinite(err))
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (kind, err.max(), err.mean())
