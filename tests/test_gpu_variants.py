"""The paper's two ablation forms through delta_attn_prefill_ex, against the
fp64 oracle element by element: the Eq. 5 "recompute" output (dense rows only
at the samples) and the dense tail block of the appendix "Implementation
Details" (the last rows dense), alone and together.  Cases cover gamma that
divides 128 (Delta fused in the row tile) and gamma that does not, GQA, d = 64
and 128, tails that start inside a 128-row tile, split-K inside the tail pass,
a tail of the whole sequence and gamma = 1 (both options moot).
"""
import numpy as np
import pytest
import torch

from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.inputs import LLAMA8B_N131K, generate, to_bits
from gpu_helpers import MAX_ABS, MEAN_ABS, assert_close, oracle_full, rand_qkv

import oracle

pytestmark = pytest.mark.gpu

# (B, Hq, Hkv, N, d, n_sink, window, gamma, mode, tail_dense)
CASES = [
    (1, 2, 1, 300, 128, 4, 64, 16, "recompute", 0),
    (2, 8, 2, 517, 128, 4, 100, 64, "recompute", 0),
    (1, 4, 2, 333, 64, 8, 7, 3, "recompute", 0),       # gamma 3: not a divisor of 128
    (1, 4, 1, 1536, 128, 4, 300, 48, "recompute", 0),  # split-K sampled rows
    (1, 2, 1, 300, 128, 4, 64, 16, "delta", 44),       # tail starts on a tile boundary (row 256)
    (2, 8, 2, 517, 128, 4, 100, 64, "delta", 5),       # ragged tail
    (1, 4, 2, 700, 128, 4, 100, 4, "delta", 200),      # Delta in a separate pass, tail over two tiles
    (1, 8, 1, 640, 64, 2, 128, 32, "delta", 640),      # tail = N: every row dense
    (1, 2, 2, 1, 128, 4, 16, 4, "delta", 1),           # N = 1
    (1, 4, 1, 1536, 128, 4, 300, 48, "recompute", 300),  # both; split-K inside the tail pass
    (1, 2, 1, 500, 128, 4, 64, 1, "recompute", 100),   # gamma = 1: dense causal attention
    (1, 4, 4, 520, 64, 4, 64, 4, "delta", 129),        # gamma 4 at d = 64, tail of 129 rows
]


def _ids(c):
    return "B%d_H%d-%d_N%d_d%d_s%d_w%d_g%d_%s_t%d" % c


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_variant_matches_oracle(case):
    B, Hq, Hkv, N, d, s, w, gamma, mode, tail = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case[:8]) + 7)
    ref = oracle_full(q, k, v, s, w, gamma, mode=mode, tail_dense=tail)
    ws = binding.alloc_workspace(binding.workspace_size(B, Hq, Hkv, N, d, s, w, gamma, mode, tail), "cuda")
    out = binding.delta_attn_prefill(q, k, v, s, w, gamma, workspace=ws, mode=mode, tail_dense=tail)
    assert binding.check() == binding.DA_OK
    assert_close(out, ref["A"], "prefill %s tail %d" % (mode, tail))
    # allocation by the library when no workspace is given
    out2 = binding.delta_attn_prefill(q, k, v, s, w, gamma, mode=mode, tail_dense=tail)
    assert binding.check() == binding.DA_OK
    assert torch.equal(out, out2)


def test_recompute_differs_from_delta_only_between_samples():
    """Eq. 5 and Eq. 6 agree at the sampled rows (both give the dense row) and
    the recompute rows between samples equal the sink+window output bit for
    bit (the same kernel writes them)."""
    B, Hq, Hkv, N, d, s, w, gamma = 1, 4, 2, 1100, 128, 4, 96, 16
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=11)
    rec = binding.delta_attn_prefill(q, k, v, s, w, gamma, mode="recompute")
    dlt = binding.delta_attn_prefill(q, k, v, s, w, gamma)
    sp = binding.sparse_window_attn(q, k, v, s, w, gamma)
    torch.cuda.synchronize()
    between = torch.ones(N, dtype=torch.bool, device="cuda")
    between[::gamma] = False
    assert torch.equal(rec[:, :, between], sp[:, :, between])
    # the same fp32 dense row, rounded to bf16 on each side: at most one bf16 ulp apart
    assert torch.allclose(rec[:, :, ::gamma].float(), dlt[:, :, ::gamma].float(), rtol=2.0 ** -7, atol=1e-6)


def test_invalid_variant_arguments():
    q, k, v = rand_qkv(1, 2, 2, 64, 128, seed=3)
    for mode, tail in ((2, 0), (-1, 0), (0, -1), (0, 65)):
        rc = binding.load().delta_attn_prefill_ex(q.data_ptr(), k.data_ptr(), v.data_ptr(), q.data_ptr(), 1, 2, 2,
                                                  64, 128, 4, 16, 4, mode, tail, None, 0, None)
        assert rc == binding.DA_ERR_INVALID_ARG, (mode, tail, rc)


def test_llama8b_n131k_recompute_with_tail():
    """Full-size workload (Llama-3.1-8B layer shape, N = 131072, scaled sink
    keys) with recompute and a 1000-row dense tail: rows around the tail's
    start, the last rows, and sampled and unsampled rows early on, for query
    heads on distinct KV heads, against the oracle on those rows."""
    W = LLAMA8B_N131K
    tail = 1000
    q, k, v = generate(W, device="cuda")
    ws = binding.alloc_workspace(binding.workspace_size(W.B, W.Hq, W.Hkv, W.N, W.d, W.n_sink, W.window, W.gamma,
                                                        "recompute", tail), "cuda")
    out = binding.delta_attn_prefill(q, k, v, W.n_sink, W.window, W.gamma, workspace=ws, mode="recompute",
                                     tail_dense=tail)
    assert binding.check() == binding.DA_OK
    Qb, Kb, Vb = to_bits(q), to_bits(k), to_bits(v)
    o = out.float()
    N = W.N
    errs = []
    for h in (0, 17, 30):
        for (r0, r1) in ((0, 2 * W.gamma), (N - tail - 40, N - tail + 24), (N - 16, N)):
            ref = oracle.delta_attn(Qb, Kb, Vb, W.n_sink, W.window, W.gamma, heads=(h, h + 1), rows=(r0, r1),
                                    mode="recompute", tail_dense=tail)["A"][0, 0]
            errs.append(np.abs(o[0, h, r0:r1].double().cpu().numpy() - ref).reshape(-1))
    err = np.concatenate(errs)
    assert np.all(np.isfinite(err))
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (err.max(), err.mean())
