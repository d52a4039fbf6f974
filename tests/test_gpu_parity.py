"""CUDA path (through the C ABI) against the fp64 oracle, element by element.

Small shapes are compared in full: several 128-row tiles and a ragged tail,
every branch of the launch sequence (Delta fused inside the row tile when
gamma divides 128, the separate Delta pass otherwise, gamma = 1 dense), GQA
ratios 1/2/4/8, d = 64 and 128, split-K and the degenerate cases.
"""
import numpy as np
import pytest
import torch

from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.flops import n_samples
from paper_2505_11254_gb300.inputs import TINY_N2048, generate
from gpu_helpers import assert_close, oracle_full, rand_qkv

pytestmark = pytest.mark.gpu

# (B, Hq, Hkv, N, d, n_sink, window, gamma)
CASES = [
    (1, 2, 1, 300, 128, 4, 64, 16),       # ragged N, GQA 2
    (2, 8, 2, 517, 128, 4, 100, 64),      # B = 2, GQA 4, ragged, gamma 64
    (1, 8, 1, 640, 64, 2, 128, 32),       # GQA 8, d = 64
    (1, 2, 2, 400, 128, 0, 50, 5),        # gamma does not divide 128, no sinks
    (1, 4, 2, 333, 64, 8, 7, 3),          # gamma 3, small window
    (1, 2, 1, 700, 128, 4, 2048, 200),    # window >= N, gamma > 128
    (1, 2, 2, 256, 128, 300, 16, 8),      # n_sink >= window and > N
    (1, 2, 2, 1, 128, 4, 16, 4),          # N = 1
    (1, 2, 1, 500, 128, 4, 64, 1),        # gamma = 1: dense causal attention
    (1, 4, 4, 129, 64, 1, 1, 128),        # window = 1, gamma = 128
    (1, 2, 2, 1000, 128, 4, 256, 1000),   # a single sample
    (1, 4, 1, 1536, 128, 4, 300, 48),     # gamma 48 (not a divisor of 128), split-K
    (1, 4, 2, 700, 128, 4, 100, 4),       # gamma 4 at d = 128: Delta built in a separate pass
    (2, 2, 2, 300, 128, 2, 40, 2),        # gamma 2
    (1, 16, 1, 400, 128, 4, 64, 16),      # GQA 16: 16 heads x 8 samples per dense tile
    (1, 6, 2, 350, 64, 3, 50, 8),         # GQA 3 (not a power of two): one head per dense tile
    (1, 4, 4, 520, 64, 4, 64, 4),         # gamma 4 at d = 64: fused in the tile
    (1, 4, 2, 1200, 128, 16, 200, 16),    # 16 sinks: the narrow sink tile, every key of it visible
    (1, 4, 2, 1200, 128, 17, 200, 16),    # 17 sinks: the full-width sink tile
    (1, 2, 1, 900, 64, 15, 128, 32),      # narrow sink tile at d = 64
    (1, 2, 2, 1100, 128, 1, 300, 64),     # one sink key
]


def _ids(c):
    return "B%d_H%d-%d_N%d_d%d_s%d_w%d_g%d" % c


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_prefill_matches_oracle(case):
    B, Hq, Hkv, N, d, s, w, gamma = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case))
    ref = oracle_full(q, k, v, s, w, gamma)
    out = binding.delta_attn_prefill(q, k, v, s, w, gamma)
    assert binding.check() == binding.DA_OK
    assert_close(out, ref["A"], "prefill")


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_standalone_entry_points_match_oracle(case):
    B, Hq, Hkv, N, d, s, w, gamma = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case) + 1)
    ref = oracle_full(q, k, v, s, w, gamma)
    ns = n_samples(N, gamma)
    s_samp = torch.empty((B, Hq, ns, d), dtype=torch.float32, device="cuda")
    o_sp = binding.sparse_window_attn(q, k, v, s, w, gamma, s_sampled=s_samp)
    d_samp = binding.strided_dense_attn(q, k, v, gamma)
    torch.cuda.synchronize()
    assert_close(o_sp, ref["S"], "sparse_window_attn")
    assert_close(s_samp, ref["S"][:, :, ::gamma], "sparse rows at the samples")
    assert_close(d_samp, ref["D"], "strided_dense_attn")
    out = binding.delta_apply(o_sp, s_samp, d_samp, gamma)
    assert_close(out, ref["A"], "delta_apply")
    # S_{k gamma} taken from the bf16 sparse output, in place
    o_sp2 = o_sp.clone()
    binding.delta_apply(o_sp2, None, d_samp, gamma, out=o_sp2)
    assert binding.check() == binding.DA_OK
    assert_close(o_sp2, ref["A"], "delta_apply in place")


def test_tiny_workload_full():
    """The tiny seeded workload (B1 H4 d64 N2048 w256 gamma16), every element."""
    q, k, v = generate(TINY_N2048, device="cuda")
    W = TINY_N2048
    ref = oracle_full(q, k, v, W.n_sink, W.window, W.gamma)
    out = binding.delta_attn_prefill(q, k, v, W.n_sink, W.window, W.gamma)
    assert binding.check() == binding.DA_OK
    assert_close(out, ref["A"], "tiny workload")
    # the sparse part alone differs from the corrected output: Delta is not zero
    assert float(np.abs(ref["A"] - ref["S"]).max()) > 1e-2


def test_caller_workspace_and_determinism():
    q, k, v = rand_qkv(1, 8, 2, 1200, 128, seed=7)
    nbytes = binding.workspace_size(1, 8, 2, 1200, 128, 4, 256, 16)
    ws = binding.alloc_workspace(nbytes, "cuda")
    a = binding.delta_attn_prefill(q, k, v, 4, 256, 16, workspace=ws)
    b = binding.delta_attn_prefill(q, k, v, 4, 256, 16, workspace=ws)
    c = binding.delta_attn_prefill(q, k, v, 4, 256, 16)
    assert binding.check() == binding.DA_OK
    assert torch.equal(a, b) and torch.equal(a, c), "results must be bit-identical across calls"
    small = binding.alloc_workspace(max(nbytes - 256, 16), "cuda")
    with pytest.raises(binding.DeltaAttnError) as e:
        binding.delta_attn_prefill(q, k, v, 4, 256, 16, workspace=small)
    assert e.value.status == binding.DA_ERR_WORKSPACE


def test_closed_form_zero_keys():
    """K = 0: uniform softmax, so S_i is the mean of v over W(i) and D_i the
    prefix mean: the kernels must reproduce these means (within bf16)."""
    B, Hq, Hkv, N, d, s, w, gamma = 1, 2, 1, 700, 128, 4, 100, 16
    q, _, v = rand_qkv(B, Hq, Hkv, N, d, seed=3)
    k = torch.zeros_like(v)
    vf = v.double().cpu().numpy()[0, 0]
    pre = np.concatenate([np.zeros((1, d)), np.cumsum(vf, axis=0)])
    out = binding.delta_attn_prefill(q, k, v, s, w, gamma).double().cpu().numpy()
    for i in range(N):
        a = max(0, i - w + 1)
        S_i = (pre[i + 1] - pre[a] + pre[min(s, a)]) / ((i - a + 1) + min(s, a))
        ks = (i // gamma) * gamma
        aks = max(0, ks - w + 1)
        S_k = (pre[ks + 1] - pre[aks] + pre[min(s, aks)]) / ((ks - aks + 1) + min(s, aks))
        want = pre[ks + 1] / (ks + 1) if i == ks else S_i + pre[ks + 1] / (ks + 1) - S_k
        assert np.abs(out[0, 0, i] - want).max() <= 2e-2, i


def test_window_one_no_sinks_is_identity():
    """window = 1, n_sink = 0: the sparse output is v_i itself."""
    q, k, v = rand_qkv(1, 2, 2, 384, 128, seed=5)
    o = binding.sparse_window_attn(q, k, v, 0, 1, 16)
    torch.cuda.synchronize()
    assert (o.float() - v.float()).abs().max().item() == 0.0


def test_timeout_path_reports_and_recovers():
    """A wait that nothing completes gives up after its limit and reports
    DA_ERR_TIMEOUT; the context stays usable."""
    assert binding.check() == binding.DA_OK
    binding.debug_timeout(20_000_000)  # 20 ms
    assert binding.check() == binding.DA_ERR_TIMEOUT
    assert binding.check() == binding.DA_OK  # cleared
    q, k, v = rand_qkv(1, 2, 2, 256, 64, seed=9)
    ref = oracle_full(q, k, v, 4, 32, 16)
    out = binding.delta_attn_prefill(q, k, v, 4, 32, 16)
    assert binding.check() == binding.DA_OK
    assert_close(out, ref["A"], "after timeout")


@pytest.mark.parametrize("d", [64, 128])
def test_score_jump_inside_one_key_tile(d):
    """Keys 64..127 and 320..383 scaled x32 give score jumps of more than
    64 log2 units: inside the first key tile of rows 64..127, and, for the
    rows past 384, in a tile that comes after others, so the lazy rescale of
    O and the row sum (taken only past that threshold) runs in the middle of
    rows, in both the sink+window and the dense kernels.
    Such sharp rows return nearly single values of v, and A = S + D - S_k can
    reach twice their range, so v is scaled by 1/8 (exact in bf16) to keep
    the bf16 rounding of the output itself well inside the tolerance."""
    B, Hq, Hkv, N, s, w, gamma = 1, 2, 1, 700, 4, 200, 16
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=11 + d)
    k, v = k.clone(), v * 0.125
    k[:, :, 64:128] *= 32
    k[:, :, 320:384] *= 32
    ref = oracle_full(q, k, v, s, w, gamma)
    out = binding.delta_attn_prefill(q, k, v, s, w, gamma)
    o_sp = binding.sparse_window_attn(q, k, v, s, w, gamma)
    d_samp = binding.strided_dense_attn(q, k, v, gamma)
    assert binding.check() == binding.DA_OK
    assert_close(out, ref["A"], "prefill")
    assert_close(o_sp, ref["S"], "sparse_window_attn")
    assert_close(d_samp, ref["D"], "strided_dense_attn")
