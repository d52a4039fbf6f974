"""delta_attn_prefill_rows, one rank's share of a sequence split by rows
(context parallelism), against the fp64 oracle and the whole-sequence call.

A sequence is cut into row ranges that start on a 128-row tile and a sample
group (a multiple of lcm(128, gamma)); each range is computed from its own
rows of Q and the K, V of the whole sequence, as a rank does after gathering
K and V, and the ranges together must give the whole-sequence output (Eq. 6
evaluates every row from its query and the keys up to it)."""
import numpy as np
import pytest
import torch

from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.inputs import LLAMA8B_N32K, generate
from paper_2505_11254_gb300.replicas import context_shard
from gpu_helpers import MAX_ABS, MEAN_ABS, assert_close, oracle_full, oracle_rows, rand_qkv

pytestmark = pytest.mark.gpu

# (B, Hq, Hkv, N, d, n_sink, window, gamma, ranks)
CASES = [
    (1, 4, 2, 1000, 128, 4, 200, 16, 3),     # ragged last range
    (2, 8, 2, 1536, 128, 4, 300, 64, 2),     # B = 2, GQA 4
    (1, 4, 1, 1600, 64, 2, 128, 48, 2),      # gamma 48: Delta built in its own pass, ranges of 384 rows
    (1, 2, 2, 700, 128, 0, 64, 1, 4),        # gamma = 1: dense causal rows
    (1, 2, 1, 900, 128, 300, 100, 4, 3),     # n_sink > window, gamma 4 (separate Delta pass at d = 128)
    (1, 16, 1, 1100, 64, 4, 1000, 32, 2),    # GQA 16, window covering most of the sequence
]


def _ids(c):
    return "B%d_H%d-%d_N%d_d%d_s%d_w%d_g%d_r%d" % c


def _split(q, k, v, n_sink, window, gamma, ranks):
    N = q.shape[2]
    parts = []
    for r in range(ranks):
        r0, r1 = context_shard(N, gamma, r, ranks)
        if r1 <= r0:
            continue
        q_rows = q[:, :, r0:r1].contiguous()
        ws = binding.alloc_workspace(
            binding.workspace_size_rows(q.shape[0], q.shape[1], k.shape[1], N, q.shape[3], n_sink, window, gamma,
                                        r0, r1 - r0), q.device)
        parts.append(binding.delta_attn_prefill_rows(q_rows, k, v, n_sink, window, gamma, r0, workspace=ws))
        assert binding.check() == binding.DA_OK
    return torch.cat(parts, dim=2)


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_row_ranges_match_oracle_and_whole_sequence(case):
    B, Hq, Hkv, N, d, s, w, gamma, ranks = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case) + 7)
    got = _split(q, k, v, s, w, gamma, ranks)
    ref = oracle_full(q, k, v, s, w, gamma)
    assert_close(got, ref["A"], "row ranges")
    whole = binding.delta_attn_prefill(q, k, v, s, w, gamma)
    assert_close(got, whole.double().cpu().numpy(), "row ranges vs the whole sequence")


def test_llama8b_n32k_four_ranks():
    """The 32K-token layer as four ranks of 8192 rows: sampled rows, random
    rows and each range's first and last rows against the oracle."""
    wl = LLAMA8B_N32K
    q, k, v = generate(wl, device="cuda")
    got = _split(q, k, v, wl.n_sink, wl.window, wl.gamma, 4)
    rng = np.random.default_rng(3)
    rows = sorted(set([int(i) for i in rng.integers(0, wl.N, 512)] + list(range(0, wl.N, 8 * wl.gamma)) +
                      [r for b in (8192, 16384, 24576) for r in (b - 1, b, b + 1, b + 63)]))
    for h in (0, 11, 22, 31):
        ref = oracle_rows(q, k, v, wl.n_sink, wl.window, wl.gamma, [(0, h, i) for i in rows])["A"]
        err = np.abs(got[0, h, rows].double().cpu().numpy() - ref)
        assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (h, err.max(), err.mean())


def test_row_range_keys_past_the_range_are_not_needed():
    """K and V may end at the range's last row: a range computed with K, V cut
    there equals the same range computed with the whole sequence's K, V."""
    B, Hq, Hkv, N, d, s, w, gamma = 1, 4, 2, 1024, 128, 4, 256, 16
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=91)
    r0, r1 = 256, 640
    a = binding.delta_attn_prefill_rows(q[:, :, r0:r1].contiguous(), k, v, s, w, gamma, r0)
    b = binding.delta_attn_prefill_rows(q[:, :, r0:r1].contiguous(), k[:, :, :r1].contiguous(),
                                        v[:, :, :r1].contiguous(), s, w, gamma, r0)
    assert binding.check() == binding.DA_OK
    assert torch.equal(a, b)


@pytest.mark.parametrize("row_begin, gamma", [(100, 4), (128, 48), (-128, 16)])
def test_row_range_rejects_unaligned_starts(row_begin, gamma):
    q, k, v = rand_qkv(1, 2, 1, 512, 128, seed=5)
    with pytest.raises(binding.DeltaAttnError) as e:
        binding.delta_attn_prefill_rows(q[:, :, :128].contiguous(), k, v, 4, 64, gamma, row_begin)
    assert e.value.status == binding.DA_ERR_INVALID_ARG
