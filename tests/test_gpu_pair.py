"""The two-CTA sink + window kernel (the query heads of a KV group taken two at
a time, one MMA issuer for both CTAs of a cluster) against the fp64 oracle and
against the one-CTA kernel, through the C ABI (DELTA_ATTN_PAIR=1 / 0 select
them).  The library takes the two-CTA kernel for whole sequences at d = 128
with an even GQA ratio and a window of at least 512 keys; the tests force it
at every window, and the cases cover every epilogue it is built with (the Delta
fused in the row tile, the separate Delta pass, bf16 rows for the recompute
form and sparse_window_attn, the smoothed correction), the RoPE rotation of Q
in the epilogue warps, ragged tails, several items per CTA (so every ring and
buffer index wraps) and GQA 2, 4 and 8."""
import os

import numpy as np
import pytest
import torch

from paper_2505_11254_gb300 import binding
from gpu_helpers import assert_close, oracle_full, rand_qkv

pytestmark = pytest.mark.gpu


class kernel_choice:
    """Within the block the sink + window pass runs as the two-CTA kernel
    (DELTA_ATTN_PAIR=1, wherever it applies, whatever the window) or the
    one-CTA kernel (DELTA_ATTN_PAIR=0)."""

    def __init__(self, value):
        self.value = value

    def __enter__(self):
        self.old = os.environ.get("DELTA_ATTN_PAIR")
        os.environ["DELTA_ATTN_PAIR"] = self.value

    def __exit__(self, *exc):
        if self.old is None:
            del os.environ["DELTA_ATTN_PAIR"]
        else:
            os.environ["DELTA_ATTN_PAIR"] = self.old


def one_cta_kernel():
    return kernel_choice("0")


def two_cta_kernel():
    return kernel_choice("1")


@pytest.fixture(autouse=True)
def _pair_by_default():
    """Every test of this file runs the two-CTA kernel unless it says otherwise."""
    with two_cta_kernel():
        yield


def _both(fn):
    a = fn()
    torch.cuda.synchronize()
    with one_cta_kernel():
        b = fn()
    torch.cuda.synchronize()
    assert binding.check() == binding.DA_OK
    return a, b


def _same(a, b, what):
    """The two kernels run the same arithmetic per row; their outputs agree to
    the bf16 rounding of the output at most."""
    d = (a.float() - b.float()).abs()
    assert float(d.max()) <= 2e-2 and float(d.mean()) <= 1e-4, "%s: pair vs one-CTA max %.3g mean %.3g" % (
        what, float(d.max()), float(d.mean()))


# (B, Hq, Hkv, N, d, n_sink, window, gamma)
CASES = [
    (1, 2, 1, 300, 128, 4, 64, 16),       # GQA 2, ragged N, one pair of items
    (2, 8, 2, 517, 128, 4, 100, 64),      # B = 2, GQA 4, ragged
    (1, 8, 1, 1000, 128, 4, 256, 48),     # GQA 8, Delta in its own pass (gamma does not divide 128)
    (1, 8, 2, 8192, 128, 4, 512, 64),     # 512 items: several per CTA, rings wrap
    (1, 4, 2, 1200, 128, 17, 200, 16),    # 17 sinks: a full-width sink tile
    (1, 4, 2, 700, 128, 4, 2048, 32),     # window >= N: every row dense
    (1, 2, 1, 1, 128, 4, 512, 4),         # N = 1: two items, one cluster
    (1, 4, 2, 130, 128, 0, 512, 2),       # no sinks, a 2-row ragged tile, gamma 2
]


def _ids(c):
    return "B%d_H%d-%d_N%d_d%d_s%d_w%d_g%d" % c


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_pair_prefill_matches_oracle_and_one_cta(case):
    B, Hq, Hkv, N, d, s, w, gamma = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case) + 7)
    ref = oracle_full(q, k, v, s, w, gamma)
    a, b = _both(lambda: binding.delta_attn_prefill(q, k, v, s, w, gamma))
    assert_close(a, ref["A"], "two-CTA prefill")
    assert_close(b, ref["A"], "one-CTA prefill")
    _same(a, b, "prefill")


@pytest.mark.parametrize("case", CASES[:3], ids=_ids)
def test_pair_sparse_rows_and_recompute(case):
    """EPI_BF16: sparse_window_attn (with the fp32 sampled rows) and the Eq. 5
    recompute form."""
    B, Hq, Hkv, N, d, s, w, gamma = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case) + 8)
    ref = oracle_full(q, k, v, s, w, gamma)
    ns = -(-N // gamma)
    s1 = torch.empty((B, Hq, ns, d), dtype=torch.float32, device="cuda")
    s2 = torch.empty_like(s1)
    a = binding.sparse_window_attn(q, k, v, s, w, gamma, s_sampled=s1)
    with one_cta_kernel():
        b = binding.sparse_window_attn(q, k, v, s, w, gamma, s_sampled=s2)
    torch.cuda.synchronize()
    assert binding.check() == binding.DA_OK
    assert_close(a, ref["S"], "two-CTA sparse rows")
    assert_close(s1, ref["S"][:, :, ::gamma], "two-CTA sampled sparse rows")
    _same(a, b, "sparse rows")
    assert float((s1 - s2).abs().max()) <= 1e-3
    ref_r = oracle_full(q, k, v, s, w, gamma, mode="recompute")
    ra, rb = _both(lambda: binding.delta_attn_prefill(q, k, v, s, w, gamma, mode="recompute"))
    assert_close(ra, ref_r["A"], "two-CTA recompute")
    _same(ra, rb, "recompute")


@pytest.mark.parametrize("kind, par", [("linear", ()), ("ema", (0.5,)), ("abg", (0.2, 0.05, 0.0035))])
def test_pair_smoothed(kind, par):
    B, Hq, Hkv, N, d, s, w, gamma = 1, 4, 2, 1100, 128, 4, 200, 16
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=31)
    ref = oracle_full(q, k, v, s, w, gamma, smooth=kind, smooth_params=par)
    a, b = _both(lambda: binding.delta_attn_prefill(q, k, v, s, w, gamma, smooth=kind, smooth_params=par))
    assert_close(a, ref["A"], "two-CTA smoothed (%s)" % kind)
    _same(a, b, "smoothed (%s)" % kind)


@pytest.mark.parametrize("case", [(1, 8, 2, 1500, 128, 4, 300, 64), (2, 4, 2, 700, 128, 4, 100, 48)], ids=_ids)
def test_pair_rope_fused(case):
    """Q rotated by the epilogue warps of each CTA, the leader's QK waiting for
    both rotations; K rotated in place by the call (so each call gets a copy)."""
    B, Hq, Hkv, N, d, s, w, gamma = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case) + 9)
    table = binding.rope_table(N, d, 500000.0)
    ka, kb = k.clone(), k.clone()
    a = binding.delta_attn_prefill_rope(q, ka, v, s, w, gamma, table)
    torch.cuda.synchronize()
    with one_cta_kernel():
        b = binding.delta_attn_prefill_rope(q, kb, v, s, w, gamma, table)
    torch.cuda.synchronize()
    assert binding.check() == binding.DA_OK
    assert torch.equal(ka, kb)
    _same(a, b, "RoPE-fused prefill")
    # against the oracle on the rotated inputs: rotate Q with the library and run the plain prefill
    qr = q.clone()
    binding.rope_apply(qr, table)
    torch.cuda.synchronize()
    ref = oracle_full(qr, ka, v, s, w, gamma)
    err = np.abs(a.double().cpu().numpy() - ref["A"])
    assert err.max() <= 2e-2 and err.mean() <= 2e-3, (err.max(), err.mean())


def test_pair_repeated_calls_bit_identical():
    q, k, v = rand_qkv(1, 8, 2, 4096, 128, seed=5)
    a = binding.delta_attn_prefill(q, k, v, 4, 512, 64)
    b = binding.delta_attn_prefill(q, k, v, 4, 512, 64)
    torch.cuda.synchronize()
    assert binding.check() == binding.DA_OK
    assert torch.equal(a, b)


def test_default_choice_follows_the_window():
    """Without the override the two kernels give the same bits at a short and a
    long window (the library picks one-CTA at window 256 and two-CTA at 2048)."""
    q, k, v = rand_qkv(1, 4, 2, 4608, 128, seed=12)
    env = os.environ.pop("DELTA_ATTN_PAIR")
    try:
        for w in (256, 2048):
            a = binding.delta_attn_prefill(q, k, v, 4, w, 64)
            with one_cta_kernel():
                b = binding.delta_attn_prefill(q, k, v, 4, w, 64)
            with two_cta_kernel():
                c = binding.delta_attn_prefill(q, k, v, 4, w, 64)
            torch.cuda.synchronize()
            assert torch.equal(a, b) and torch.equal(a, c)
    finally:
        os.environ["DELTA_ATTN_PAIR"] = env
    assert binding.check() == binding.DA_OK
