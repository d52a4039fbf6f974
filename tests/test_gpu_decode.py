"""Eq. 2 decoding over the cache (delta_attn_decode) against the fp64 oracle:
GQA ratios 1 to 16 (including ratios that are not powers of two), d = 64 and
128, per-sequence lengths shorter than the cache, a single key, lengths that
end inside a ring chunk, hundreds of key-range splits for one head, and the 131K-token cache of the prefill workload
with the new token's key and value appended."""
import numpy as np
import pytest
import torch

import oracle
from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.inputs import LLAMA8B_N131K, generate, to_bits
from gpu_helpers import assert_close

pytestmark = pytest.mark.gpu


def _rand(shape, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(shape, generator=g) * scale).to(torch.bfloat16).cuda()


# (B, Hq, Hkv, L, d, lens or None)
CASES = [
    (1, 32, 8, 4096, 128, None),
    (2, 8, 2, 1000, 128, [1000, 517]),
    (3, 4, 4, 300, 64, [1, 64, 300]),
    (1, 16, 2, 2049, 128, [2049]),
    (1, 16, 1, 700, 64, [650]),
    (2, 6, 2, 333, 128, [333, 200]),
    (1, 5, 1, 128, 128, [100]),
    (4, 2, 2, 70, 64, [65, 1, 70, 63]),
    # one (batch, KV head) pair: a wave of splits (more than the merge CTA's threads)
    (1, 1, 1, 65536, 64, None),
    (1, 2, 1, 40000, 128, [39999]),
]


def _ids(c):
    return "B%d_H%d-%d_L%d_d%d" % c[:5] + ("_lens" if c[5] else "")


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_decode_matches_oracle(case):
    B, Hq, Hkv, L, d, lens = case
    seed = B * 1000 + Hq * 10 + L
    q = _rand((B, Hq, d), seed, 1.5)
    K = _rand((B, Hkv, L, d), seed + 1, 1.5)
    V = _rand((B, Hkv, L, d), seed + 2)
    n = lens if lens is not None else [L] * B
    lt = torch.tensor(n, dtype=torch.int64, device="cuda") if lens is not None else None
    ws = binding.alloc_workspace(binding.decode_workspace_size(B, Hq, Hkv, max(n), d), "cuda")
    out = binding.decode(q, K, V, lens=lt, max_keys=max(n), workspace=ws)
    assert binding.check() == binding.DA_OK
    ref, dev = oracle.decode(to_bits(q), to_bits(K), to_bits(V), n)
    assert dev < 1e-12
    assert_close(out, ref, "decode")
    out2 = binding.decode(q, K, V, lens=lt, max_keys=max(n))  # library-allocated workspace
    torch.cuda.synchronize()
    assert torch.equal(out, out2)


def test_decode_after_131k_prefill():
    """The Llama-3.1-8B layer shape with the 131072-token prefill's K and V as
    the cache and one new token appended at index N (Eq. 2): all 32 heads."""
    W = LLAMA8B_N131K
    q_all, k, v = generate(W, device="cuda")
    N = W.N
    Kc = torch.zeros((1, W.Hkv, N + 1, W.d), dtype=torch.bfloat16, device="cuda")
    Vc = torch.zeros_like(Kc)
    Kc[:, :, :N] = k
    Vc[:, :, :N] = v
    Kc[:, :, N] = _rand((1, W.Hkv, W.d), 77)
    Vc[:, :, N] = _rand((1, W.Hkv, W.d), 78)
    q = _rand((1, W.Hq, W.d), 79)
    out = binding.decode(q, Kc, Vc)
    assert binding.check() == binding.DA_OK
    ref, _ = oracle.decode(to_bits(q), to_bits(Kc), to_bits(Vc), [N + 1])
    assert_close(out, ref, "decode at 131K")
