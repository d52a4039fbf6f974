"""RoPE (Sec. 2) through the C ABI against the fp64 oracle: the (cos, sin)
table, the in-place rotation of K (at most one bf16 step from the oracle's
single rounding), the prefill with RoPE fused into the Q tiles
(delta_attn_prefill_rope) over the launch paths (Delta fused in the row tile,
the separate Delta pass, gamma = 1 dense), a decode query rotated to its
position, and the 131K workload shape on sampled rows."""
import numpy as np
import pytest
import torch

import oracle
from paper_2505_11254_gb300 import binding
from paper_2505_11254_gb300.inputs import to_bits
from gpu_helpers import MAX_ABS, MEAN_ABS, assert_close, rand_qkv

pytestmark = pytest.mark.gpu

BASE = 500000.0


def _bits_to_t(bits):
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16)


def test_rope_table():
    n, d = 70000, 128
    t = binding.rope_table(n, d, BASE).cpu().numpy()
    pos = np.arange(n, dtype=np.float64)[:, None]
    ang = pos * BASE ** (-2.0 * np.arange(d // 2) / d)[None, :]
    assert np.abs(t[..., 0] - np.cos(ang)).max() <= 1e-6
    assert np.abs(t[..., 1] - np.sin(ang)).max() <= 1e-6


@pytest.mark.parametrize("d", [64, 128])
def test_rope_apply_matches_oracle(d):
    B, H, N = 2, 3, 777
    g = torch.Generator().manual_seed(d)
    x = (torch.randn((B, H, N, d), generator=g) * 2).to(torch.bfloat16)
    ref = oracle.rope(to_bits(x), BASE, pos0=1000)
    table = binding.rope_table(N + 1000, d, BASE)
    xg = x.cuda()
    binding.rope_apply(xg, table, pos0=1000)
    torch.cuda.synchronize()
    got = to_bits(xg)
    refv, gotv = oracle.bf16_bits_to_f64(ref), oracle.bf16_bits_to_f64(got)
    # fp32 rotation then one rounding vs fp64 rotation then one rounding: at
    # most one bf16 step apart, and almost always identical
    step = np.maximum(np.abs(refv), 2.0 ** -126) * 2.0 ** -7
    assert np.all(np.abs(gotv - refv) <= step)
    assert np.mean(got != ref) < 0.01


# (B, Hq, Hkv, N, d, n_sink, window, gamma)
CASES = [
    (1, 2, 1, 300, 128, 4, 64, 16),
    (2, 8, 2, 517, 128, 4, 100, 64),
    (1, 4, 2, 333, 64, 8, 7, 3),
    (1, 2, 1, 500, 128, 4, 64, 1),
    (1, 2, 2, 1, 128, 4, 16, 4),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "B%d_H%d-%d_N%d_d%d_s%d_w%d_g%d" % c)
def test_prefill_rope_matches_oracle(case):
    B, Hq, Hkv, N, d, s, w, gamma = case
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=sum(case) + 31)
    Qr = oracle.rope(to_bits(q), BASE)
    Kr = oracle.rope(to_bits(k), BASE)
    ref = oracle.delta_attn(Qr, Kr, to_bits(v), s, w, gamma)["A"]
    table = binding.rope_table(N, d, BASE)
    q0 = q.clone()
    out = binding.delta_attn_prefill_rope(q, k, v, s, w, gamma, table)
    assert binding.check() == binding.DA_OK
    assert torch.equal(q, q0)  # Q is rotated on the fly, not in memory
    assert_close(out, ref, "prefill with RoPE")
    kv = oracle.bf16_bits_to_f64(to_bits(k))
    assert np.abs(kv - oracle.bf16_bits_to_f64(Kr)).max() <= 2.0 ** -7 * np.abs(kv).max()  # K rotated in place


def test_decode_with_rotated_query():
    """Prefill-style rotated cache and a new token rotated to position N."""
    B, Hq, Hkv, N, d = 1, 8, 2, 1500, 128
    q, k, v = rand_qkv(B, Hq, Hkv, N + 1, d, seed=5)
    table = binding.rope_table(N + 1, d, BASE)
    binding.rope_apply(k, table)                       # cache keys at positions 0..N
    qn = q[:, :, N:N + 1].contiguous()
    binding.rope_apply(qn, table, pos0=N)              # the new query at position N
    out = binding.decode(qn[:, :, 0].contiguous(), k, v)
    assert binding.check() == binding.DA_OK
    ref, _ = oracle.decode(to_bits(qn[:, :, 0]), to_bits(k), to_bits(v), [N + 1])
    assert_close(out, ref, "decode with RoPE")
    qr = oracle.rope(to_bits(q[:, :, N:N + 1]), BASE, pos0=N)
    qv = oracle.bf16_bits_to_f64(to_bits(qn))
    assert np.abs(qv - oracle.bf16_bits_to_f64(qr)).max() <= 2.0 ** -7 * np.abs(qv).max()


def test_prefill_rope_131k_sampled_rows():
    """N = 131072, 32/8 heads, d = 128, gamma 64, window 2048, 4 sinks, with
    unrotated N(0,1) Q and K: sampled output rows (start, middle, end) of two
    heads on distinct KV heads against the oracle on rotated inputs."""
    B, Hq, Hkv, N, d, s, w, gamma = 1, 32, 8, 131072, 128, 4, 2048, 64
    q, k, v = rand_qkv(B, Hq, Hkv, N, d, seed=131)
    Kr = oracle.rope(to_bits(k), BASE)
    table = binding.rope_table(N, d, BASE)
    out = binding.delta_attn_prefill_rope(q, k, v, s, w, gamma, table)
    assert binding.check() == binding.DA_OK
    Qb = to_bits(q)
    rows = []
    for h in (2, 29):
        for i in (0, 1, 5, 63, 64, 65, 4097, 70000, N - 65, N - 64, N - 1):
            rows.append((0, h, i))
    # rotate only the query rows the oracle reads: each row and its sample row
    Qr = np.zeros_like(Qb)
    for (_, h, i) in rows:
        for r in (i, (i // gamma) * gamma):
            Qr[0, h, r] = oracle.rope(Qb[0:1, h:h + 1, r:r + 1], BASE, pos0=r)[0, 0, 0]
    ref = oracle.rows(Qr, Kr, to_bits(v), s, w, gamma, rows)["A"]
    got = torch.stack([out[0, h, i] for (_, h, i) in rows]).double().cpu().numpy()
    err = np.abs(got - ref)
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (err.max(), err.mean())
