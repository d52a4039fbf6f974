"""Shared helpers of the GPU tests: oracle calls on the same bf16 tensors the
kernels read, and the tolerance of the comparison.

Tolerance (bf16 inputs, fp32 accumulation, bf16 output): max-abs <= 2e-2 and
mean-abs <= 2e-3 against the fp64 oracle, element by element.
"""
import numpy as np
import torch

import oracle
from paper_2505_11254_gb300.inputs import to_bits

MAX_ABS = 2e-2
MEAN_ABS = 2e-3


def rand_qkv(B, Hq, Hkv, N, d, seed=0, scale=1.0, device="cuda"):
    g = torch.Generator(device="cpu").manual_seed(seed)
    q = (torch.randn((B, Hq, N, d), generator=g) * scale).to(torch.bfloat16)
    k = (torch.randn((B, Hkv, N, d), generator=g) * scale).to(torch.bfloat16)
    v = torch.randn((B, Hkv, N, d), generator=g).to(torch.bfloat16)
    return q.to(device), k.to(device), v.to(device)


def oracle_full(q, k, v, n_sink, window, gamma, **kw):
    return oracle.delta_attn(to_bits(q), to_bits(k), to_bits(v), n_sink, window, gamma, **kw)


def oracle_rows(q, k, v, n_sink, window, gamma, bhi):
    return oracle.rows(to_bits(q), to_bits(k), to_bits(v), n_sink, window, gamma, bhi)


def assert_close(got, ref, what, max_abs=MAX_ABS, mean_abs=MEAN_ABS):
    got = got.detach().float().cpu().numpy().astype(np.float64) if isinstance(got, torch.Tensor) else got
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    assert np.all(np.isfinite(got)), "%s: non-finite values" % what
    err = np.abs(got - ref)
    mx, mn = float(err.max()) if err.size else 0.0, float(err.mean()) if err.size else 0.0
    assert mx <= max_abs and mn <= mean_abs, "%s: max-abs %.3g mean-abs %.3g" % (what, mx, mn)
    return mx, mn


GUARD = 4096   # guard bytes on each side
PATTERN = 0xA5


class Guarded:
    """A tensor of the given shape and dtype inside a buffer with guard bytes
    on both sides, 256-byte aligned like a fresh allocation."""

    def __init__(self, shape, dtype, device="cuda"):
        self.nbytes = int(torch.tensor([], dtype=dtype).element_size() * torch.Size(shape).numel())
        self.buf = torch.full((2 * GUARD + self.nbytes + 256,), PATTERN, dtype=torch.uint8, device=device)
        self.t = self.buf[GUARD:GUARD + self.nbytes].view(dtype).view(shape)

    def intact(self):
        if self.buf.is_cuda:
            torch.cuda.synchronize()
        head = self.buf[:GUARD]
        tail = self.buf[GUARD + self.nbytes:]
        return bool((head == PATTERN).all()) and bool((tail == PATTERN).all())


def guarded_ws(nbytes, device="cuda"):
    return Guarded((max(int(nbytes), 16),), torch.uint8, device)
