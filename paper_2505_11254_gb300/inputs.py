"""Seeded synthetic inputs for the Delta Attention prefill.

This module is the one piece shared by the CUDA path's tests/bench and the
CPU oracle: it only draws random tensors and holds none of the method's
arithmetic.  The workloads mirror the paper's single-layer long-context
prefills (Llama-3.1-8B-shaped attention: 32 query heads, 8 KV heads, d=128,
StreamingLLM with 4 sinks and a 2K window, gamma = 64; Sec. 4 and the latency
ablation) with synthetic N(0,1) activations standing in for real prompts.

Recipe (per sequence b, with its own generator when ``per_sequence_seeds``):
  Q, K, V are drawn in that order, head by head, as fp32 N(0,1) [N, d] slabs;
  RoPE (rotate-half pairs c, c+d/2; theta_c = base^(-2c/d); position = row
  index; angles in fp64) is applied to Q and K when ``rope``; key rows
  0..n_scaled_sinks-1 of every KV head are multiplied by ``sink_scale``;
  everything is rounded to bf16 (round-to-nearest-even, torch's cast).
"""
from dataclasses import dataclass, replace
from typing import Optional

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    Hq: int
    Hkv: int
    d: int
    N: int
    n_sink: int
    window: int
    gamma: int
    rope: bool = True
    rope_base: float = 500000.0
    sink_scale: float = 1.0
    n_scaled_sinks: int = 4
    seed: int = 0
    per_sequence_seeds: bool = False

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)

    def as_dict(self) -> dict:
        return dict(self.__dict__)


# The five seeded workloads.  Names say what they are.
TINY_N2048 = Workload("tiny_b1_h4_d64_n2048_w256_g16", 1, 4, 4, 64, 2048, 4, 256, 16, rope=False)
LLAMA8B_N32K = Workload("llama8b_b1_n32768_w2048_g64", 1, 32, 8, 128, 32768, 4, 2048, 64)
LLAMA8B_N131K = Workload("llama8b_b1_n131072_w2048_g64_sinks8x", 1, 32, 8, 128, 131072, 4, 2048, 64,
                         sink_scale=8.0)
LLAMA8B_N1M = Workload("llama8b_b1_n1048576_w2048_g64", 1, 32, 8, 128, 1048576, 4, 2048, 64)
SWEEP_B4_N64K = Workload("llama8b_b4_n65536_sweep", 4, 32, 8, 128, 65536, 4, 2048, 64,
                         per_sequence_seeds=True)

WORKLOADS = {w.name: w for w in (TINY_N2048, LLAMA8B_N32K, LLAMA8B_N131K, LLAMA8B_N1M, SWEEP_B4_N64K)}
SWEEP_WINDOWS = (512, 2048, 8192)
SWEEP_GAMMAS = (16, 32, 64, 128)


def _rope(x: torch.Tensor, cos: torch.Tensor, sin: torch.Tensor) -> torch.Tensor:
    h = x.shape[-1] // 2
    x1, x2 = x[:, :h], x[:, h:]
    return torch.cat([x1 * cos - x2 * sin, x2 * cos + x1 * sin], dim=-1)


def _rope_tables(N: int, d: int, base: float, device):
    inv = base ** (-(torch.arange(0, d // 2, dtype=torch.float64, device=device) * 2.0 / d))
    ang = torch.arange(N, dtype=torch.float64, device=device)[:, None] * inv[None, :]
    return ang.cos().float(), ang.sin().float()


def generate(w: Workload, device="cpu", N: Optional[int] = None):
    """Return (Q, K, V) bf16 tensors on `device`: Q [B,Hq,N,d], K/V [B,Hkv,N,d]."""
    N = w.N if N is None else N
    dev = torch.device(device)
    Q = torch.empty((w.B, w.Hq, N, w.d), dtype=torch.bfloat16, device=dev)
    K = torch.empty((w.B, w.Hkv, N, w.d), dtype=torch.bfloat16, device=dev)
    V = torch.empty((w.B, w.Hkv, N, w.d), dtype=torch.bfloat16, device=dev)
    cos = sin = None
    if w.rope:
        cos, sin = _rope_tables(N, w.d, w.rope_base, dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(w.seed)
    for b in range(w.B):
        if w.per_sequence_seeds:
            gen = torch.Generator(device=dev)
            gen.manual_seed(w.seed + b)
        for name, T in (("Q", Q), ("K", K), ("V", V)):
            for h in range(T.shape[1]):
                x = torch.randn((N, w.d), generator=gen, device=dev, dtype=torch.float32)
                if w.rope and name != "V":
                    x = _rope(x, cos, sin)
                if name == "K" and w.sink_scale != 1.0:
                    x[: w.n_scaled_sinks] *= w.sink_scale
                T[b, h].copy_(x.to(torch.bfloat16))
                del x
    return Q, K, V


def checksum(t: torch.Tensor, chunk: int = 1 << 26) -> int:
    """Sum of the bf16 bit patterns as signed 16-bit integers (record keeping),
    taken over slices of `chunk` elements so that no full-size wider copy is
    made; the same bits give the same value on any device."""
    flat = t.contiguous().view(-1).view(torch.int16)
    total = 0
    for i in range(0, flat.numel(), chunk):
        total += int(flat[i:i + chunk].to(torch.int64).sum().item())
    return total


def checksums(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor) -> dict:
    return {"kind": "sum of bf16 bit patterns as int16", "Q": checksum(q), "K": checksum(k), "V": checksum(v)}


def to_bits(t: torch.Tensor):
    """bf16 tensor -> numpy uint16 array of its bit patterns (host copy)."""
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view("uint16")
