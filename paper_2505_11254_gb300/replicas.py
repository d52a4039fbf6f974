"""Data-parallel replicas and head shards of the Delta Attention prefill
across GPUs.

The prefill partitions into independent problems (sequences; (batch, KV head)
groups with their query heads) with no exchange.  Two ways to use N GPUs, one
process per GPU (launched by torchrun), no collective on the data path:
  * replicas: N independent seeded sequences, one per rank (weak scaling);
  * head shards: one prefill whose (batch, KV head) pairs are split over the
    ranks (strong scaling), optionally followed by an all-gather of O;
  * context shards: one prefill split by rows, after an all-gather of the K
    and V row shards (strong scaling).
Timing uses a barrier on both sides of the timed loop and the maximum of the
per-rank times; whole-job throughput is the work of all ranks over that time.

Works with NCCL on GPUs and with gloo on CPU (used by the host-side tests).
"""
import os

import torch


class Replicas:
    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.backend = None

    def init(self, backend=None):
        """Join the process group (when WORLD_SIZE > 1) and select this rank's GPU."""
        if self.world > 1:
            import torch.distributed as dist
            self.backend = backend or ("nccl" if torch.cuda.is_available() else "gloo")
            if self.backend == "nccl":
                torch.cuda.set_device(self.local)
            if not dist.is_initialized():
                dist.init_process_group(backend=self.backend)
        elif torch.cuda.is_available():
            torch.cuda.set_device(self.local)
        return self

    def _device(self):
        return torch.device("cuda", self.local) if self.backend == "nccl" else torch.device("cpu")

    def barrier(self):
        if self.world > 1:
            import torch.distributed as dist
            dist.barrier()

    def max(self, x: float) -> float:
        """Maximum of a per-rank value over all ranks."""
        if self.world == 1:
            return x
        import torch.distributed as dist
        t = torch.tensor([x], dtype=torch.float64, device=self._device())
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    def seed(self, base: int) -> int:
        """Seed of this rank's independent problem."""
        return base + self.rank

    def throughput(self, units_per_rank: float, max_seconds: float) -> float:
        """Whole-job throughput: the units all ranks processed over the slowest rank's time."""
        return self.world * units_per_rank / max_seconds

    def close(self):
        if self.world > 1:
            import torch.distributed as dist
            if dist.is_initialized():
                dist.destroy_process_group()


# ---------------------------------------------------------------- head shards
# One prefill split over ranks.  The (batch, KV head) pairs of Alg. 1 are
# independent problems (each query head reads only its own KV head), so rank r
# takes a contiguous range of the B * Hkv pairs with the G query heads of each
# pair and runs the unchanged single-GPU path on it, with no exchange on the
# data path.  In the [B * Hkv, G, N, d] view of Q and O (and [B * Hkv, 1, N, d]
# of K and V) a contiguous pair range is one contiguous slice, which the
# library takes as a problem of (p1 - p0) sequences with G query heads and one
# KV head.

def head_shard(B: int, Hkv: int, rank: int, world: int):
    """Pair range [p0, p1) of rank `rank`: the B * Hkv pairs split into
    `world` contiguous ranges whose sizes differ by at most one."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("rank %d outside a world of %d" % (rank, world))
    pairs = B * Hkv
    return rank * pairs // world, (rank + 1) * pairs // world


def shard_views(Q, K, V, Hkv: int, p0: int, p1: int):
    """Views of Q [B, Hq, N, d] and K, V [B, Hkv, N, d] holding the pairs
    [p0, p1): Q as [p1 - p0, G, N, d], K and V as [p1 - p0, 1, N, d]."""
    B, Hq, N, d = Q.shape
    G = Hq // Hkv
    q = Q.reshape(B * Hkv, G, N, d)[p0:p1]
    k = K.reshape(B * Hkv, 1, N, d)[p0:p1]
    v = V.reshape(B * Hkv, 1, N, d)[p0:p1]
    return q, k, v


def gather_shards(O_part, B: int, Hq: int, Hkv: int, world: int):
    """All-gather of the per-rank outputs O_part [p1 - p0, G, N, d] into the
    whole [B, Hq, N, d] output (every rank receives it).  Shards are padded to
    the largest range so that the collective moves equal-sized buffers."""
    import torch.distributed as dist
    G, N, d = O_part.shape[1:]
    ranges = [head_shard(B, Hkv, r, world) for r in range(world)]
    width = max(p1 - p0 for p0, p1 in ranges)
    pad = O_part.new_zeros((width, G, N, d))
    pad[: O_part.shape[0]].copy_(O_part)
    bufs = [torch.empty_like(pad) for _ in range(world)]
    dist.all_gather(bufs, pad)
    out = O_part.new_empty((B * Hkv, G, N, d))
    for (p0, p1), buf in zip(ranges, bufs):
        out[p0:p1].copy_(buf[: p1 - p0])
    return out.reshape(B, Hq, N, d)


# ------------------------------------------------------------ context shards
# One sequence split by rows (context parallelism).  Rank r computes the rows
# [r0, r1) of every (b, head) with delta_attn_prefill_rows from its rows of Q
# and the keys and values of rows 0 .. r1 - 1: the sink keys, the window before
# r0 and, for its sampled rows' dense attention, every earlier key.  The one
# exchange is an all-gather of the K and V row shards; a range starts on a
# 128-row tile and a sample group, so its correction needs no other rank's Q.

def context_shard(N: int, gamma: int, rank: int, world: int):
    """Row range [r0, r1) of rank `rank`: the sequence cut at multiples of
    lcm(128, gamma) into `world` ranges whose unit counts differ by at most
    one (a rank may get none when the sequence has fewer units than ranks)."""
    import math
    if world < 1 or not 0 <= rank < world:
        raise ValueError("rank %d outside a world of %d" % (rank, world))
    unit = math.lcm(128, gamma)
    n_units = -(-N // unit)
    u0, u1 = rank * n_units // world, (rank + 1) * n_units // world
    return min(u0 * unit, N), min(u1 * unit, N)


def _gather_rows(part, N: int, gamma: int, world: int):
    """All-gather of per-rank row ranges [.., r1 - r0, ..] (dim 2) into the
    whole [.., N, ..] tensor on every rank (padded to the longest range)."""
    import torch.distributed as dist
    ranges = [context_shard(N, gamma, r, world) for r in range(world)]
    width = max(r1 - r0 for r0, r1 in ranges)
    shape = list(part.shape)
    shape[2] = width
    pad = part.new_zeros(shape)
    pad[:, :, : part.shape[2]].copy_(part)
    bufs = [torch.empty_like(pad) for _ in range(world)]
    dist.all_gather(bufs, pad)
    shape[2] = N
    out = part.new_empty(shape)
    for (r0, r1), buf in zip(ranges, bufs):
        out[:, :, r0:r1].copy_(buf[:, :, : r1 - r0])
    return out


def gather_kv(K_part, V_part, N: int, gamma: int, world: int):
    """The context-parallel exchange: every rank's rows of K and V gathered
    into the whole [B, Hkv, N, d] K and V on every rank."""
    return _gather_rows(K_part, N, gamma, world), _gather_rows(V_part, N, gamma, world)


def gather_context(O_part, N: int, gamma: int, world: int):
    """All-gather of the per-rank output rows into the whole [B, Hq, N, d] O."""
    return _gather_rows(O_part, N, gamma, world)
