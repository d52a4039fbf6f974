"""Data-parallel replicas of the Delta Attention prefill across GPUs.

The prefill partitions into independent problems (sequences; (batch, KV head)
groups with their query heads) with no exchange, so N GPUs run N independent
problems: one process per GPU (launched by torchrun), each with its own seeded
sequence, and no collective on the data path.  Timing uses a barrier on both
sides of the timed loop and the maximum of the per-rank times; whole-job
throughput is the total work of all ranks over that time (weak scaling).

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
