"""Independent replicas across ranks (one process per GPU).

The sweep has no data-path exchange: every rank runs its own copy of the
workload on its own GPU.  The only collectives are a barrier around the timed
region and the maximum of the per-rank times, so the job rate is the units
all ranks processed divided by the slowest rank's time (weak scaling).
"""
from __future__ import annotations

import os
from typing import Optional, Tuple


def env() -> Tuple[int, int, int]:
    """(world size, rank, local rank) from the launcher's environment."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


class Replicas:
    def __init__(self, backend: Optional[str] = None, device=None):
        import torch
        self.world, self.rank, self.local = env()
        self.dist = None
        self.device = device
        if self.world > 1:
            import torch.distributed as dist
            if backend is None:
                backend = "nccl" if torch.cuda.is_available() else "gloo"
            kw = {}
            if backend == "nccl" and device is not None:
                kw["device_id"] = device
            dist.init_process_group(backend, **kw)
            self.dist = dist
            self.backend = backend

    def barrier(self):
        if self.dist is not None:
            self.dist.barrier()

    def max(self, value: float) -> float:
        """Maximum of a per-rank value over all ranks."""
        if self.dist is None:
            return float(value)
        import torch
        dev = self.device if self.backend == "nccl" else "cpu"
        t = torch.tensor([float(value)], dtype=torch.float64, device=dev)
        self.dist.all_reduce(t, op=self.dist.ReduceOp.MAX)
        return float(t.item())

    def job_rate(self, units_per_rank: float, seconds_this_rank: float) -> Tuple[float, float]:
        """(whole-job units per second, slowest rank's seconds)."""
        t = self.max(seconds_this_rank)
        return self.world * units_per_rank / t, t

    def close(self):
        if self.dist is not None:
            self.dist.destroy_process_group()
            self.dist = None
