"""Replica bookkeeping for running the benchmark on N GPUs (one process per
GPU under torchrun).  Images are independent, so every rank infers its own
batches and no data-path collective exists: ranks take disjoint slices of
the seeded input set, each timing is the maximum over ranks, and the
whole-job throughput counts the images of every rank."""


def input_slices(rank: int, batch: int, per_rank: int = 2) -> list:
    """First image index of each of rank `rank`'s `per_rank` batches."""
    return [(per_rank * rank + j) * batch for j in range(per_rank)]


def reduce_max(value: float, dist=None, device: str = "cpu") -> float:
    """Maximum of `value` over the ranks of the default process group
    (`dist` is torch.distributed, or None for one process).  `device` is
    where the reduction runs: "cuda" for NCCL, "cpu" for gloo."""
    if dist is None:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, batch: int, steps: int, seconds: float) -> float:
    """Images per second of the whole job: `world` ranks, `steps` batches of
    `batch` images each, in `seconds` (the maximum over ranks)."""
    return world * batch * steps / seconds
