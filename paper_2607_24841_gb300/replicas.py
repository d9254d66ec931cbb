"""Host-side logic of running the block-denoise path as N independent replicas.

Generating a block is independent per sequence, so N GPUs run N independent block
streams with no data-path collective (weak scaling).  One process per GPU; the only
communication is host-side bookkeeping over torch.distributed: a rendezvous, barriers
around the timed region, and the maximum step time over ranks, from which the
whole-job throughput is computed.  Rank 0 alone reports.
"""
import os


def world_info():
    """(world, rank, local_rank) from the launcher's environment (1, 0, 0 without one)."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def init(world, backend=None):
    """Join the process group when world > 1 (NCCL on GPUs, gloo on CPU)."""
    if world <= 1:
        return
    import torch
    import torch.distributed as dist
    if not dist.is_initialized():
        dist.init_process_group(backend or ("nccl" if torch.cuda.is_available() else "gloo"))


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, x, device=None):
    """The largest x over all ranks (the slowest replica sets the job's time)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_replica, world, ms):
    """Whole-job units per second: every replica processed units_per_replica in ms."""
    return units_per_replica * world / (ms / 1e3)


def finish(world):
    if world > 1:
        import torch.distributed as dist
        if dist.is_initialized():
            dist.destroy_process_group()
