"""Host side of multi-GPU runs: one process per GPU, launched by torchrun.

The E-step + M-step shards by prefix: every quantity of the method (beta and
zeta over the K proposals, N_b, the loss and the gradient rows) is local to
one prefix, so each rank takes prefixes of its own and no collective touches
the data path.  The only collectives are the barriers around the timed
region and the maximum of the ranks' times, which is the job's time.  These
helpers are the same for the NCCL runs on GPUs and the gloo runs on CPU that
test them.
"""
import os

import torch


def env():
    """(rank, world size, local rank) from the launcher's environment."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def init(world, backend):
    """Join the process group (rendezvous from MASTER_ADDR / MASTER_PORT)."""
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        dist.init_process_group(backend)


def rank_seed(base, rank):
    """Seed of the prefixes rank `rank` draws: every rank has its own batch
    (weak scaling), so seeds must differ between ranks."""
    return int(base) + 1000 * int(rank)


def barrier(world, device=None):
    """All ranks meet; on a GPU the device is drained too."""
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    if device is not None and torch.device(device).type == "cuda":
        torch.cuda.synchronize(device)


def max_over_ranks(x, world, device="cpu"):
    """The largest of the ranks' values of x (a time): the job ends when its
    slowest rank does."""
    if world <= 1:
        return float(x)
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank, world, ms):
    """Whole-job throughput: the units every rank processed over the job's time."""
    return units_per_rank * world / (ms / 1e3)
