"""Host-side logic of the multi-GPU path.  Units (window, head) are independent
(the method attends within a window), so several GPUs split them with no
data-path collective: each rank runs the library on its own contiguous range of
windows; only the timing is reduced across ranks."""
import torch


def window_range(n_windows: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous [start, stop) range of windows for `rank`; the first
    n_windows % world ranks take one extra window."""
    if world < 1 or not 0 <= rank < world or n_windows < 0:
        raise ValueError("need 0 <= rank < world and n_windows >= 0")
    base, extra = divmod(n_windows, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def max_over_ranks(x: float, device=None) -> float:
    """Largest `x` over the ranks of the default process group (x itself
    without one).  The device is the backend's: CUDA for nccl, CPU for gloo."""
    if not (torch.distributed.is_available() and torch.distributed.is_initialized()):
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def aggregate_rate(items_per_rank: float, steps: int, max_ms: float, world: int) -> float:
    """Whole-job throughput: every rank's items over the slowest rank's time."""
    return world * items_per_rank * steps / (max_ms * 1e-3)
