"""Data-parallel GRPO update across torch.distributed ranks (host logic).

The batch of one step is sharded by prompt group: every rank owns whole
groups of G responses, so the group advantage of Eq. 2 stays local.  Eq. 1
averages over the whole step's batch, so the aggregation's normaliser is
global: the token count N_valid (token-mean) or the response count n_resp
(per-response mean), summed over ranks before the loss is formed.  With that
normaliser on every rank, the losses and LM-head gradients of the ranks add
up to those of the whole batch; the one data exchange is the sum of dW (and
of the scalar loss).  dH stays with the rank that owns the tokens.

`compute` is the per-rank loss call; by default the CUDA library's
grpo_loss_fwd_bwd_events, whose per-chunk events let each vocabulary chunk's
dW all-reduce start on a communication stream while the later chunks still
compute.  Collectives go through torch.distributed (NCCL on GPUs, gloo on
CPUs).
"""
from __future__ import annotations

from typing import Callable, Optional, Tuple

import torch


def shard_groups(n_groups: int, world: int, rank: int) -> Tuple[int, int]:
    """Contiguous range [start, stop) of prompt groups owned by `rank`; sizes
    differ by at most one, lower ranks take the remainder."""
    if world < 1 or not 0 <= rank < world or n_groups < 0:
        raise ValueError("bad world/rank/n_groups")
    base, extra = divmod(n_groups, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def shard_rows(n_groups: int, G: int, L: int, world: int, rank: int) -> Tuple[slice, slice]:
    """(response slice, padded-row slice) of `rank`'s groups in a batch laid out
    as n_groups * G responses of L padded rows each."""
    g0, g1 = shard_groups(n_groups, world, rank)
    return slice(g0 * G, g1 * G), slice(g0 * G * L, g1 * G * L)


def global_count(local: float, device: torch.device, group=None) -> float:
    """Sum of a per-rank count over the ranks of `group`."""
    import torch.distributed as dist
    t = torch.tensor([float(local)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    return float(t.item())


def default_compute(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, clip_eps, beta, agg_mode, norm,
                    ws=None, out=None):
    from . import binding
    return binding.loss_fwd_bwd(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, clip_eps, beta,
                                agg_mode, ws=ws, out=out, norm=norm)


def dp_loss_fwd_bwd(H, W, targets, mask, old_logp, ref_logp, adv, n_resp: int, L: int, clip_eps: float,
                    beta: float, agg_mode: int, local_count: float, group=None,
                    compute: Optional[Callable] = None, **kw):
    """One data-parallel GRPO loss forward + backward over this rank's shard.

    local_count: this rank's N_valid (agg_mode 0) or n_resp (agg_mode 1),
    known on the host from the response lengths.  Returns (loss, dH, dW) where
    loss and dW are summed over ranks (the whole batch's values) and dH is this
    rank's rows.
    """
    import torch.distributed as dist
    dev = W.device if isinstance(W, torch.Tensor) else torch.device("cpu")
    norm = global_count(local_count, dev if dev.type == "cuda" else torch.device("cpu"), group)
    if norm <= 0:
        norm = 1.0  # an all-padding step: every weight is 0 anyway
    if compute is None and dev.type == "cuda":
        return _overlapped(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, clip_eps, beta, agg_mode,
                           norm, group, **kw)
    compute = compute or default_compute
    loss, dH, dW = compute(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, clip_eps, beta, agg_mode,
                           norm, **kw)
    dist.all_reduce(dW, op=dist.ReduceOp.SUM, group=group)
    dist.all_reduce(loss, op=dist.ReduceOp.SUM, group=group)
    return loss, dH, dW


def chunk_rows(V: int, cols: int):
    """Row slices of dW, one per backward vocabulary chunk of `cols` rows."""
    if cols <= 0:
        return []
    return [slice(c0, min(V, c0 + cols)) for c0 in range(0, V, cols)]


def _overlapped(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, clip_eps, beta, agg_mode, norm, group,
                ws=None, out=None, comm_stream=None):
    """The library call with one event per vocabulary chunk; on a communication
    stream, each chunk's rows of dW are all-reduced as soon as its event fires,
    overlapping the backward of the later chunks.  The caller's current stream
    waits for every collective before this returns."""
    import torch.distributed as dist
    from . import binding
    dev = W.device
    rows = chunk_rows(W.shape[0], binding.vocab_chunk_cols(W.shape[0]))
    events = [torch.cuda.Event() for _ in rows]
    loss, dH, dW = binding.loss_fwd_bwd(H, W, targets, mask, old_logp, ref_logp, adv, n_resp, L, clip_eps, beta,
                                        agg_mode, ws=ws, out=out, norm=norm, chunk_events=events)
    comm = comm_stream or torch.cuda.Stream(dev)
    works = []
    with torch.cuda.stream(comm):
        for ev, r in zip(events, rows):
            comm.wait_event(ev)
            works.append(dist.all_reduce(dW[r], op=dist.ReduceOp.SUM, group=group, async_op=True))
        works.append(dist.all_reduce(loss, op=dist.ReduceOp.SUM, group=group, async_op=True))
    for wk in works:
        wk.wait()
    torch.cuda.current_stream(dev).wait_stream(comm)
    return loss, dH, dW
