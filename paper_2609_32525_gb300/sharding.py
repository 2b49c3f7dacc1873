"""Multi-rank host logic: point sharding of one coupling (App. G.4) and the
job-level timing of runs on several GPUs.  torch.distributed only: the local
compute is passed in (sharded_forward / sharded_backward take an object whose
methods run it; flashslice.ShardedCoupling runs it through the C ABI).

Point-sharded forward of one coupling over R ranks, rank r holding points
point_range(N, r, R) of every batch:
  1. fs_slice_fwd(..., finalize=0) on the local points: unnormalised U and S;
  2. allreduce_partials(U, S): the sums over all points (the one exchange step,
     B*H*G*(d+1) floats: 33 KB at H = 8, G = 32, d = 32);
  3. fs_slice_finalize, fs_mix, then fs_deslice_fwd on the local points.
The point-sharded backward, given each rank's dO of its points:
  4. fs_deslice_bwd on the local points: a partial d_tokens_mixed (its points'
     share of the sum over n), the local dx_mid and partial dW, dbias, dtau;
  5. allreduce_sums(d_tokens_mixed): the second exchange, B*H*G*d floats;
  6. fs_mix_bwd (the same on every rank: its inputs are now global, so dM is the
     whole gradient and is not exchanged), then fs_slice_bwd on the local
     points with the global tokens and weight sums: dfx, and dx_mid, dW, dbias,
     dtau added;
  7. allreduce_sums(dW, dbias, dtau): the parameter gradients of all points.
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def point_range(N: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous, balanced point range [n0, n1) of `rank` among `world` ranks."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("rank must lie in [0, world)")
    return N * rank // world, N * (rank + 1) // world


def _distributed() -> bool:
    return dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1


def allreduce_partials(U: torch.Tensor, S: torch.Tensor, group=None) -> None:
    """Sum the unnormalised numerators U [B,H,G,d] and weight sums S [B,H,G] of
    all ranks in place (before fs_slice_finalize).  A single process sums nothing."""
    if not _distributed():
        return
    dist.all_reduce(U, op=dist.ReduceOp.SUM, group=group)
    dist.all_reduce(S, op=dist.ReduceOp.SUM, group=group)


def allreduce_sums(*tensors: torch.Tensor, group=None) -> None:
    """Sum each tensor over all ranks in place: the backward's partial
    d_tokens_mixed, and the parameter gradients dW, dbias, dtau at the end.  A single
    process sums nothing."""
    if not _distributed():
        return
    for t in tensors:
        dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)


def sharded_forward(ops, group=None):
    """The point-sharded forward of one coupling on this rank's points (steps 1-3
    above).  `ops` runs the local compute: ops.slice_partials() -> (U, S), the
    unnormalised numerators and weight sums of the local points; ops.finalize(U, S)
    -> tokens; ops.mix(tokens) -> tokens_mixed; ops.deslice(tokens_mixed) -> out of
    the local points.  The one exchange happens here, between the first two."""
    U, S = ops.slice_partials()
    allreduce_partials(U, S, group)
    tokens = ops.finalize(U, S)
    return ops.deslice(ops.mix(tokens))


def sharded_backward(ops, group=None):
    """The point-sharded backward after sharded_forward (steps 4-7 above).
    ops.deslice_bwd() -> the local points' share of d_tokens_mixed;
    ops.mix_bwd(d_tokens_mixed) -> (d_tokens, dM), the whole gradient on every rank;
    ops.slice_bwd(d_tokens) -> (dW, dbias, dtau), the local points' parameter
    gradients of both backward calls.  Returns dM and the summed (dW, dbias, dtau)."""
    dzp = ops.deslice_bwd()
    allreduce_sums(dzp, group=group)
    dz, dM = ops.mix_bwd(dzp)
    grads = ops.slice_bwd(dz)
    allreduce_sums(*grads, group=group)
    return dM, grads


def job_time_ms(local_ms: float, device=None) -> float:
    """Job time of a timed region: the maximum over ranks of their local times
    (every rank must call it; a single process returns its own time)."""
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(local_ms)
    t = torch.tensor([float(local_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(points_per_rank: int, world: int, ms: float) -> float:
    """Whole-job throughput in Mpoints/s: every rank's points over the job time."""
    return world * points_per_rank / (ms * 1e-3) / 1e6
