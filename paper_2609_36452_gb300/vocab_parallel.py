"""Vocabulary-parallel commit step over the ranks of a torch.distributed group.

Each rank holds a contiguous slice of the LM head's rows (a context created with the slice's
size and told its offset with ``set_vocab_shard``).  One step is the library's
``rpd_step_shard_partials`` on every rank, one all-gather of the per-row softmax statistics
(16 bytes per projected row and rank), and ``rpd_step_shard_finish`` on every rank, which
merges the slices' statistics and commits; every rank ends with the same commits.  This
module only arranges the exchange: the statistics, the merge and the commit are computed by
the library's kernels.
"""
from __future__ import annotations


def shard_bounds(V: int, world: int, rank: int, align: int = 256):
    """Rows [v0, v1) of a V-row head held by `rank` of `world`: contiguous slices in rank order,
    each boundary a multiple of `align` (the head kernel's vocabulary tile) except the end."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("rank must be in [0, world)")
    tiles = (V + align - 1) // align
    t0, t1 = tiles * rank // world, tiles * (rank + 1) // world
    return min(V, t0 * align), min(V, t1 * align)


def sharded_step(ctx, hidden, mask, tau, budget, out_commit, out_token, out_stats, group=None,
                 partials=None, gathered=None):
    """One commit step with the head split over the group's ranks (rank r holds slice r).

    hidden [K][N][d], mask [N] (in/out), out_* as in ``Rpd.step``.  ``partials`` [K][N][4] and
    ``gathered`` [world][K][N][4] float32 buffers may be passed in to avoid allocations.
    Every rank must call it with the same mask."""
    import torch
    import torch.distributed as dist

    world = dist.get_world_size(group)
    K, N = ctx.K, mask.numel()
    dev = mask.device
    if partials is None:
        partials = torch.empty(K, N, 4, dtype=torch.float32, device=dev)
    if gathered is None:
        gathered = torch.empty(world, K, N, 4, dtype=torch.float32, device=dev)
    ctx.step_shard_partials(hidden, mask, partials)
    # rank-major concatenation: the same memory as gathered[rank][K][N][4]
    dist.all_gather_into_tensor(gathered.view(world * K, N, 4), partials, group=group)
    ctx.step_shard_finish(gathered, mask, tau, budget, out_commit, out_token, out_stats)
    return gathered
