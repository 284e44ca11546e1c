"""Multi-GPU layout of the boundary: which token rows a rank owns, and the one
exchange of the subspace update.

The boundary calls work on independent token rows, so N GPUs split a batch of
T tokens into N contiguous row ranges (U, T_fixed and P replicated on every
rank) and need no collective on the data path; the projection likewise splits
by weight columns.  The Grassmann update (Sec. 4.5) is the one place where
data-parallel replicas must agree: each replica accumulates its own
M_r = sum over its tokens of G^T (G U), and the step needs the sum over
replicas, M = sum_r M_r, which `allreduce_grassmann` forms in place before every
replica takes the same step.
"""


def token_shard(T, world, rank):
    """[start, stop) of the token rows owned by `rank` out of `world`: contiguous,
    sizes differing by at most one, together covering 0..T-1 exactly once."""
    if world < 1 or not 0 <= rank < world or T < 0:
        raise ValueError("bad shard request")
    base, extra = divmod(T, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def allreduce_grassmann(M, group=None):
    """Sum the replicas' Grassmann accumulations M [d, k] in place (every rank
    ends with the same M); a no-op outside torch.distributed."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(M, op=dist.ReduceOp.SUM, group=group)
    return M
