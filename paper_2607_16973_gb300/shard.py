"""Search over a corpus split by rows across devices, one process per GPU.

Each rank holds one contiguous, block-aligned row range of the corpus (codes,
scales and, when filtering, tenant ids); the rotation, the codebook and the
queries are replicated.  A sharded search is: every rank runs tq_search on its
own rows, the ranks exchange their k best per query (an all-gather of
nq * k * 12 bytes per rank), and tq_merge_topk keeps the k best of the union.
That is exact: each global top-k member is in the top-k of the shard that holds
it, and (score desc, id asc) is a total order on distinct rows.  Encoding
shards the same way and needs no exchange.
"""
from __future__ import annotations


def shard_rows(n: int, world: int, rank: int, align: int = 64) -> tuple[int, int]:
    """Row range [lo, hi) of `rank` among `world` shards of n rows: contiguous,
    starting on a multiple of `align` (the filter block size, so no tenant
    block straddles two shards), sizes differing by at most `align` rows."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside [0, {world})")
    if n < 0 or align < 1:
        raise ValueError("n must be >= 0 and align >= 1")
    blocks = (n + align - 1) // align
    b0 = blocks * rank // world
    b1 = blocks * (rank + 1) // world
    return min(n, b0 * align), min(n, b1 * align)


def to_global(ids, offset: int):
    """Local shard ids -> corpus ids (padding -1 stays -1), in place."""
    if offset:
        ids.add_((ids >= 0).to(ids.dtype) * offset)
    return ids


def gather_topk(ids, scores, offset: int, group=None):
    """The exchange step: every rank contributes its [nq, k] result (local ids,
    shifted here by its shard offset); returns [world, nq, k] ids and scores of
    all ranks, in rank order, on every rank.  Works on CPU tensors (gloo) and
    CUDA tensors (NCCL)."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    g_ids = to_global(ids.clone(), offset)
    nq, k = ids.shape
    # rank-major concatenation along the first dimension, viewed as [world, nq, k]
    out_i = torch.empty((world * nq, k), dtype=ids.dtype, device=ids.device)
    out_s = torch.empty((world * nq, k), dtype=scores.dtype, device=scores.device)
    dist.all_gather_into_tensor(out_i, g_ids.contiguous(), group=group)
    dist.all_gather_into_tensor(out_s, scores.contiguous(), group=group)
    return out_i.view(world, nq, k), out_s.view(world, nq, k)


def sharded_search(Q, R, centroids, bits: int, codes, scale, k: int, offset: int, group=None, **search_kw):
    """tq_search over this rank's rows, the all-gather of every rank's top-k,
    and tq_merge_topk: (ids [nq, k] global, scores [nq, k]) on every rank.

    An id map is refused: its search reports external ids, which the merge
    would take for local rows (shifting them by the offset and breaking ties
    by them), and each rank knows only its own rows' external ids."""
    import torch
    from . import merge_topk, search
    if search_kw.get("idmap") is not None:
        raise ValueError("sharded_search takes no id map: results are global rows")
    if codes.shape[0] == 0:  # an empty shard contributes only empty slots
        ids = torch.full((Q.shape[0], k), -1, dtype=torch.int64, device=Q.device)
        scores = torch.full((Q.shape[0], k), float("-inf"), dtype=torch.float32, device=Q.device)
    else:
        ids, scores = search(Q, R, centroids, bits, codes, scale, k, **search_kw)
    cand_i, cand_s = gather_topk(ids, scores, offset, group)
    return merge_topk(cand_i, cand_s, k, stream=search_kw.get("stream"))
