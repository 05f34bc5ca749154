"""Step (1) over a vocabulary split across ranks: the logits of a tensor-parallel LM head,
each rank holding the columns of one contiguous vocabulary slice.

Each rank summarises its slice of every slot row in one partial record (running maximum,
sum of exponentials below it, the slice's top-K values and vocabulary ids), the records
are all-gathered once (rows x (8 + 8K) bytes per rank), and the merge kernel combines them
into exactly the whole-row result: the log-sum-exp is associative over (max, sum) pairs and
every global top-K element is among its slice's top-K. The record layout is the C ABI's
(``lilicorr_topk_lse_partial``): float m, float s, float val[K], int32 id[K].

Host logic only (slice bounds, record packing, the gather); the records themselves are
written and merged by the CUDA kernels through ``topk_lse_partial`` / ``topk_lse_merge``.
"""
from __future__ import annotations

from typing import List, Optional, Tuple

import numpy as np
import torch
import torch.distributed as dist


def bounds(V: int, P: int) -> List[Tuple[int, int]]:
    """Contiguous vocabulary slices [a, b) of P ranks; the first V % P get one id more."""
    if P < 1 or V < P:
        raise ValueError("need 1 <= P <= V")
    q, r = divmod(V, P)
    out, a = [], 0
    for p in range(P):
        b = a + q + (1 if p < r else 0)
        out.append((a, b))
        a = b
    return out


def pack_records(m: np.ndarray, s: np.ndarray, vals: np.ndarray, ids: np.ndarray) -> torch.Tensor:
    """Host records [rows, 8 + 8K] uint8 from m, s [rows] fp32, vals [rows, K] fp32 and
    ids [rows, K] int32 (the layout the kernels write)."""
    rows, K = vals.shape
    rec = np.empty((rows, 8 + 8 * K), dtype=np.uint8)
    rec[:, 0:4] = np.ascontiguousarray(m, dtype=np.float32).reshape(rows, 1).view(np.uint8)
    rec[:, 4:8] = np.ascontiguousarray(s, dtype=np.float32).reshape(rows, 1).view(np.uint8)
    rec[:, 8:8 + 4 * K] = np.ascontiguousarray(vals, dtype=np.float32).view(np.uint8)
    rec[:, 8 + 4 * K:] = np.ascontiguousarray(ids, dtype=np.int32).view(np.uint8)
    return torch.from_numpy(rec)


def unpack_records(rec: torch.Tensor, K: int):
    """(m, s, vals, ids) numpy arrays of records [rows, 8 + 8K] (any device)."""
    a = rec.detach().cpu().contiguous().numpy()
    if a.ndim != 2 or a.shape[1] != 8 + 8 * K:
        raise ValueError("records must be [rows, 8 + 8K] bytes")
    m = a[:, 0:4].copy().view(np.float32).reshape(-1)
    s = a[:, 4:8].copy().view(np.float32).reshape(-1)
    vals = a[:, 8:8 + 4 * K].copy().view(np.float32)
    ids = a[:, 8 + 4 * K:].copy().view(np.int32)
    return m, s, vals, ids


def gather_records(rec: torch.Tensor, group: Optional[dist.ProcessGroup] = None) -> torch.Tensor:
    """All-gather every rank's records [rows, bytes] into [world, rows, bytes], rank order.
    The one collective of the sharded pass."""
    world = dist.get_world_size(group)
    out = [torch.empty_like(rec) for _ in range(world)]
    dist.all_gather(out, rec.contiguous(), group=group)
    return torch.stack(out)


def topk_lse_sharded(logits_shard: torch.Tensor, K: int, V: int,
                     group: Optional[dist.ProcessGroup] = None):
    """Whole-row (ids, logp, lse) of logits sharded by vocabulary over the ranks of
    ``group``: this rank holds columns bounds(V, world)[rank] of every row. Every rank
    returns the same result."""
    from . import topk_lse_merge, topk_lse_partial
    world, rank = dist.get_world_size(group), dist.get_rank(group)
    a, b = bounds(V, world)[rank]
    if logits_shard.shape[-1] != b - a:
        raise ValueError(f"rank {rank} must hold {b - a} vocabulary columns")
    rec = topk_lse_partial(logits_shard.reshape(-1, b - a), K, a)
    return topk_lse_merge(gather_records(rec, group), K)
