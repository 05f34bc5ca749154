"""Shared test helpers: device uploads and the tie-aware path comparison.

A greedy step whose runner-up score (by the oracle) lies within the float
tolerance of the best counts as a tie: when the GPU's choice differs there, the
choice must still be within tolerance of the oracle's best, and the slots after
it are excluded from the comparison (they are conditioned on a different
predecessor).
"""
from __future__ import annotations

import functools
from typing import Dict, List, Tuple

import numpy as np

import oracle
import workloads

TOL_VEC = {"f32": 1e-5, "bf16": 2e-3}    # in/out vectors and pair scores
TOL_LOGP = 1e-3                            # log-probs and log-normaliser


def to_dev(a: np.ndarray, dtype: str, device="cuda"):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype == "bf16":
        t = t.to(torch.bfloat16)
    return t.to(device)


def compare_path(choice: np.ndarray, A: np.ndarray, P: np.ndarray, tol: float) -> Tuple[int, int]:
    """Walk the oracle's scores along the GPU's choices. Returns (slots compared,
    tied steps seen). Raises AssertionError on a difference that is not a tie."""
    L = len(choice)
    ties = 0
    prev = None
    for s in range(L):
        row = np.asarray(A if s == 0 else P[s - 1, prev], dtype=np.float64)
        best = int(np.argmax(row))             # first maximum
        srt = np.sort(row)
        if len(row) > 1 and srt[-1] - srt[-2] <= tol:
            ties += 1
        c = int(choice[s])
        if c != best:
            assert row[best] - row[c] <= tol, (
                f"step {s}: gpu picked {c} ({row[c]:.6f}), oracle best {best} ({row[best]:.6f})")
            return s, ties
        prev = c
    return L, ties


@functools.lru_cache(maxsize=2)
def workload_data(name: str, tier: int = 0):
    wl = workloads.WORKLOADS[name]
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds(tier), tier)
    return wl, W, inp


def oracle_topk_rows(logits: np.ndarray, K: int, rows: List[int]):
    out = []
    for r in rows:
        out.append(oracle.topk_lse(logits[r], K))
    return out


def embed_fn(wl):
    return lambda ids: workloads.embed_rows(wl.V, wl.H, wl.dtype, ids)
