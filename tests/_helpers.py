"""Shared test helpers: device uploads and the tie-aware path comparison.

A greedy step whose runner-up score (by the oracle) lies within the float
tolerance of the best counts as a tie. The path check follows the GPU's own
choices through the oracle's full score tensor, so every slot is checked even
after a tie sends the two walks different ways.
"""
from __future__ import annotations

import dataclasses
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


@dataclasses.dataclass
class PathCheck:
    prefix: int       # steps where the GPU path equals the oracle's, from the start
    ties: int         # tied steps along the GPU path (oracle runner-up within tol)
    exact: int        # steps of the identical prefix that are not ties: a wrong
                      # candidate there would have failed the comparison


def check_path(choice: np.ndarray, A: np.ndarray, P: np.ndarray, tol: float) -> PathCheck:
    """Check the GPU's chosen path against the oracle's scores.

    (1) Every step, followed along the GPU's own path through the oracle's full score
        tensor, picks a candidate within ``tol`` of the best continuation of the GPU's
        previous choice (a valid greedy step, ties allowed).
    (2) Up to the first step where the two paths differ, they are identical, and that
        step must be a tie (oracle runner-up within ``tol``)."""
    L = len(choice)
    ties = exact = 0
    prefix = None
    prev = None
    oprev = None
    for s in range(L):
        row = np.asarray(A if s == 0 else P[s - 1, prev], dtype=np.float64)
        c = int(choice[s])
        assert row.max() - row[c] <= tol, (
            f"step {s}: gpu picked {c} ({row[c]:.6f}), best continuation {row.max():.6f}")
        srt = np.sort(row)
        tied = len(row) > 1 and srt[-1] - srt[-2] <= tol
        ties += int(tied)
        if prefix is None:
            orow = np.asarray(A if s == 0 else P[s - 1, oprev], dtype=np.float64)
            ob = int(np.argmax(orow))
            if ob != c:
                assert orow.max() - orow[c] <= tol
                prefix = s
            else:
                exact += int(not tied)
            oprev = ob
        prev = c
    return PathCheck(L if prefix is None else prefix, ties, exact)


def compare_path(choice: np.ndarray, A: np.ndarray, P: np.ndarray, tol: float) -> Tuple[int, int]:
    """check_path's (identical prefix length, tied steps)."""
    r = check_path(choice, A, P, tol)
    return r.prefix, r.ties


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
