"""Pins of the oracle's top-K + log-normaliser (Sec. 3.2; App. A "Serving") against
closed forms, library routines, brute force and hand-worked tie cases."""
import json
import math
import os

import numpy as np
import pytest
import scipy.special
import torch

import oracle
import workloads

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _f(v):
    return float(v) if not isinstance(v, str) else float(v.replace("inf", "inf"))


def test_lse_matches_scipy_logsumexp():
    rng = np.random.default_rng(11)
    for V, std in [(7, 1.0), (1000, 3.0), (32000, 2.0), (151936, 0.3)]:
        x = rng.standard_normal(V) * std
        _, _, lse = oracle.topk_lse(x, min(4, V))
        assert abs(lse - scipy.special.logsumexp(x)) < 1e-9 * max(1.0, abs(lse))


def test_constant_row_closed_form():
    # all logits equal c: lse = c + log V, ids are the K lowest ids, logp = -log V
    for V, K, c in [(5, 5, 0.0), (1000, 8, -3.5), (151936, 16, 12.25)]:
        ids, logp, lse = oracle.topk_lse(np.full(V, c), K)
        assert abs(lse - (c + math.log(V))) < 1e-9 * max(1, abs(c))
        assert list(ids) == list(range(K))
        assert np.allclose(logp, -math.log(V), atol=1e-9)


def test_normalisation_invariants():
    rng = np.random.default_rng(5)
    x = rng.standard_normal(5000) * 4
    ids, logp, lse = oracle.topk_lse(x, 16)
    assert abs(np.sum(np.exp(x - lse)) - 1.0) < 1e-12      # sum_v p_v = 1
    assert lse >= x.max()
    assert np.all(logp <= 0)
    assert np.all(np.diff(logp) <= 0)                      # non-increasing in rank


def test_matches_torch_topk_on_tie_free_rows():
    rng = np.random.default_rng(7)
    for V, K in [(100, 1), (4097, 8), (151936, 16)]:
        x = rng.standard_normal(V)
        assert len(np.unique(x)) == V
        ids, logp, _ = oracle.topk_lse(x, K)
        tv, ti = torch.topk(torch.from_numpy(x), K)
        assert list(ids) == ti.tolist()
        assert np.allclose(x[ids], tv.numpy())
        assert np.allclose(logp, torch.log_softmax(torch.from_numpy(x), 0)[ti].numpy(), atol=1e-12)


def test_brute_force_selection_small_rows():
    # K largest by repeated removal of the (largest value, lowest id) element
    rng = np.random.default_rng(3)
    for _ in range(200):
        V = int(rng.integers(1, 12))
        K = int(rng.integers(1, V + 1))
        x = rng.integers(-3, 4, size=V).astype(float) * 0.5     # many ties
        left = list(range(V))
        want = []
        for _k in range(K):
            best = left[0]
            for v in left[1:]:
                if x[v] > x[best]:
                    best = v
            want.append(best)
            left.remove(best)
        ids, _, _ = oracle.topk_lse(x, K)
        assert list(ids) == want


def test_golden_ties():
    g = json.load(open(os.path.join(GOLD, "topk_ties.json")))
    for case in g["cases"]:
        x = np.array([_f(v) for v in case["x"]])
        ids, _, _ = oracle.topk_lse(x, case["K"])
        assert list(ids) == case["ids"], case


def test_rejects_nonfinite_rows():
    with pytest.raises(ValueError):
        oracle.topk_lse(np.array([1.0, np.nan, 2.0]), 1)
    with pytest.raises(ValueError):
        oracle.topk_lse(np.full(4, -np.inf), 1)
    with pytest.raises(ValueError):
        oracle.topk_lse(np.zeros(3), 4)


def test_quantised_workload_has_ties_and_zero_signs():
    # the tie-stress recipe must actually produce tied logits near the top and -0.0 values
    wl = workloads.WORKLOADS["ties_b256"]
    inp = workloads.sequence_inputs(wl, wl.seeds()[0])
    row = inp["logits"][0]
    ids, _, _ = oracle.topk_lse(row, wl.K)
    top = row[ids]
    assert len(np.unique(top)) < wl.K
    assert np.any(np.signbit(row) & (row == 0))
