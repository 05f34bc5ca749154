"""GPU parity of steps (3) and (4): cosine pair scores (Eq. "pair"; Sec. 3.5) and the
greedy walk (Sec. 3.5), against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from _helpers import to_dev

pytestmark = pytest.mark.gpu


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


@pytest.mark.parametrize("B,L,K,d,unit", [(1, 8, 4, 64, True), (3, 16, 8, 256, True),
                                          (2, 16, 16, 512, True), (5, 1, 3, 40, True),
                                          (2, 6, 32, 24, False), (4, 3, 1, 8, False),
                                          (7, 15, 8, 1024, True), (2, 5, 20, 36, True),
                                          (3, 4, 32, 256, False)])
def test_pair_scores_match_oracle(B, L, K, d, unit):
    ll = _ll()
    rng = np.random.default_rng(B * 100 + L * 10 + K + d)
    out = rng.standard_normal((B, L, K, d)).astype(np.float32)
    inn = rng.standard_normal((B, L, K, d)).astype(np.float32) * 0.1
    anc = rng.standard_normal((B, d)).astype(np.float32) * 7
    if unit:
        out /= np.linalg.norm(out, axis=-1, keepdims=True)
        inn /= np.linalg.norm(inn, axis=-1, keepdims=True)
        anc /= np.linalg.norm(anc, axis=-1, keepdims=True)
    A, P = ll.pair_scores(to_dev(out, "f32"), to_dev(inn, "f32"), to_dev(anc, "f32"))
    A, P = A.cpu().numpy(), P.cpu().numpy()
    assert A.size // B + P.size // B == (L - 1) * K * K + K
    for b in range(B):
        oA, oP = oracle.pair_scores(out[b].astype(np.float64), inn[b].astype(np.float64),
                                    anc[b].astype(np.float64))
        assert np.abs(A[b] - oA).max() <= 1e-5
        if L > 1:
            assert np.abs(P[b] - oP).max() <= 1e-5


@pytest.mark.parametrize("B,L,K", [(1, 8, 4), (9, 16, 8), (3, 16, 16), (2, 1, 5), (4, 12, 1),
                                   (2, 64, 32)])
def test_greedy_walk_matches_oracle_exactly(B, L, K):
    ll = _ll()
    rng = np.random.default_rng(L * 31 + K)
    A = rng.uniform(-1, 1, (B, K)).astype(np.float32)
    P = rng.uniform(-1, 1, (B, max(L - 1, 0), K, K)).astype(np.float32)
    if K > 2:   # plant exact ties: the walk must take the lower index
        A[:, 2] = A.max(axis=1)
        P[:, :, :, K - 1] = P.max(axis=3)
    ids = rng.integers(0, 151936, (B, L, K)).astype(np.int32)
    choice, tokens, margin = ll.greedy_walk(to_dev(A, "f32"), to_dev(P, "f32"), to_dev(ids, "f32"))
    choice, tokens, margin = choice.cpu().numpy(), tokens.cpu().numpy(), margin.cpu().numpy()
    for b in range(B):
        c, m = oracle.greedy_walk(A[b].astype(np.float64), P[b].astype(np.float64))
        assert np.array_equal(choice[b], c)
        assert np.array_equal(tokens[b], ids[b, np.arange(L), c])
        if K == 1:
            assert np.all(np.isinf(margin[b]))
        else:
            assert np.allclose(margin[b], m, atol=1e-6)


def test_teaser_toy_on_gpu():
    ll = _ll()
    A = np.array([[0.34, 0.81, 0.22]], np.float32)
    P = np.zeros((1, 0, 3, 3), np.float32)
    ids = np.array([[[11, 22, 33]]], np.int32)
    choice, tokens, _ = ll.greedy_walk(to_dev(A, "f32"), to_dev(P, "f32"), to_dev(ids, "f32"))
    assert int(choice[0, 0]) == 1 and int(tokens[0, 0]) == 22
