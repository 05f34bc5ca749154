"""Pins of the oracle's pair scores, greedy walk and exact path (Eq. "pair",
Sec. 3.5, Eq. "pathscore", App. E) by brute force and special cases."""
import itertools
import json
import os

import numpy as np

import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _random_unit(rng, *shape):
    v = rng.standard_normal(shape)
    return v / np.linalg.norm(v, axis=-1, keepdims=True)


def _lattice(rng, L, K, d):
    out = _random_unit(rng, L, K, d)
    inn = _random_unit(rng, L, K, d)
    anc = _random_unit(rng, d)
    return out, inn, anc


def test_teaser_toy():
    g = json.load(open(os.path.join(GOLD, "teaser_toy.json")))
    A = np.array(g["anchor_scores"])
    c, _ = oracle.greedy_walk(A, np.zeros((0, 3, 3)))
    assert c[0] == g["expected_choice"]


def test_term_count():
    rng = np.random.default_rng(0)
    for L, K in [(8, 4), (15, 8), (16, 16), (1, 3)]:
        out, inn, anc = _lattice(rng, L, K, 5)
        A, P = oracle.pair_scores(out, inn, anc)
        # (B-2) K^2 + K with block B = L + 1 (Sec. 3.5)
        assert A.size + P.size == (L - 1) * K * K + K


def test_pair_scores_are_cosines_and_local():
    rng = np.random.default_rng(1)
    L, K, d = 5, 3, 7
    out = rng.standard_normal((L, K, d)) * 3          # not unit: cosine must normalise
    inn = rng.standard_normal((L, K, d)) * 0.1
    anc = rng.standard_normal(d)
    A, P = oracle.pair_scores(out, inn, anc)
    assert np.all(np.abs(P) <= 1 + 1e-12) and np.all(np.abs(A) <= 1 + 1e-12)
    # P[s] depends only on out[s] and in[s+1]; swap roles check with explicit angles
    for s in range(L - 1):
        for k in range(K):
            for k2 in range(K):
                a, b = out[s, k], inn[s + 1, k2]
                ang = np.arccos(np.clip(P[s, k, k2], -1, 1))
                # law of cosines on the unit-normalised vectors
                ua, ub = a / np.linalg.norm(a), b / np.linalg.norm(b)
                assert abs(np.linalg.norm(ua - ub) ** 2 - (2 - 2 * np.cos(ang))) < 1e-9
    out2 = out.copy()
    out2[2] += 1.0
    _, P2 = oracle.pair_scores(out2, inn, anc)
    changed = [s for s in range(L - 1) if not np.allclose(P[s], P2[s])]
    assert changed == [2]


def _lexicographic_greedy(A, P):
    """Brute force: the path whose per-step score vector (A[c1], P[c1,c2], ...) is
    lexicographically largest, every path enumerated."""
    L, K = P.shape[0] + 1, A.shape[0]
    best, best_vec = None, None
    for c in itertools.product(range(K), repeat=L):
        vec = [A[c[0]]] + [P[s - 1, c[s - 1], c[s]] for s in range(1, L)]
        if best is None or vec > best_vec:
            best, best_vec = c, vec
    return np.array(best)


def test_greedy_is_lexicographic_maximiser_and_viterbi_is_exact():
    rng = np.random.default_rng(2)
    for L, K in [(4, 3), (6, 2), (5, 4), (8, 4)]:
        out, inn, anc = _lattice(rng, L, K, 6)
        A, P = oracle.pair_scores(out, inn, anc)
        c, _ = oracle.greedy_walk(A, P)
        assert list(c) == list(_lexicographic_greedy(A, P))
        cv, gv = oracle.viterbi(A, P)
        scores = {p: g for p, g in oracle.brute_force_paths(A, P)}
        gmax = max(scores.values())
        assert abs(gv - gmax) < 1e-9
        assert abs(scores[tuple(cv)] - gmax) < 1e-9
        assert oracle.path_score(A, P, c) <= gv + 1e-12


def test_greedy_can_differ_from_exact():
    # hand lattice where the greedy first pick blocks the best total (App. E motivation)
    A = np.array([0.9, 0.8])
    P = np.array([[[-0.9, -0.9], [0.9, 0.9]]])   # from cand 0 everything is bad
    c, _ = oracle.greedy_walk(A, P)
    cv, _ = oracle.viterbi(A, P)
    assert list(c) == [0, 0] and list(cv) == [1, 0]


def test_k_equals_one_is_per_slot_argmax():
    rng = np.random.default_rng(4)
    out, inn, anc = _lattice(rng, 6, 1, 4)
    A, P = oracle.pair_scores(out, inn, anc)
    c, marg = oracle.greedy_walk(A, P)
    assert list(c) == [0] * 6
    assert np.all(np.isinf(marg))


def test_walk_ties_take_lower_index_and_margin():
    A = np.array([0.5, 0.5, 0.1])
    P = np.array([[[0.2, 0.3, 0.3], [0, 0, 0], [0, 0, 0]]])
    c, marg = oracle.greedy_walk(A, P)
    assert list(c) == [0, 1]
    assert marg[0] == 0.0 and marg[1] == 0.0
