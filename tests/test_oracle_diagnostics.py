"""CPU pins of the oracle's diagnostics: the local next-candidate distributions of
Eq. "localar", the decision gaps of Eq. "margin", and coverage / oracle prefix / prefix
acceptance (Sec. 3.3 "Oracle-prefix supervision"; Sec. 3.1)."""
import itertools

import numpy as np
import pytest
from scipy.special import logsumexp, softmax

import oracle


def _scores(L, K, seed):
    rng = np.random.default_rng(seed)
    return rng.uniform(-1, 1, K), rng.uniform(-1, 1, (L - 1, K, K))


def test_local_softmax_matches_library_softmax():
    A, P = _scores(6, 5, 1)
    pa, pp = oracle.local_softmax(A, P, 8.0)
    assert np.allclose(pa, softmax(8.0 * A))
    assert np.allclose(pp, softmax(8.0 * P, axis=-1))
    assert np.allclose(pp.sum(-1), 1.0) and np.isclose(pa.sum(), 1.0)


def test_constant_rows_are_uniform():
    pa, pp = oracle.local_softmax(np.full(4, 0.3), np.full((2, 4, 4), -0.7), 8.0)
    assert np.allclose(pa, 0.25) and np.allclose(pp, 0.25)


def test_chain_rule_defines_a_distribution_over_paths():
    # Eq. "localar" factorises the path distribution: the products over all K^L paths sum to 1
    L, K = 4, 3
    A, P = _scores(L, K, 2)
    total = 0.0
    for c in itertools.product(range(K), repeat=L):
        prob, _, lp = oracle.path_probs(A, P, c, 8.0)
        assert np.isclose(np.exp(lp), np.prod(prob))
        total += np.prod(prob)
    assert np.isclose(total, 1.0)


def test_log_prob_is_path_score_minus_normalisers():
    # log P(c) = g(c) - sum_s logsumexp(z_s), g of Eq. "pathscore" from its own function
    L, K, sigma = 7, 6, 8.0
    A, P = _scores(L, K, 3)
    c, _ = oracle.greedy_walk(A, P)
    _, _, lp = oracle.path_probs(A, P, c, sigma)
    norm = logsumexp(sigma * A) + sum(logsumexp(sigma * P[s - 1, c[s - 1]]) for s in range(1, L))
    assert np.isclose(lp, oracle.path_score(A, P, c, sigma) - norm)


def test_gaps_of_the_greedy_walk():
    L, K = 9, 8
    A, P = _scores(L, K, 4)
    c, marg = oracle.greedy_walk(A, P)
    _, gap, _ = oracle.path_probs(A, P, c, 8.0)
    assert (gap > 0).all()                        # every greedy step is a strict argmax here
    assert np.allclose(gap, 8.0 * marg)           # the decision gap is sigma times the walk margin
    _, gap1, _ = oracle.path_probs(A, P, c, 1.0)
    assert np.allclose(gap, 8.0 * gap1)           # linear in sigma
    # any other candidate at a step has a negative gap there
    c2 = c.copy()
    c2[3] = (c[3] + 1) % K
    _, gap2, _ = oracle.path_probs(A, P, c2, 8.0)
    assert gap2[3] < 0


def test_one_candidate():
    A, P = _scores(5, 1, 5)
    prob, gap, lp = oracle.path_probs(A, P, [0] * 5, 8.0)
    assert np.allclose(prob, 1.0) and np.isinf(gap).all() and lp == 0.0


@pytest.mark.parametrize("ids,tokens,truth,covered,prefix,accepted", [
    # worked by hand: slot 2 misses the truth among its candidates
    ([[5, 1], [7, 2], [3, 4], [11, 12]], [5, 7, 3, 11], [5, 7, 9, 11], [1, 1, 0, 1], 2, 2),
    # every slot covered, the walk picks a wrong candidate at slot 1
    ([[5, 1], [2, 7], [9, 4]], [5, 2, 9], [5, 7, 9], [1, 1, 1], 3, 1),
    # the first slot misses: nothing is accepted
    ([[1, 2], [3, 4]], [1, 3], [9, 3], [0, 1], 0, 0),
    # everything right
    ([[8, 6], [6, 8]], [8, 6], [8, 6], [1, 1], 2, 2),
])
def test_block_acceptance_worked_cases(ids, tokens, truth, covered, prefix, accepted):
    cov, pre, acc = oracle.block_acceptance(np.array(ids), np.array(tokens), np.array(truth))
    assert list(cov) == covered and pre == prefix and acc == accepted


def test_accepted_never_exceeds_oracle_prefix():
    rng = np.random.default_rng(6)
    for _ in range(200):
        L, K = 6, 3
        ids = rng.integers(0, 6, (L, K))
        truth = rng.integers(0, 6, L)
        tokens = ids[np.arange(L), rng.integers(0, K, L)]   # chosen among the candidates
        _, pre, acc = oracle.block_acceptance(ids, tokens, truth)
        assert acc <= pre
