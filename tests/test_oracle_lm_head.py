"""CPU pins of the oracle's LM-head projection + step (1): special cases that reduce to
the already pinned top-K (identity and one-hot vocabularies), the shift invariance of
log-probabilities, and brute-force dot products on a tiny vocabulary."""
import numpy as np

import oracle


def test_identity_vocabulary_is_plain_topk():
    rng = np.random.default_rng(1)
    h = rng.normal(size=64)
    ids, logp, lse, x = oracle.lm_head_topk(h, np.eye(64), 8)
    rid, rlogp, rlse = oracle.topk_lse(h, 8)
    assert np.array_equal(ids, rid) and np.allclose(logp, rlogp) and np.isclose(lse, rlse)
    assert np.allclose(x, h)


def test_scaled_one_hot_rows():
    # row v of W picks hidden coordinate perm[v] with weight a_v: logit v = a_v h[perm[v]]
    rng = np.random.default_rng(2)
    H, V = 16, 40
    h = rng.normal(size=H)
    perm = rng.integers(0, H, V)
    a = rng.uniform(0.5, 2.0, V)
    W = np.zeros((V, H))
    W[np.arange(V), perm] = a
    ids, logp, lse, x = oracle.lm_head_topk(h, W, 5)
    want = a * h[perm]
    assert np.allclose(x, want)
    assert np.isclose(lse, np.log(np.exp(want).sum()))
    assert list(ids) == list(np.lexsort((np.arange(V), -want))[:5])


def test_a_common_row_shift_moves_only_the_normaliser():
    # adding w0 to every vocabulary row adds h.w0 to every logit
    rng = np.random.default_rng(3)
    H, V = 32, 500
    h = rng.normal(size=H)
    W = rng.normal(0, 0.1, (V, H))
    w0 = rng.normal(size=H)
    ids, logp, lse, _ = oracle.lm_head_topk(h, W, 8)
    ids2, logp2, lse2, _ = oracle.lm_head_topk(h, W + w0, 8)
    assert np.array_equal(ids, ids2) and np.allclose(logp, logp2)
    assert np.isclose(lse2 - lse, h @ w0)


def test_brute_force_dots():
    rng = np.random.default_rng(4)
    H, V = 7, 12
    h = rng.normal(size=H)
    W = rng.normal(size=(V, H))
    _, _, lse, x = oracle.lm_head_topk(h, W, 3)
    for v in range(V):
        assert np.isclose(x[v], sum(W[v, j] * h[j] for j in range(H)))
    assert np.isclose(lse, np.log(sum(np.exp(sum(W[v, j] * h[j] for j in range(H))) for v in range(V))))
