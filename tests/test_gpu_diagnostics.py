"""GPU parity of the block diagnostics against the oracle: the local next-candidate
distributions (Eq. "localar"), probabilities and decision gaps (Eq. "margin") along a path,
and coverage / oracle prefix / prefix acceptance (bit-exact), including a planted-token
workload through the whole selection call."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from _helpers import to_dev

pytestmark = pytest.mark.gpu
SIGMA = 8.0


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _scores(B, L, K, seed):
    rng = np.random.default_rng(seed)
    return (rng.uniform(-1, 1, (B, K)).astype(np.float32),
            rng.uniform(-1, 1, (B, max(L - 1, 0), K, K)).astype(np.float32))


@pytest.mark.parametrize("B,L,K", [(3, 8, 4), (2, 16, 8), (2, 16, 32), (4, 1, 5), (2, 6, 1)])
def test_local_softmax(B, L, K):
    ll = _ll()
    A, P = _scores(B, L, K, seed=L * 31 + K)
    pa, pp = ll.local_softmax(to_dev(A, "f32"), to_dev(P, "f32"), SIGMA)
    pa, pp = pa.cpu().numpy(), pp.cpu().numpy()
    for b in range(B):
        oa, op = oracle.local_softmax(A[b], P[b], SIGMA)
        assert np.abs(pa[b] - oa).max() <= 1e-6
        if L > 1:
            assert np.abs(pp[b] - op).max() <= 1e-6


@pytest.mark.parametrize("B,L,K", [(3, 8, 4), (2, 16, 8), (2, 16, 32), (4, 1, 5), (2, 6, 1)])
def test_path_probs_greedy_and_random_paths(B, L, K):
    ll = _ll()
    A, P = _scores(B, L, K, seed=L * 17 + K)
    rng = np.random.default_rng(3)
    paths = [np.stack([oracle.greedy_walk(A[b], P[b])[0] for b in range(B)]),
             rng.integers(0, K, (B, L))]
    for c in paths:
        prob, gap, lp = ll.path_probs(to_dev(A, "f32"), to_dev(P, "f32"),
                                      to_dev(c.astype(np.int32), "f32"), SIGMA)
        prob, gap, lp = prob.cpu().numpy(), gap.cpu().numpy(), lp.cpu().numpy()
        for b in range(B):
            op, og, olp = oracle.path_probs(A[b], P[b], c[b], SIGMA)
            assert np.allclose(prob[b], op, rtol=1e-5, atol=1e-7)
            if K == 1:
                assert np.isinf(gap[b]).all()
            else:
                assert np.abs(gap[b] - og).max() <= 1e-5 * SIGMA
            assert abs(lp[b] - olp) <= 1e-4 * max(1.0, abs(olp))


def test_path_probs_flags_a_choice_out_of_range():
    ll = _ll()
    A, P = _scores(1, 4, 4, seed=9)
    c = np.array([[0, 4, 1, 2]], np.int32)
    prob, gap, lp = ll.path_probs(to_dev(A, "f32"), to_dev(P, "f32"), to_dev(c, "f32"), SIGMA)
    prob = prob.cpu().numpy()
    assert np.isfinite(prob[0, 0]) and np.isnan(prob[0, 1]) and np.isnan(lp.cpu().numpy()[0])


def test_block_acceptance_random_and_worked():
    ll = _ll()
    rng = np.random.default_rng(11)
    B, L, K = 257, 16, 8
    ids = rng.integers(0, 12, (B, L, K)).astype(np.int32)
    truth = rng.integers(0, 12, (B, L)).astype(np.int32)
    tokens = ids[np.arange(B)[:, None], np.arange(L)[None, :], rng.integers(0, K, (B, L))]
    tokens[:5] = truth[:5]                                    # some blocks fully right
    cov, pre, acc = ll.block_acceptance(to_dev(ids, "f32"), to_dev(tokens, "f32"),
                                        to_dev(truth, "f32"))
    cov, pre, acc = cov.cpu().numpy(), pre.cpu().numpy(), acc.cpu().numpy()
    for b in range(B):
        oc, op, oa = oracle.block_acceptance(ids[b], tokens[b], truth[b])
        assert np.array_equal(cov[b], oc) and pre[b] == op and acc[b] == oa


def test_acceptance_of_a_planted_workload():
    """single_request plants a boosted token per slot (+8 over N(0, 3)): that token is the
    ground truth; the chosen tokens are scored against it."""
    ll = _ll()
    wl0 = workloads.WORKLOADS["single_request"]
    seeds = wl0.block_seeds()[:4]
    inp = workloads.batch_inputs(wl0, seeds)
    W = workloads.head_weights(wl0)
    head = ll.Head.from_workload(wl0, W, workloads.embed_table(wl0.V, wl0.H, wl0.dtype))
    try:
        B = len(seeds)
        args = [to_dev(inp[k], wl0.dtype) for k in ("logits", "hidden", "target")]
        ws = head.workspace(B)
        tokens = ll.select_block(head, *args, ws=ws)
        ids = ll.select_block_intermediates(head, B, ws)["ids"].clone()
        truth = to_dev(inp["planted"].astype(np.int32), "f32")
        cov, pre, acc = ll.block_acceptance(ids, tokens, truth)
        torch.cuda.synchronize()
        ids_h, tok_h = ids.cpu().numpy(), tokens.cpu().numpy()
        for b in range(B):
            oc, op, oa = oracle.block_acceptance(ids_h[b], tok_h[b], inp["planted"][b])
            assert np.array_equal(cov.cpu().numpy()[b], oc)
            assert pre.cpu().numpy()[b] == op and acc.cpu().numpy()[b] == oa
            assert oa <= op
    finally:
        head.close()
