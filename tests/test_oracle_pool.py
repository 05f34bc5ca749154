"""CPU checks of the parity tests' own machinery: the oracle process pool returns what the
oracle returns when called directly, and the tie-aware path check rejects a wrong step,
counts ties and counts the exactly compared steps."""
import numpy as np
import pytest

import _oracle_pool
import oracle
import workloads
from _helpers import check_path


def _small_wl():
    return workloads.Workload("pool_check", B=3, L=5, V=700, K=4, d=64, H=64, dtype="bf16",
                              logit_kind="quantised_normal", logit_param=(2.0, 0.25),
                              seed_base=321)


@pytest.mark.parametrize("which", ["tiny_f32", "small"])
def test_pool_matches_direct_oracle(which):
    wl = workloads.WORKLOADS["tiny_f32"] if which == "tiny_f32" else _small_wl()
    seeds = wl.seeds()
    refs = _oracle_pool.select(wl, seeds)
    W = workloads.head_weights(wl)
    emb = lambda ids: workloads.embed_rows(wl.V, wl.H, wl.dtype, ids)
    for s, r in zip(seeds, refs):
        inp = workloads.sequence_inputs(wl, s)
        d = oracle.select_sequence(inp["logits"], inp["hidden"], inp["target"], emb, W, wl.K)
        for k in ("ids", "logp", "lse", "out", "in", "anchor", "A", "P", "choice", "tokens"):
            assert np.array_equal(np.asarray(r[k]), np.asarray(d[k])), k


def test_path_check_counts_and_rejects():
    K, L = 3, 4
    A = np.array([0.9, 0.1, 0.2])
    P = np.zeros((L - 1, K, K))
    P[0, 0] = [0.1, 0.8, 0.3]
    P[1, 1] = [0.5, 0.5005, 0.1]          # a tie under 1e-3
    P[2, 1] = [0.2, 0.1, 0.7]
    P[2, 0] = [0.6, 0.1, 0.2]
    # the oracle's path: 0, 1, 1, 2; the untied steps are 0, 1 and 3
    pc = check_path(np.array([0, 1, 1, 2]), A, P, 1e-3)
    assert (pc.prefix, pc.ties, pc.exact) == (4, 1, 3)
    # taking the other side of the tie is allowed; the paths then part at step 2
    P[2, 0] = [0.6, 0.1, 0.2]
    pc = check_path(np.array([0, 1, 0, 0]), A, P, 1e-3)
    assert (pc.prefix, pc.ties, pc.exact) == (2, 1, 2)
    # a wrong untied step fails
    with pytest.raises(AssertionError):
        check_path(np.array([0, 2, 1, 2]), A, P, 1e-3)
    with pytest.raises(AssertionError):
        check_path(np.array([1, 1, 1, 2]), A, P, 1e-3)
