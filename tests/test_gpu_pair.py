"""GPU parity of the two-CTA scoring-network kernel (129-256 nodes per sequence: two
128-node tiles on a cluster of two CTAs that exchange their keys and values per head;
Sec. 3.2, App. A) against the oracle's fp64 network and against the unfused chain of
kernels on the same inputs: a full 256-node sequence, ragged node counts, K not a multiple
of 8, and more sequences than clusters fit on the GPU (each cluster then runs several
sequences in turn)."""
import numpy as np
import pytest
import torch

import workloads
from test_gpu_fused import TOL, _ll, _oracle_check, _run, _topk, _wl

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,L,K", [(1, 16, 16), (3, 9, 15), (2, 20, 12), (2, 26, 5)])
def test_pair_matches_oracle_and_unfused(B, L, K):
    ll = _ll()
    wl = _wl(B, L, K, seed=9800 + L * K)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    ids, logp = _topk(wl, inp["logits"])
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        assert ll.test_fused_path(head, 2), "this head shape should take the two-CTA kernel"
        out, inn, anc = _run(ll, head, wl, ids, logp, inp, True)
        assert np.isfinite(out).all() and np.isfinite(inn).all()
        assert np.allclose(np.linalg.norm(out, axis=-1), 1, atol=1e-5)
        _oracle_check(wl, W, inp, ids, logp, out, inn, anc, range(B))
        out2, inn2, _ = _run(ll, head, wl, ids, logp, inp, False)
        assert np.abs(out - out2).max() <= TOL and np.abs(inn - inn2).max() <= TOL
    finally:
        head.close()


def test_pair_more_sequences_than_clusters():
    ll = _ll()
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    B = nsm + 7                                  # two CTAs each: more than one round
    wl = _wl(B, 16, 16, V=1000, H=256, seed=9900)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    x = inp["logits"]
    ids = np.argsort(-x, axis=-1, kind="stable")[..., :wl.K]
    logp = np.take_along_axis(x.astype(np.float64), ids, -1) - 10.0
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        out, inn, anc = _run(ll, head, wl, ids, logp, inp, True)
        again = _run(ll, head, wl, ids, logp, inp, True)      # a second call, same head
        assert np.array_equal(out, again[0]) and np.array_equal(inn, again[1])
        out2, inn2, _ = _run(ll, head, wl, ids, logp, inp, False)
        assert np.abs(out - out2).max() <= TOL and np.abs(inn - inn2).max() <= TOL
        _oracle_check(wl, W, inp, ids, logp, out, inn, anc, range(B))
    finally:
        head.close()
