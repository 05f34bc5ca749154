"""GPU parity of the cluster scoring-network kernel (four CTAs per sequence exchanging
column slices through distributed shared memory; Sec. 3.2, App. A) against the oracle's
fp64 network and against the unfused chain of kernels on the same inputs: a full 128-node
tile, padded and ragged node counts, K = 16, one slot with one candidate, and more clusters
than fit on the GPU at once."""
import numpy as np
import pytest
import torch

import workloads
from test_gpu_fused import TOL, _ll, _oracle_check, _topk, _wl
from _helpers import to_dev

pytestmark = pytest.mark.gpu


def _run(ll, head, wl, ids, logp, inp, mode):
    ll.test_fused_path(head, mode)
    try:
        res = ll.embed_in_out(head, to_dev(ids.astype(np.int32), "f32"),
                              to_dev(logp.astype(np.float32), "f32"),
                              to_dev(inp["hidden"], wl.dtype), to_dev(inp["target"], wl.dtype))
        torch.cuda.synchronize()
    finally:
        ll.test_fused_path(None, 1)
    return [t.cpu().numpy() for t in res]


@pytest.mark.parametrize("B,L,K", [(1, 16, 8), (3, 5, 3), (2, 8, 16), (2, 1, 1)])
def test_cluster_matches_oracle_and_unfused(B, L, K):
    ll = _ll()
    wl = _wl(B, L, K)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    ids, logp = _topk(wl, inp["logits"])
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        assert ll.test_fused_path(head, 3), "this head shape should take the cluster kernel"
        ws = head.workspace(B)
        out, inn, anc = _run(ll, head, wl, ids, logp, inp, 3)
        assert np.isfinite(out).all() and np.isfinite(inn).all()
        assert np.allclose(np.linalg.norm(out, axis=-1), 1, atol=1e-5)
        _oracle_check(wl, W, inp, ids, logp, out, inn, anc, range(B))
        out2, inn2, _ = _run(ll, head, wl, ids, logp, inp, 0)
        assert np.abs(out - out2).max() <= TOL and np.abs(inn - inn2).max() <= TOL
    finally:
        head.close()


def test_cluster_more_sequences_than_fit():
    ll = _ll()
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    B = nsm // 2 + 5                                  # 4 CTAs each: about two waves
    wl = _wl(B, 4, 4, V=1000, H=256, seed=9600)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    x = inp["logits"]
    ids = np.argsort(-x, axis=-1, kind="stable")[..., :wl.K]
    logp = np.take_along_axis(x.astype(np.float64), ids, -1) - 10.0
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        out, inn, anc = _run(ll, head, wl, ids, logp, inp, 3)
        again = _run(ll, head, wl, ids, logp, inp, 3)
        assert np.array_equal(out, again[0]) and np.array_equal(inn, again[1])
        out2, inn2, _ = _run(ll, head, wl, ids, logp, inp, 0)
        assert np.abs(out - out2).max() <= TOL and np.abs(inn - inn2).max() <= TOL
        _oracle_check(wl, W, inp, ids, logp, out, inn, anc, [0, B // 2, B - 1])
    finally:
        head.close()
