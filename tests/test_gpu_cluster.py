"""GPU parity of the cluster scoring-network kernel (four CTAs per sequence exchanging
column slices through distributed shared memory; Sec. 3.2, App. A) against the oracle's
fp64 network and against the unfused chain of kernels on the same inputs: a full 128-node
tile, padded and ragged node counts, K = 16, one slot with one candidate, and more clusters
than fit on the GPU at once. Its fused tail (the pair scores of Eq. "pair" and the greedy
walk of Sec. 3.5, summed over the four CTAs' column slices) against the pair kernel and the
oracle through the whole selection call."""
import numpy as np
import pytest
import torch

import workloads
import oracle
from test_gpu_fused import TOL, _ll, _oracle_check, _topk, _wl
from _helpers import TOL_LOGP, compare_path, embed_fn, to_dev

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
        _oracle_check(wl, W, inp, ids, logp, out, inn, anc, range(B))
    finally:
        head.close()


def _maxabs(x):
    return float(np.abs(x).max()) if x.size else 0.0


def _select(ll, head, wl, inp, mode):
    B = inp["logits"].shape[0]
    ll.test_fused_path(head, mode)
    try:
        ws = head.workspace(B)
        tok = ll.select_block(head, to_dev(inp["logits"], wl.dtype), to_dev(inp["hidden"], wl.dtype),
                              to_dev(inp["target"], wl.dtype), ws=ws)
        torch.cuda.synchronize()
        assert ws.status() == 0
        inter = {k: v.cpu().numpy() for k, v in ll.select_block_intermediates(head, B, ws).items()}
    finally:
        ll.test_fused_path(None, 1)
    return tok.cpu().numpy(), inter


@pytest.mark.parametrize("B,L,K", [(1, 16, 8), (3, 5, 3), (2, 8, 16), (2, 1, 1), (1, 4, 32),
                                   (2, 2, 1)])
def test_cluster_tail_matches_pair_kernel_and_oracle(B, L, K):
    ll = _ll()
    wl = _wl(B, L, K, seed=9700 + 10 * L + K)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        assert ll.test_fused_path(head, 3), "this head shape should take the cluster kernel"
        tok, it = _select(ll, head, wl, inp, 3)
        tok0, it0 = _select(ll, head, wl, inp, 0)
        assert np.array_equal(it["ids"], it0["ids"])
        assert _maxabs(it["A"] - it0["A"]) <= TOL and _maxabs(it["P"] - it0["P"]) <= TOL
        for b in range(B):
            r = oracle.select_sequence(inp["logits"][b], inp["hidden"][b], inp["target"][b],
                                       embed_fn(wl), W, wl.K)
            assert np.array_equal(it["ids"][b], r["ids"])
            assert np.abs(it["logp"][b] - r["logp"]).max() <= TOL_LOGP
            assert _maxabs(it["A"][b] - r["A"]) <= TOL
            assert _maxabs(it["P"][b] - r["P"]) <= TOL
            n, ties = compare_path(it["choice"][b], r["A"], r["P"], TOL)
            assert np.array_equal(tok[b, :n], r["tokens"][:n])
            if ties == 0:
                assert n == wl.L and np.array_equal(tok[b], r["tokens"])
            assert np.array_equal(tok[b], it["ids"][b][np.arange(wl.L), it["choice"][b]])
    finally:
        head.close()
