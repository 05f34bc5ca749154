"""GPU parity of the fused scoring-network kernel (one CTA per sequence, Sec. 3.2; App. A)
against the oracle's fp64 network, and against the unfused chain of kernels on the same
inputs. Shapes cover a full 128-node tile, padded and ragged node counts, one slot with
one candidate, K = 16, and more sequences than SMs (CTAs that take several sequences)."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from _helpers import TOL_VEC, to_dev

pytestmark = pytest.mark.gpu
TOL = TOL_VEC["bf16"]


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _wl(B, L, K, V=3000, H=512, seed=9000):
    return workloads.Workload(f"fused_b{B}_l{L}_k{K}", B=B, L=L, V=V, K=K, d=256, H=H,
                              dtype="bf16", logit_kind="normal_planted",
                              logit_param=(3.0, 8.0), seed_base=seed)


def _topk(wl, logits):
    B = logits.shape[0]
    ids = np.zeros((B, wl.L, wl.K), np.int64)
    logp = np.zeros((B, wl.L, wl.K))
    for b in range(B):
        for s in range(wl.L):
            ids[b, s], logp[b, s], _ = oracle.topk_lse(logits[b, s], wl.K)
    return ids, logp


def _run(ll, head, wl, ids, logp, inp, fused):
    ll.test_fused_path(head, 2 if fused else 0)
    try:
        res = ll.embed_in_out(head, to_dev(ids.astype(np.int32), "f32"),
                              to_dev(logp.astype(np.float32), "f32"),
                              to_dev(inp["hidden"], wl.dtype), to_dev(inp["target"], wl.dtype))
        torch.cuda.synchronize()
    finally:
        ll.test_fused_path(None, 1)
    return [t.cpu().numpy() for t in res]


def _oracle_check(wl, W, inp, ids, logp, out, inn, anc, seqs):
    for b in seqs:
        E_rows = workloads.embed_rows(wl.V, wl.H, wl.dtype, ids[b].reshape(-1)).reshape(
            wl.L, wl.K, wl.H)
        o, i, a = oracle.head_forward(ids[b], logp[b].astype(np.float32).astype(np.float64),
                                      inp["hidden"][b], inp["target"][b], E_rows, W)
        errs = (np.abs(out[b] - o).max(), np.abs(inn[b] - i).max(), np.abs(anc[b] - a).max())
        assert max(errs) <= TOL, (b, errs)


@pytest.mark.parametrize("B,L,K", [(1, 16, 8), (3, 5, 3), (2, 8, 16), (2, 1, 1)])
def test_fused_matches_oracle_and_unfused(B, L, K):
    ll = _ll()
    wl = _wl(B, L, K)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    ids, logp = _topk(wl, inp["logits"])
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        assert ll.test_fused_path(head, 1), "this head shape should take the fused kernel"
        out, inn, anc = _run(ll, head, wl, ids, logp, inp, True)
        assert np.isfinite(out).all() and np.isfinite(inn).all()
        assert np.allclose(np.linalg.norm(out, axis=-1), 1, atol=1e-5)
        _oracle_check(wl, W, inp, ids, logp, out, inn, anc, range(B))
        out2, inn2, anc2 = _run(ll, head, wl, ids, logp, inp, False)
        assert np.abs(out - out2).max() <= TOL and np.abs(inn - inn2).max() <= TOL
        assert np.abs(anc - anc2).max() <= 1e-6      # the anchor is not on the fused path
    finally:
        head.close()


def test_fused_more_sequences_than_sms():
    ll = _ll()
    nsm = torch.cuda.get_device_properties(0).multi_processor_count
    B = 2 * nsm + 5
    wl = _wl(B, 4, 4, V=1000, H=256, seed=9500)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    # the oracle's top-K is exact but slow; these ids need only be valid candidates
    x = inp["logits"]
    ids = np.argsort(-x, axis=-1, kind="stable")[..., :wl.K]
    logp = np.take_along_axis(x.astype(np.float64), ids, -1) - 10.0
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        assert ll.test_fused_path(head, 1)
        out, inn, anc = _run(ll, head, wl, ids, logp, inp, True)
        again = _run(ll, head, wl, ids, logp, inp, True)       # a second call, same head
        assert np.array_equal(out, again[0]) and np.array_equal(inn, again[1])
        out2, inn2, _ = _run(ll, head, wl, ids, logp, inp, False)
        assert np.abs(out - out2).max() <= TOL and np.abs(inn - inn2).max() <= TOL
        _oracle_check(wl, W, inp, ids, logp, out, inn, anc, range(B))
    finally:
        head.close()
