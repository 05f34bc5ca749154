"""GPU parity of the chain's tcgen05 attention core (App. A: bidirectional attention over
the L*K nodes with the slot-distance and same-slot biases; 128 queries per CTA, S and
P V on the tensor cores) against the mma.sync kernel on the same inputs and against the
oracle's fp64 network: 32- and 64-wide heads, 9 to 256 nodes per sequence (ragged, K not a
multiple of 8, one query tile and two, full 256-node tiles)."""
import numpy as np
import pytest
import torch

import workloads
from test_gpu_fused import TOL, _ll, _oracle_check, _topk
from _helpers import to_dev

pytestmark = pytest.mark.gpu


def _run(ll, head, wl, ids, logp, inp, attn_mode):
    ll.test_fused_path(head, 0)                        # the chain of kernels
    prev = ll.test_attention_path(attn_mode)
    try:
        res = ll.embed_in_out(head, to_dev(ids.astype(np.int32), "f32"),
                              to_dev(logp.astype(np.float32), "f32"),
                              to_dev(inp["hidden"], wl.dtype), to_dev(inp["target"], wl.dtype))
        torch.cuda.synchronize()
    finally:
        ll.test_attention_path(prev)
        ll.test_fused_path(None, 1)
    return [t.cpu().numpy() for t in res]


@pytest.mark.parametrize("B,L,K,d", [(2, 5, 8, 256), (2, 3, 3, 256), (2, 16, 16, 256),
                                     (1, 16, 8, 512), (2, 9, 15, 512), (3, 1, 4, 256),
                                     (2, 16, 16, 512), (1, 32, 8, 512)])
def test_umma_attention_matches_mma_sync_and_oracle(B, L, K, d):
    ll = _ll()
    wl = workloads.Workload(f"umma_b{B}_l{L}_k{K}_d{d}", B=B, L=L, V=2000, K=K, d=d, H=256,
                            dtype="bf16", logit_kind="normal_planted", logit_param=(3.0, 8.0),
                            seed_base=9900 + 7 * L + K + d)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    ids, logp = _topk(wl, inp["logits"])
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        out, inn, anc = _run(ll, head, wl, ids, logp, inp, 1)
        assert np.isfinite(out).all() and np.isfinite(inn).all()
        out0, inn0, _ = _run(ll, head, wl, ids, logp, inp, 0)
        assert np.abs(out - out0).max() <= TOL and np.abs(inn - inn0).max() <= TOL
        _oracle_check(wl, W, inp, ids, logp, out, inn, anc, range(B))
    finally:
        head.close()
