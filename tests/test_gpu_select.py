"""GPU parity of the fused path lilicorr_select_block (steps 1-4) on every workload:
top-K ids bit-exact, log-probs within 1e-3, pair scores within the vector tolerance,
and chosen tokens equal to the oracle's up to tied walk steps."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from _helpers import TOL_LOGP, TOL_VEC, compare_path, embed_fn, to_dev, workload_data

pytestmark = pytest.mark.gpu


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _select_and_check(wl, W, inp, seqs):
    ll = _ll()
    E = workloads.embed_table(wl.V, wl.H, wl.dtype)
    head = ll.Head.from_workload(wl, W, E)
    B = inp["logits"].shape[0]
    ws = head.workspace(B)
    tokens = ll.select_block(head, to_dev(inp["logits"], wl.dtype), to_dev(inp["hidden"], wl.dtype),
                             to_dev(inp["target"], wl.dtype), ws=ws)
    torch.cuda.synchronize()
    assert ws.status() == 0
    inter = {k: v.cpu().numpy() for k, v in ll.select_block_intermediates(head, B, ws).items()}
    tokens = tokens.cpu().numpy()
    tol = TOL_VEC[wl.dtype]
    stats = {"slots": 0, "compared": 0, "ties": 0}
    for b in seqs:
        r = oracle.select_sequence(inp["logits"][b], inp["hidden"][b], inp["target"][b],
                                   embed_fn(wl), W, wl.K)
        assert np.array_equal(inter["ids"][b], r["ids"])
        assert np.abs(inter["logp"][b] - r["logp"]).max() <= TOL_LOGP
        assert np.abs(inter["lse"][b] - r["lse"]).max() <= TOL_LOGP
        assert np.abs(inter["A"][b] - r["A"]).max() <= tol
        assert np.abs(inter["P"][b] - r["P"]).max() <= tol
        n, ties = compare_path(inter["choice"][b], r["A"], r["P"], tol)
        assert np.array_equal(tokens[b, :n], r["tokens"][:n])
        if ties == 0:
            assert n == wl.L and np.array_equal(tokens[b], r["tokens"])
        assert np.array_equal(tokens[b], inter["ids"][b][np.arange(wl.L), inter["choice"][b]])
        stats["slots"] += wl.L
        stats["compared"] += n
        stats["ties"] += ties
    head.close()
    print(f"{wl.name}: {stats}")
    return stats


def test_tiny_f32_select():
    wl, W, inp = workload_data("tiny_f32")
    _select_and_check(wl, W, inp, range(wl.B))


def test_single_request_blocks():
    wl = workloads.WORKLOADS["single_request"]
    W = workloads.head_weights(wl)
    for seed in wl.block_seeds()[:3]:
        inp = workloads.batch_inputs(wl, [seed])
        _select_and_check(wl, W, inp, [0])


@pytest.mark.parametrize("name,tier", [("serving_b32", 0), ("entropy_tiers_b64", 0),
                                       ("entropy_tiers_b64", 1), ("entropy_tiers_b64", 2),
                                       ("ties_b256", 0)])
def test_batched_workloads_sampled(name, tier):
    wl, W, inp = workload_data(name, tier)
    B = inp["logits"].shape[0]
    _select_and_check(wl, W, inp, [0, B // 2, B - 1])
