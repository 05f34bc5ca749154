"""GPU parity of step (2), the scoring network (Sec. 3.2; App. A), against the oracle's
fp64 restatement: unit out/in vectors and anchor within 1e-5 (fp32 head) or 2e-3
(bf16 head). The oracle's own top-K feeds both sides, isolating the network."""
import numpy as np
import pytest
import torch

import oracle
import workloads
import _oracle_pool
from _helpers import TOL_VEC, embed_fn, to_dev, workload_data

pytestmark = pytest.mark.gpu


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _oracle_topk(wl, logits):
    B = logits.shape[0]
    ids = np.zeros((B, wl.L, wl.K), np.int64)
    logp = np.zeros((B, wl.L, wl.K))
    for b in range(B):
        for s in range(wl.L):
            ids[b, s], logp[b, s], _ = oracle.topk_lse(logits[b, s], wl.K)
    return ids, logp


def _check_head(wl, W, inp, ids, logp, seqs):
    ll = _ll()
    E = workloads.embed_table(wl.V, wl.H, wl.dtype)
    head = ll.Head.from_workload(wl, W, E)
    out, inn, anc = ll.embed_in_out(head, to_dev(ids.astype(np.int32), "f32"),
                                    to_dev(logp.astype(np.float32), "f32"),
                                    to_dev(inp["hidden"], wl.dtype), to_dev(inp["target"], wl.dtype))
    torch.cuda.synchronize()
    out, inn, anc = out.cpu().numpy(), inn.cpu().numpy(), anc.cpu().numpy()
    tol = TOL_VEC[wl.dtype]
    assert np.allclose(np.linalg.norm(out, axis=-1), 1, atol=1e-5)
    assert np.allclose(np.linalg.norm(inn, axis=-1), 1, atol=1e-5)
    emb = embed_fn(wl)
    for b in seqs:
        E_rows = emb(ids[b].reshape(-1)).reshape(wl.L, wl.K, wl.H)
        o, i, a = oracle.head_forward(ids[b], logp[b].astype(np.float32).astype(np.float64),
                                      inp["hidden"][b], inp["target"][b], E_rows, W)
        e_out, e_in, e_anc = np.abs(out[b] - o).max(), np.abs(inn[b] - i).max(), np.abs(anc[b] - a).max()
        assert e_out <= tol and e_in <= tol and e_anc <= tol, (b, e_out, e_in, e_anc)
    head.close()


def test_tiny_f32_head():
    wl, W, inp = workload_data("tiny_f32")
    ids, logp = _oracle_topk(wl, inp["logits"])
    _check_head(wl, W, inp, ids, logp, range(wl.B))


@pytest.mark.parametrize("name,tier", [("serving_b32", 0), ("entropy_tiers_b64", 2),
                                       ("ties_b256", 0)])
def test_bf16_heads_every_sequence(name, tier):
    """The oracle's own top-K of every sequence feeds both sides; every sequence's
    vectors are compared (the oracle network fanned out over the host cores)."""
    wl, W, inp = workload_data(name, tier)
    seeds = wl.seeds(tier)
    ids, logp, _ = _oracle_pool.topk(wl, seeds, tier)
    lp32 = logp.astype(np.float32).astype(np.float64)    # what the GPU receives
    refs = _oracle_pool.network(wl, seeds, ids, lp32, tier)
    ll = _ll()
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        out, inn, anc = ll.embed_in_out(head, to_dev(ids.astype(np.int32), "f32"),
                                        to_dev(logp.astype(np.float32), "f32"),
                                        to_dev(inp["hidden"], wl.dtype),
                                        to_dev(inp["target"], wl.dtype))
        torch.cuda.synchronize()
    finally:
        head.close()
    out, inn, anc = out.cpu().numpy(), inn.cpu().numpy(), anc.cpu().numpy()
    tol = TOL_VEC[wl.dtype]
    worst = 0.0
    for b, r in enumerate(refs):
        e = max(np.abs(out[b] - r["out"]).max(), np.abs(inn[b] - r["in"]).max(),
                np.abs(anc[b] - r["anchor"]).max())
        assert e <= tol, (b, e)
        worst = max(worst, e)
    print(f"{name} tier {tier}: {len(refs)} sequences, worst vector error {worst:.2e}")


def test_max_nodes_fp32_head():
    # L*K = 512 nodes per sequence, the largest the library accepts
    wl = workloads.Workload("max_nodes", B=2, L=32, V=4096, K=16, d=64, H=64, dtype="f32",
                            logit_kind="normal_planted", logit_param=(2.0, 6.0), seed_base=77)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    ids, logp = _oracle_topk(wl, inp["logits"])
    _check_head(wl, W, inp, ids, logp, range(wl.B))
