"""GPU parity of step (2), the scoring network (Sec. 3.2; App. A), against the oracle's
fp64 restatement: unit out/in vectors and anchor within 1e-5 (fp32 head) or 2e-3
(bf16 head). The oracle's own top-K feeds both sides, isolating the network."""
import numpy as np
import pytest
import torch

import oracle
import workloads
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


@pytest.mark.parametrize("name", ["serving_b32", "ties_b256"])
def test_bf16_heads_sampled_sequences(name):
    wl, W, inp = workload_data(name)
    # top-K of every sequence by the oracle is slow at full size; sampled sequences use
    # the oracle's ids, the rest use a cheap argpartition (their vectors are not checked)
    B = wl.B
    ids = np.zeros((B, wl.L, wl.K), np.int64)
    logp = np.zeros((B, wl.L, wl.K))
    seqs = [0, B - 1]
    x = inp["logits"]
    for b in range(B):
        if b in seqs:
            for s in range(wl.L):
                ids[b, s], logp[b, s], _ = oracle.topk_lse(x[b, s], wl.K)
        else:
            part = np.argpartition(-x[b], wl.K, axis=1)[:, :wl.K]
            ids[b] = part
            logp[b] = -np.arange(wl.K, dtype=float)
    _check_head(wl, W, inp, ids, logp, seqs)


def test_max_nodes_fp32_head():
    # L*K = 512 nodes per sequence, the largest the library accepts
    wl = workloads.Workload("max_nodes", B=2, L=32, V=4096, K=16, d=64, H=64, dtype="f32",
                            logit_kind="normal_planted", logit_param=(2.0, 6.0), seed_base=77)
    W = workloads.head_weights(wl)
    inp = workloads.batch_inputs(wl, wl.seeds())
    ids, logp = _oracle_topk(wl, inp["logits"])
    _check_head(wl, W, inp, ids, logp, range(wl.B))
