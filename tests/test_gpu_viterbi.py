"""GPU parity of the exact best path (App. E, Viterbi) against the oracle: random and
quantised (tied) score tensors, brute force over all K^L paths on tiny lattices, the edge
shapes (one slot, one candidate, the maximum L and K), and the fused selection call on the
workloads, where the chosen path must score within the float tolerance of the optimum and
never below the greedy path."""
import numpy as np
import pytest
import torch

import oracle
import workloads
from _helpers import to_dev, workload_data

pytestmark = pytest.mark.gpu
SIGMA = 8.0


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _scores(B, L, K, seed, quant=None):
    rng = np.random.default_rng(seed)
    A = rng.uniform(-1, 1, (B, K)).astype(np.float32)
    P = rng.uniform(-1, 1, (B, max(L - 1, 0), K, K)).astype(np.float32)
    if quant:
        A = (np.round(A / quant) * quant).astype(np.float32)
        P = (np.round(P / quant) * quant).astype(np.float32)
    ids = rng.integers(0, 50000, (B, L, K)).astype(np.int32)
    return A, P, ids


def _gpu(ll, A, P, ids):
    c, t, g = ll.best_path(to_dev(A, "f32"), to_dev(P, "f32"), to_dev(ids, "f32"), SIGMA)
    torch.cuda.synchronize()
    return c.cpu().numpy(), t.cpu().numpy(), g.cpu().numpy()


@pytest.mark.parametrize("B,L,K,quant", [(7, 8, 4, None), (5, 16, 8, None), (3, 16, 16, 0.125),
                                         (4, 12, 8, 0.25), (2, 1, 8, None), (3, 9, 1, None),
                                         (2, 64, 32, None)])
def test_best_path_matches_oracle(B, L, K, quant):
    ll = _ll()
    A, P, ids = _scores(B, L, K, seed=100 + L * K, quant=quant)
    c, t, g = _gpu(ll, A, P, ids)
    for b in range(B):
        oc, og = oracle.viterbi(A[b].astype(np.float64), P[b].astype(np.float64), SIGMA)
        assert np.array_equal(c[b], oc), (b, c[b], oc)
        assert np.array_equal(t[b], ids[b][np.arange(L), oc])
        assert abs(g[b] - og) <= 1e-5 * max(1.0, abs(og)) * L, (b, g[b], og)


def test_best_path_is_the_brute_force_maximum():
    ll = _ll()
    B, L, K = 6, 5, 3
    A, P, ids = _scores(B, L, K, seed=7)
    c, _, g = _gpu(ll, A, P, ids)
    for b in range(B):
        best = max(oracle.brute_force_paths(A[b].astype(np.float64), P[b].astype(np.float64), SIGMA),
                   key=lambda x: x[1])
        assert abs(g[b] - best[1]) <= 1e-5 * L
        assert abs(oracle.path_score(A[b], P[b], c[b], SIGMA) - best[1]) <= 1e-5 * L


def test_best_path_rejects_bad_arguments():
    ll = _ll()
    A, P, ids = _scores(1, 4, 4, seed=1)
    dA, dP, dI = to_dev(A, "f32"), to_dev(P, "f32"), to_dev(ids, "f32")
    out = torch.empty((1, 4), dtype=torch.int32, device="cuda")
    lib = ll.lib()
    assert lib.lilicorr_best_path(1, 4, 4, dA.data_ptr(), dP.data_ptr(), dI.data_ptr(), 0.0,
                                  out.data_ptr(), out.data_ptr(), None, None) == ll.ERR_ARG
    assert lib.lilicorr_best_path(1, 65, 4, dA.data_ptr(), dP.data_ptr(), dI.data_ptr(), 8.0,
                                  out.data_ptr(), out.data_ptr(), None, None) == ll.ERR_SHAPE


@pytest.mark.parametrize("name", ["tiny_f32", "single_request"])
def test_select_block_viterbi(name):
    ll = _ll()
    wl, W, inp = workload_data(name)
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype))
    try:
        B = min(wl.B, 2)
        args = [to_dev(inp[k][:B], wl.dtype) for k in ("logits", "hidden", "target")]
        ws = head.workspace(B)
        tok_v = ll.select_block(head, *args, ws=ws, walk="viterbi")
        torch.cuda.synchronize()
        inter = ll.select_block_intermediates(head, B, ws)
        A = inter["A"].cpu().numpy().astype(np.float64)
        P = inter["P"].cpu().numpy().astype(np.float64)
        choice = inter["choice"].cpu().numpy()
        ids = inter["ids"].cpu().numpy()
        tok_g = ll.select_block(head, *args, ws=ws, walk="greedy")
        torch.cuda.synchronize()
        choice_g = ll.select_block_intermediates(head, B, ws)["choice"].cpu().numpy()
        for b in range(B):
            _, g_opt = oracle.viterbi(A[b], P[b], SIGMA)
            g_v = oracle.path_score(A[b], P[b], choice[b], SIGMA)
            g_g = oracle.path_score(A[b], P[b], choice_g[b], SIGMA)
            assert g_opt - g_v <= SIGMA * 1e-5 * wl.L, (b, g_opt, g_v)
            assert g_v >= g_g - SIGMA * 1e-5 * wl.L
            assert np.array_equal(tok_v.cpu().numpy()[b], ids[b][np.arange(wl.L), choice[b]])
    finally:
        head.close()
