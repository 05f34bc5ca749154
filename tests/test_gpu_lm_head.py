"""GPU parity of the LM-head projection fused with step (1) against the oracle: top-K ids
(exact where the fp64 logits are not within fp32 rounding of each other; otherwise the
chosen logits must match rank by rank), log-probabilities and normaliser within 1e-3, on
one and several row blocks (ragged), ragged vocabulary tiles, K up to 32 and the full
Qwen3-sized vocabulary; up to 16 rows take the kernel with the vocabulary tile as the A
operand, more rows the one with the hidden rows as A."""
import numpy as np
import pytest
import torch

import oracle
from _helpers import TOL_LOGP

pytestmark = pytest.mark.gpu


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _check(h, W, ids, logp, lse, K, rows_to_check):
    for r in rows_to_check:
        oid, olp, olse, x = oracle.lm_head_topk(h[r], W, K)
        g = ids[r]
        # logits of the chosen ids, rank by rank, against the oracle's K largest
        tol = 1e-4 * max(1.0, np.abs(x).max())
        assert np.abs(x[g] - x[oid]).max() <= tol, (r, g, oid)
        for k in range(K):
            near = np.abs(x - x[oid[k]]) <= tol
            if near.sum() == 1:                          # a unique value at this rank
                assert g[k] == oid[k], (r, k, g, oid)
        assert abs(lse[r] - olse) <= TOL_LOGP, (r, lse[r], olse)
        assert np.abs(logp[r] - (x[g] - olse)).max() <= TOL_LOGP


@pytest.mark.parametrize("rows,H,V,K", [(1, 64, 1000, 4), (16, 256, 33000, 8), (130, 512, 5000, 16),
                                        (20, 128, 257, 32), (16, 4096, 151936, 8),
                                        (16, 128, 1000, 32), (5, 64, 4097, 16), (13, 192, 20000, 32),
                                        (2, 64, 100, 8), (33, 64, 5000, 8), (64, 256, 33000, 16),
                                        (64, 4096, 151936, 8), (65, 128, 3000, 8)])
def test_lm_head_topk_matches_oracle(rows, H, V, K):
    ll = _ll()
    g = torch.Generator(device="cuda").manual_seed(rows * 31 + H + V)
    hid = torch.randn((rows, H), generator=g, device="cuda").to(torch.bfloat16)
    W = (0.02 * torch.randn((V, H), generator=g, device="cuda")).to(torch.bfloat16)
    ids, logp, lse = ll.lm_head_topk(hid, W, K)
    torch.cuda.synchronize()
    h64 = hid.float().cpu().numpy().astype(np.float64)
    W64 = W.float().cpu().numpy().astype(np.float64)
    check = range(rows) if rows * V <= 20 * 40000 else list(range(0, rows, 13)) + [rows - 1]
    _check(h64, W64, ids.cpu().numpy(), logp.cpu().numpy(), lse.cpu().numpy(), K, check)


def test_lm_head_topk_flags_nonfinite_and_rejects_shapes():
    ll = _ll()
    hid = torch.randn((4, 64), device="cuda").to(torch.bfloat16)
    hid[:, 3] = 1.0
    W = torch.randn((300, 64), device="cuda").to(torch.bfloat16)
    W[17, 3] = float("inf")                              # logit 17 of every row is +inf
    ws = ll.Workspace(ll.lib().lilicorr_lm_head_topk_workspace_bytes(4, 64, 300, 8))
    ll.lm_head_topk(hid, W, 8, ws=ws)
    assert ws.status() == ll.ERR_NONFINITE
    with pytest.raises(ll.LilicorrError):
        ll.lm_head_topk(torch.randn((4, 100), device="cuda").to(torch.bfloat16),
                        torch.randn((300, 100), device="cuda").to(torch.bfloat16), 8)   # H % 64
