"""GPU parity of the vocabulary-sharded step (1), simulated on one device: every shard's
partial record against the oracle's shard summary, and the merge of P shards against the
whole-row kernel (ids bit-exact, normaliser within fp32 rounding) and the oracle (ids
bit-exact, log-probs and normaliser within 1e-3), on random, tie-heavy (quantised), narrow
and all -inf shards."""
import numpy as np
import pytest
import torch

import oracle
from _helpers import TOL_LOGP, to_dev
from paper_2608_20530_gb300 import shards

pytestmark = pytest.mark.gpu


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _logits(rows, V, seed, quant=None):
    rng = np.random.default_rng(seed)
    x = rng.normal(0.0, 3.0, (rows, V)).astype(np.float32)
    if quant:
        x = (np.round(x / quant) * quant).astype(np.float32)
    return x


def _sharded(ll, xd, K, P):
    V = xd.shape[-1]
    recs = [ll.topk_lse_partial(xd[:, a:b].contiguous(), K, a) for a, b in shards.bounds(V, P)]
    return recs, ll.topk_lse_merge(torch.stack(recs), K)


@pytest.mark.parametrize("rows,V,K,P,dtype,quant", [
    (16, 151936, 8, 2, "bf16", None), (16, 151936, 8, 8, "bf16", None),
    (8, 151936, 16, 3, "bf16", 0.25), (4, 32000, 4, 5, "f32", None),
    (33, 4099, 32, 7, "bf16", 0.5), (3, 300, 8, 64, "f32", None),
    (5, 151936, 8, 152, "bf16", None)])
def test_merged_shards_match_the_whole_row(rows, V, K, P, dtype, quant):
    ll = _ll()
    x = _logits(rows, V, rows * 7 + P, quant)
    xd = to_dev(x, dtype)
    xr = xd.float().cpu().numpy().astype(np.float64)      # the values the kernels see
    recs, (ids, logp, lse) = _sharded(ll, xd, K, P)
    wids, wlogp, wlse = ll.topk_lse(xd, K)
    torch.cuda.synchronize()
    ids, logp, lse = ids.cpu().numpy(), logp.cpu().numpy(), lse.cpu().numpy()
    assert np.array_equal(ids, wids.cpu().numpy())
    assert np.abs(lse - wlse.cpu().numpy()).max() <= 2e-6 * max(1.0, np.abs(lse).max())
    assert np.abs(logp - wlogp.cpu().numpy()).max() <= 2e-6 * max(1.0, np.abs(logp).max())
    for r in range(0, rows, max(1, rows // 6)):
        oid, olp, olse = oracle.topk_lse(xr[r], K)
        assert np.array_equal(ids[r], oid), (r, ids[r], oid)
        assert abs(lse[r] - olse) <= TOL_LOGP and np.abs(logp[r] - olp).max() <= TOL_LOGP
    # the records themselves against the oracle's shard summaries
    for (a, b), rec in zip(shards.bounds(V, P), recs):
        m, s, vals, rids = shards.unpack_records(rec, K)
        for r in (0, rows - 1):
            om, os_, ov, oi = oracle.topk_lse_partial(xr[r, a:b], K, a)
            assert m[r] == om and abs(s[r] - os_) <= 1e-4 * os_
            assert np.array_equal(rids[r], oi) and np.array_equal(vals[r].astype(np.float64), ov)


def test_narrow_and_all_minus_inf_shards():
    ll = _ll()
    rows, V, K = 4, 64, 8
    x = _logits(rows, V, 11)
    x[:, 22:43] = -np.inf                    # the middle shard of three, [22, 43), only -inf
    xd = to_dev(x, "f32")
    recs, (ids, logp, lse) = _sharded(ll, xd, K, 3)
    m, s, vals, rids = shards.unpack_records(recs[1], K)
    assert np.all(m == -np.inf) and np.all(s == 0.0) and np.all(vals == -np.inf)
    assert np.array_equal(rids, np.tile(np.arange(22, 30), (rows, 1)))   # ties: lower ids
    for r in range(rows):
        oid, olp, olse = oracle.topk_lse(x[r].astype(np.float64), K)
        assert np.array_equal(ids.cpu().numpy()[r], oid)
        assert abs(lse.cpu().numpy()[r] - olse) <= TOL_LOGP
    # a shard narrower than K pads its record with (-inf, -1)
    rec = ll.topk_lse_partial(xd[:, :5].contiguous(), K, 0)
    _, _, vals, rids = shards.unpack_records(rec, K)
    assert np.all(rids[:, 5:] == -1) and np.all(vals[:, 5:] == -np.inf)
    assert np.array_equal(np.sort(rids[:, :5], axis=1), np.tile(np.arange(5), (rows, 1)))


def test_merge_flags_a_nan_row_and_rejects_too_many_shards():
    ll = _ll()
    x = _logits(3, 1000, 5)
    x[1, 777] = np.nan
    xd = to_dev(x, "f32")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    recs = [ll.topk_lse_partial(xd[:, a:b].contiguous(), 8, a) for a, b in shards.bounds(1000, 2)]
    ll.topk_lse_merge(torch.stack(recs), 8, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == ll.ERR_NONFINITE
    many = torch.zeros((257, 3, ll.topk_partial_bytes(32)), dtype=torch.uint8, device="cuda")
    with pytest.raises(ll.LilicorrError):
        ll.topk_lse_merge(many, 32)                    # 257 x 32 keys exceed the merge area
