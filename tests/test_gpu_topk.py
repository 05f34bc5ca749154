"""GPU parity of step (1), top-K + log-normaliser (Sec. 3.2; App. A "Serving"), against
the oracle: ids bit-exact, log-probs and log-normaliser within 1e-3, on every row of
every full-size workload (the oracle fanned out over the host cores) and on ragged,
tied, -0/-inf and non-finite rows."""
import numpy as np
import pytest
import torch

import oracle
import workloads
import _oracle_pool
from _helpers import TOL_LOGP, to_dev, workload_data

pytestmark = pytest.mark.gpu


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _close(a, b, tol):
    """Equal infinities at the same places, finite entries within tol."""
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    inf = np.isinf(b)
    return np.array_equal(np.isinf(a), inf) and np.all(a[inf] == b[inf]) and \
        (not np.any(~inf) or np.abs(a[~inf] - b[~inf]).max() <= tol)


def _check_rows(x: np.ndarray, K: int, ids, logp, lse, rows):
    for r in rows:
        oid, olp, olse = oracle.topk_lse(x[r], K)
        assert np.array_equal(ids[r], oid), f"row {r}: {ids[r]} vs {oid}"
        assert abs(lse[r] - olse) <= TOL_LOGP, (r, lse[r], olse)
        assert _close(logp[r], olp, TOL_LOGP), (r, logp[r], olp)


def _run(x: np.ndarray, K: int, dtype: str):
    ll = _ll()
    t = to_dev(x, dtype)
    ws = ll.Workspace(ll.lib().lilicorr_topk_lse_workspace_bytes(x.shape[0], x.shape[1], K))
    ids, logp, lse = ll.topk_lse(t, K, ws=ws)
    torch.cuda.synchronize()
    return ids.cpu().numpy(), logp.cpu().numpy(), lse.cpu().numpy(), ws.status()


def test_tiny_workload_all_rows():
    wl, _, inp = workload_data("tiny_f32")
    x = inp["logits"].reshape(-1, wl.V)
    ids, logp, lse, st = _run(x, wl.K, wl.dtype)
    assert st == 0
    _check_rows(x, wl.K, ids, logp, lse, range(x.shape[0]))


def _check_all(ids, logp, lse, oids, ologp, olse):
    """Every row: ids bit-exact, log-probs and normaliser within 1e-3."""
    bad = np.nonzero(~np.all(ids == oids, axis=-1))[0]
    assert bad.size == 0, f"{bad.size} rows differ, first {bad[0]}: {ids[bad[0]]} vs {oids[bad[0]]}"
    assert np.abs(lse - olse).max() <= TOL_LOGP
    assert np.abs(logp - ologp).max() <= TOL_LOGP


@pytest.mark.parametrize("name,tier", [("serving_b32", 0), ("entropy_tiers_b64", 0),
                                       ("entropy_tiers_b64", 1), ("entropy_tiers_b64", 2),
                                       ("ties_b256", 0)])
def test_full_size_workloads_every_row(name, tier):
    """One call over the whole batch (the launch of the batched selection), every row
    against the oracle's full sort."""
    wl, _, inp = workload_data(name, tier)
    x = inp["logits"].reshape(-1, wl.V)
    ids, logp, lse, st = _run(x, wl.K, wl.dtype)
    assert st == 0
    oids, ologp, olse = _oracle_pool.topk(wl, wl.seeds(tier), tier)
    _check_all(ids, logp, lse, oids.reshape(ids.shape), ologp.reshape(logp.shape),
               olse.reshape(lse.shape))


def test_single_request_every_block():
    """All 1000 blocks of the batch-1 workload, each its own 16-row call (the split-row
    launch the batch-1 selection makes), against the oracle."""
    ll = _ll()
    wl = workloads.WORKLOADS["single_request"]
    seeds = wl.block_seeds()
    oids, ologp, olse = _oracle_pool.topk(wl, seeds)
    ws = ll.Workspace(ll.lib().lilicorr_topk_lse_workspace_bytes(wl.L, wl.V, wl.K))
    got = []
    for i0 in range(0, len(seeds), 100):
        inp = workloads.batch_inputs(wl, seeds[i0:i0 + 100])
        t = to_dev(inp["logits"], wl.dtype)
        outs = [ll.topk_lse(t[j], wl.K, ws=ws) for j in range(t.shape[0])]
        torch.cuda.synchronize()
        got += [[o.cpu().numpy() for o in r] for r in outs]
        del t, inp
    assert ws.status() == 0
    ids = np.stack([g[0] for g in got])
    logp = np.stack([g[1] for g in got])
    lse = np.stack([g[2] for g in got])
    _check_all(ids, logp, lse, oids, ologp, olse)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("rows,V,K", [(1, 1, 1), (3, 7, 7), (37, 1001, 5), (5, 9, 8),
                                      (2, 151936, 32), (1, 151936, 1), (300, 4096, 16),
                                      (64, 33, 32)])
def test_shapes_and_ragged_rows(dtype, rows, V, K):
    rng = np.random.default_rng(rows * 1000 + V + K)
    x = rng.standard_normal((rows, V)).astype(np.float32) * 3
    if dtype == "bf16":
        x = workloads.round_to_bf16(x)
    ids, logp, lse, st = _run(x, K, dtype)
    assert st == 0
    _check_rows(x, K, ids, logp, lse, range(rows))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_ties_zero_signs_and_minus_inf(dtype):
    V = 5000
    x = np.zeros((6, V), dtype=np.float32)
    x[0] = 1.5                                            # all equal: ids 0..K-1
    x[1] = np.where(np.arange(V) % 2 == 0, -0.0, 0.0)     # -0 == +0
    x[1, 4321] = -1.0
    x[2] = np.round(np.random.default_rng(1).standard_normal(V) * 2) * 0.25
    x[3] = -np.inf
    x[3, [17, 4000, 2]] = [3.0, 3.0, -2.0]                 # mostly -inf, a tie at the top
    x[4] = np.random.default_rng(2).standard_normal(V)
    x[4, 100:200] = -np.inf
    x[5] = 0.5
    x[5, 4999] = 0.75                                      # maximum in the very last element
    if dtype == "bf16":
        x = workloads.round_to_bf16(x)                     # both sides see the stored values
    ids, logp, lse, st = _run(x, 16, dtype)
    assert st == 0
    _check_rows(x, 16, ids, logp, lse, range(6))


@pytest.mark.parametrize("dtype,rows,V", [("bf16", 4, 151936), ("bf16", 512, 151936),
                                          ("bf16", 3, 151937), ("f32", 6, 151937)])
def test_full_width_tie_rows(dtype, rows, V):
    """Vocabulary-wide runs of equal values: the K lowest ids among the tied maxima win,
    on rows split over several CTAs (few rows) and on one CTA per row (512 rows), and with
    rows that start off a 16-byte boundary (V odd), whose scalar head holds the lowest
    ids and scalar tail the highest."""
    K = 8
    rng = np.random.default_rng(rows + V)
    x = (rng.standard_normal((rows, V)) * 3).astype(np.float32)
    special = [
        np.full(V, 0.5, np.float32),                                    # all equal
        np.where(np.arange(V) % 3 == 0, 0.0, -0.0).astype(np.float32),  # -0 == +0
        (np.arange(V) % 7).astype(np.float32),                          # 21,706 tied maxima
        np.round(rng.standard_normal(V) * 8) * 0.25,                    # quantised
        np.full(V, -1.0, np.float32),                                   # maximum at the end
        np.full(V, 2.0, np.float32),                                    # minimum at the start
    ]
    special[1][V // 2] = -1.0
    special[4][-1] = 1.0
    special[5][0] = 1.0
    for r in range(min(rows, len(special))):
        x[r] = special[r]
    if dtype == "bf16":
        x = workloads.round_to_bf16(x)
    ids, logp, lse, st = _run(x, K, dtype)
    assert st == 0
    _check_rows(x, K, ids, logp, lse, list(range(min(rows, len(special)))) +
                list(range(len(special), rows, 50)))


@pytest.mark.parametrize("bad", ["nan", "all_minus_inf", "plus_inf"])
def test_nonfinite_rows_set_device_status(bad):
    x = np.random.default_rng(0).standard_normal((4, 3000)).astype(np.float32)
    if bad == "nan":
        x[2, 5] = np.nan
    elif bad == "all_minus_inf":
        x[1] = -np.inf
    else:
        x[3, 7] = np.inf
    _, _, _, st = _run(x, 4, "f32")
    assert st == 5
    ids, logp, lse, st2 = _run(np.zeros((2, 10), np.float32), 3, "f32")
    assert st2 == 0


def test_workspace_reuse_and_split_path_repeatable():
    ll = _ll()
    rng = np.random.default_rng(9)
    x = to_dev(workloads.round_to_bf16(rng.standard_normal((16, 151936)).astype(np.float32)), "bf16")
    ws = ll.Workspace(ll.lib().lilicorr_topk_lse_workspace_bytes(16, 151936, 8))
    outs = [ll.topk_lse(x, 8, ws=ws) for _ in range(5)]
    torch.cuda.synchronize()
    for o in outs[1:]:
        assert torch.equal(o[0], outs[0][0]) and torch.equal(o[2], outs[0][2])
    assert ws.status() == 0
