"""CPU pins of the vocabulary-sharded step (1): shard summaries merged in any order give
exactly the whole-row top-K and log-normaliser, and the host side of the sharded path
(shard bounds, the public record layout, the all-gather) on two gloo ranks."""
import os

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2608_20530_gb300 import shards


def _row(V, seed, quant=None):
    rng = np.random.default_rng(seed)
    x = rng.normal(0.0, 2.0, V)
    if quant:
        x = np.round(x / quant) * quant              # many ties across shard borders
    return x


@pytest.mark.parametrize("V,K,P,quant", [(1000, 8, 2, None), (1000, 8, 7, None),
                                         (4096, 16, 4, 0.25), (97, 4, 5, 0.5),
                                         (50, 32, 3, None)])
def test_merged_shards_equal_the_whole_row(V, K, P, quant):
    x = _row(V, V + K + P, quant)
    ids, logp, lse = oracle.topk_lse(x, K)
    parts = [oracle.topk_lse_partial(x[a:b], K, a) for a, b in shards.bounds(V, P)]
    mids, mlogp, mlse = oracle.merge_partials(parts, K)
    assert np.array_equal(mids, ids)
    assert abs(mlse - lse) <= 1e-12 * max(1.0, abs(lse))
    assert np.allclose(mlogp, logp, rtol=0, atol=1e-12)
    # the order of the shards does not matter
    r = oracle.merge_partials(parts[::-1], K)
    assert np.array_equal(r[0], ids) and abs(r[2] - lse) <= 1e-12 * max(1.0, abs(lse))


def test_ties_across_shards_go_to_the_lower_id():
    x = np.zeros(12)
    x[[2, 5, 9, 11]] = 3.0                             # four equal maxima in three shards
    parts = [oracle.topk_lse_partial(x[a:b], 3, a) for a, b in [(0, 4), (4, 8), (8, 12)]]
    ids, _, _ = oracle.merge_partials(parts, 3)
    assert list(ids) == [2, 5, 9]


def test_narrow_and_empty_shards():
    x = _row(40, 3)
    x[10:20] = -np.inf                                 # a shard that holds only -inf
    ids, _, lse = oracle.topk_lse(x, 8)
    b = [(0, 3), (3, 10), (10, 20), (20, 40)]
    parts = [oracle.topk_lse_partial(x[a:e], 8, a) for a, e in b]
    assert parts[2][0] == -np.inf and parts[2][1] == 0.0 and (parts[2][3] >= 10).all()
    assert (parts[0][3][3:] == -1).all()              # 3 columns: padded to K
    mids, _, mlse = oracle.merge_partials(parts, 8)
    assert np.array_equal(mids, ids) and abs(mlse - lse) < 1e-12


def test_single_shard_is_the_identity():
    x = _row(300, 5)
    ids, logp, lse = oracle.topk_lse(x, 8)
    mids, mlogp, mlse = oracle.merge_partials([oracle.topk_lse_partial(x, 8, 0)], 8)
    assert np.array_equal(mids, ids) and np.allclose(mlogp, logp) and abs(mlse - lse) < 1e-12


def test_bounds_cover_the_vocabulary():
    for V, P in [(151936, 8), (10, 3), (7, 7), (5, 1)]:
        b = shards.bounds(V, P)
        assert b[0][0] == 0 and b[-1][1] == V and len(b) == P
        assert all(b[i][1] == b[i + 1][0] for i in range(P - 1))
        assert max(e - a for a, e in b) - min(e - a for a, e in b) <= 1
    with pytest.raises(ValueError):
        shards.bounds(3, 4)


def test_record_layout_round_trip():
    rng = np.random.default_rng(2)
    K, rows = 8, 5
    m = rng.normal(size=rows).astype(np.float32)
    s = rng.uniform(1, 2, rows).astype(np.float32)
    vals = np.sort(rng.normal(size=(rows, K)).astype(np.float32), axis=1)[:, ::-1]
    ids = rng.integers(0, 1000, (rows, K)).astype(np.int32)
    rec = shards.pack_records(m, s, vals, ids)
    assert rec.dtype == torch.uint8 and tuple(rec.shape) == (rows, 8 + 8 * K)
    m2, s2, v2, i2 = shards.unpack_records(rec, K)
    assert np.array_equal(m2, m) and np.array_equal(s2, s)
    assert np.array_equal(v2, vals) and np.array_equal(i2, ids)


def _rank(rank, world, port, V, K, rows, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        x = np.stack([_row(V, 100 + r) for r in range(rows)])
        a, b = shards.bounds(V, world)[rank]
        parts = [oracle.topk_lse_partial(x[r, a:b], K, a) for r in range(rows)]
        rec = shards.pack_records(np.array([p[0] for p in parts], np.float32),
                                  np.array([p[1] for p in parts], np.float32),
                                  np.stack([p[2] for p in parts]).astype(np.float32),
                                  np.stack([p[3] for p in parts]).astype(np.int32))
        allrec = shards.gather_records(rec)           # [world, rows, bytes], shard order
        out = []
        for r in range(rows):
            per = []
            for p in range(world):
                m, s, v, i = shards.unpack_records(allrec[p, r:r + 1], K)
                per.append((float(m[0]), float(s[0]), v[0].astype(np.float64), i[0].astype(np.int64)))
            out.append(oracle.merge_partials(per, K))
        for r in range(rows):
            ids, _, lse = oracle.topk_lse(x[r], K)
            assert np.array_equal(out[r][0], ids)
            assert abs(out[r][2] - lse) <= 1e-5 * max(1.0, abs(lse))   # records hold fp32
        q.put((rank, "ok"))
    except Exception as e:                            # reported to the parent
        q.put((rank, repr(e)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_gather_and_merge():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + os.getpid() % 1000
    procs = [ctx.Process(target=_rank, args=(r, 2, port, 5000, 8, 3, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
    assert res == {0: "ok", 1: "ok"}, res
