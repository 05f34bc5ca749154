"""CPU checks of the seeded input generators shared by the oracle and the GPU tests: they
hold none of the method's arithmetic, only the draws and the bf16 storage rounding, so
they are checked against torch's own bf16 conversion and against the recipe each
workload states (planted boosts, a 0.25 grid with ties, Gumbel tiers, chunked embedding
rows that regenerate the table)."""
import numpy as np
import torch

import workloads
from workloads import Workload


def _small(kind, param, dtype="bf16", tiers=()):
    return Workload("t_" + kind, B=3, L=4, V=3000, K=4, d=64, H=32, dtype=dtype,
                    logit_kind=kind, logit_param=param, seed_base=77, tiers=tiers)


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    a = np.concatenate([rng.standard_normal(4096).astype(np.float32) * 50,
                        np.array([0.0, -0.0, 1.0 + 2.0**-8, 1.0 + 3 * 2.0**-8, -1.0 - 2.0**-8,
                                  3.3895314e38, 1e-40], np.float32)])  # ties to even, subnormal
    want = torch.from_numpy(a).to(torch.bfloat16).float().numpy()
    got = workloads.round_to_bf16(a)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
    assert np.array_equal(workloads.bf16_bits_to_f32(workloads.bf16_bits(got)), got)


def test_draws_are_seeded_and_stored_exactly():
    wl = _small("scaled_normal", (1.0, 5.0))
    a, b = workloads.sequence_inputs(wl, 5), workloads.sequence_inputs(wl, 5)
    c = workloads.sequence_inputs(wl, 6)
    for k in ("logits", "hidden", "target"):
        assert np.array_equal(a[k], b[k]) and not np.array_equal(a[k], c[k])
        assert np.array_equal(workloads.round_to_bf16(a[k]), a[k])     # exact in bf16
    assert a["logits"].shape == (4, 3000) and a["hidden"].shape == (4, 32)
    assert a["target"].shape == (wl.n_tgt, 32)
    bi = workloads.batch_inputs(wl, [5, 6])
    assert np.array_equal(bi["logits"][0], a["logits"]) and np.array_equal(bi["logits"][1],
                                                                           c["logits"])


def test_logit_recipes():
    wl = _small("normal_planted", (2.0, 6.0), dtype="f32")
    inp = workloads.sequence_inputs(wl, 1)
    p = inp["planted"]
    assert p.shape == (4,) and ((0 <= p) & (p < 3000)).all()
    x = inp["logits"]
    # the boost lifts the planted entry well above the row's typical values
    assert (x[np.arange(4), p] > np.median(x, axis=1) + 3.0).all()

    q = workloads.sequence_inputs(_small("quantised_normal", (2.0, 0.25)), 1)["logits"]
    assert np.array_equal(q / 0.25, np.round(q / 0.25))                # on the 0.25 grid
    assert len(np.unique(q[0])) < 200                                  # many ties per row

    g = _small("gumbel", (), tiers=(0.3, 1.0, 3.0))
    s = [workloads.sequence_inputs(g, seed, tier=t)["logits"].std()
         for t, seed in enumerate(g.seeds(0)[:1] + g.seeds(1)[:1] + g.seeds(2)[:1])]
    assert s[0] > s[1] > s[2]                                          # 1/tau scales the noise
    assert g.seeds(1)[0] == 77 + 100


def test_embedding_rows_regenerate_the_table():
    V, H = 5000, 16                                                    # three chunks
    workloads._EMBED_CACHE.clear()
    ids = np.array([0, 2047, 2048, 4999, 17, 4096])
    rows = workloads.embed_rows(V, H, "bf16", ids)                     # regenerated per chunk
    table = workloads.embed_table(V, H, "bf16")
    assert np.array_equal(rows, workloads.bf16_bits_to_f32(table[ids]))
    assert np.array_equal(workloads.embed_rows(V, H, "bf16", ids), rows)   # from the cache
    assert abs(float(workloads.bf16_bits_to_f32(table).std()) - 0.02) < 1e-3
    workloads._EMBED_CACHE.clear()
