"""GPU parity of the fused path lilicorr_select_block (steps 1-4) on every sequence of
every workload: top-K ids bit-exact, log-probs within 1e-3, pair scores within the vector
tolerance, and the chosen path checked step by step against the oracle's scores (equal up
to the first tied step, every step a valid greedy choice). The oracle runs on the host
cores in a process pool."""
import numpy as np
import pytest
import torch

import _oracle_pool
import workloads
from _helpers import TOL_LOGP, TOL_VEC, check_path, to_dev, workload_data

pytestmark = pytest.mark.gpu


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _gpu_select(ll, head, wl, inp):
    """One select_block call over the batch in ``inp``; tokens and intermediates."""
    B = inp["logits"].shape[0]
    ws = head.workspace(B)
    tokens = ll.select_block(head, to_dev(inp["logits"], wl.dtype), to_dev(inp["hidden"], wl.dtype),
                             to_dev(inp["target"], wl.dtype), ws=ws)
    torch.cuda.synchronize()
    assert ws.status() == 0
    inter = {k: v.cpu().numpy() for k, v in ll.select_block_intermediates(head, B, ws).items()}
    return tokens.cpu().numpy(), inter


def check_against_oracle(wl, tokens, inter, refs):
    """Compare every sequence of a GPU selection with the oracle's; returns path stats."""
    tol = TOL_VEC[wl.dtype]
    stats = {"sequences": 0, "slots": 0, "prefix": 0, "exact": 0, "ties": 0}
    for b, r in enumerate(refs):
        assert np.array_equal(inter["ids"][b], r["ids"]), f"sequence {b}: top-K ids differ"
        assert np.abs(inter["logp"][b] - r["logp"]).max() <= TOL_LOGP
        assert np.abs(inter["lse"][b] - r["lse"]).max() <= TOL_LOGP
        assert np.abs(inter["A"][b] - r["A"]).max() <= tol, b
        assert np.abs(inter["P"][b] - r["P"]).max() <= tol, b
        pc = check_path(inter["choice"][b], r["A"], r["P"], tol)
        assert np.array_equal(tokens[b, :pc.prefix], r["tokens"][:pc.prefix])
        if pc.ties == 0:
            assert pc.prefix == wl.L and np.array_equal(tokens[b], r["tokens"])
        assert np.array_equal(tokens[b], inter["ids"][b][np.arange(wl.L), inter["choice"][b]])
        stats["sequences"] += 1
        stats["slots"] += wl.L
        stats["prefix"] += pc.prefix
        stats["exact"] += pc.exact
        stats["ties"] += pc.ties
    return stats


def select_and_check(wl, inp, seeds, tier=0, embed_std=workloads.WEIGHT_STD):
    """select_block over the batch ``inp`` (sequence b drawn from seeds[b]) against the
    oracle's selection of every sequence."""
    ll = _ll()
    W = workloads.head_weights(wl)
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype, std=embed_std))
    try:
        tokens, inter = _gpu_select(ll, head, wl, inp)
    finally:
        head.close()
    refs = _oracle_pool.select(wl, seeds, tier, embed_std=embed_std)
    stats = check_against_oracle(wl, tokens, inter, refs)
    print(f"{wl.name} tier {tier} embed std {embed_std}: {stats}")
    return stats


def select_blocks_and_check(wl, seeds, embed_std=workloads.WEIGHT_STD):
    """Batch-1 calls, one per block seed (the launch of the batch-1 selection)."""
    ll = _ll()
    W = workloads.head_weights(wl)
    head = ll.Head.from_workload(wl, W, workloads.embed_table(wl.V, wl.H, wl.dtype, std=embed_std))
    toks, inters = [], []
    try:
        for s in seeds:
            t, it = _gpu_select(ll, head, wl, workloads.batch_inputs(wl, [s]))
            toks.append(t[0])
            inters.append(it)
    finally:
        head.close()
    inter = {k: np.stack([it[k][0] for it in inters]) for k in inters[0]}
    refs = _oracle_pool.select(wl, seeds, embed_std=embed_std)
    stats = check_against_oracle(wl, np.stack(toks), inter, refs)
    print(f"{wl.name} {len(seeds)} blocks, embed std {embed_std}: {stats}")
    return stats


def test_tiny_f32_select():
    wl, _, inp = workload_data("tiny_f32")
    st = select_and_check(wl, inp, wl.seeds())
    assert st["exact"] >= 4          # fp32: few ties under 1e-5


def test_single_request_blocks():
    wl = workloads.WORKLOADS["single_request"]
    select_blocks_and_check(wl, wl.block_seeds()[:100])


@pytest.mark.parametrize("name,tier", [("serving_b32", 0), ("entropy_tiers_b64", 0),
                                       ("entropy_tiers_b64", 1), ("entropy_tiers_b64", 2),
                                       ("ties_b256", 0)])
def test_batched_workloads_every_sequence(name, tier):
    wl, _, inp = workload_data(name, tier)
    select_and_check(wl, inp, wl.seeds(tier), tier)
