"""GPU check of lilicorr_topk_lse_noalloc, the top-K entry point for callers that cannot
allocate device memory (it keeps its scratch in a fixed array inside the library instead
of a caller workspace). Its outputs must match lilicorr_topk_lse on the same logits, on
two calls in a row (the second call must not see the first call's leftovers).

This file is named to be collected last, so a run that stops at the first failure has
already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

import workloads

pytestmark = pytest.mark.gpu

TOL = 1e-3   # log-probs and log-normaliser, as in the other top-K tests


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _logits(seed, rows, V, dtype):
    x = np.random.default_rng(seed).standard_normal((rows, V)).astype(np.float32) * 3
    if dtype == "bf16":
        x = workloads.round_to_bf16(x)
        return torch.from_numpy(x).to(torch.bfloat16).cuda()
    return torch.from_numpy(x).cuda()


@pytest.mark.parametrize("rows,V,K,dtype", [(16, 151936, 8, "bf16"), (512, 32000, 16, "bf16"),
                                            (37, 1001, 5, "f32")])
def test_noalloc_matches_workspace_call_twice(rows, V, K, dtype):
    ll = _ll()
    for call, seed in enumerate((rows + 1, rows + 2)):      # two calls in a row
        x = _logits(seed, rows, V, dtype)
        ids_ref, logp_ref, lse_ref = ll.topk_lse(x, K)
        ids, logp, lse = ll.topk_lse_noalloc(x, K)
        torch.cuda.synchronize()
        assert torch.equal(ids, ids_ref), f"call {call}: ids differ"
        assert (logp - logp_ref).abs().max().item() <= TOL
        assert (lse - lse_ref).abs().max().item() <= TOL


def test_noalloc_rejects_sizes_beyond_its_scratch():
    ll = _ll()
    lib = ll.lib()
    assert lib.lilicorr_topk_lse_noalloc_max_bytes() == 4 << 20
    x = torch.empty(1, dtype=torch.bfloat16, device="cuda")
    out = torch.empty(1, dtype=torch.int32, device="cuda")
    f = torch.empty(1, dtype=torch.float32, device="cuda")
    # 1e6 rows of 16 candidates need far more than 4 MiB of tickets and partials;
    # the call is rejected on the host before anything is enqueued
    st = lib.lilicorr_topk_lse_noalloc(x.data_ptr(), 1, 1_000_000, 151936, 16, out.data_ptr(),
                                       f.data_ptr(), f.data_ptr(),
                                       torch.cuda.current_stream().cuda_stream)
    assert st == 7


@pytest.mark.parametrize("bad", ["nan", "plus_inf", "all_minus_inf"])
def test_noalloc_nonfinite_row_has_nonfinite_lse(bad):
    """The status word of this entry point is not reported; a non-finite row shows as a
    non-finite lse instead (the other rows are unaffected)."""
    ll = _ll()
    x = np.random.default_rng(3).standard_normal((6, 4000)).astype(np.float32)
    if bad == "nan":
        x[2, 17] = np.nan
    elif bad == "plus_inf":
        x[2, 17] = np.inf
    else:
        x[2] = -np.inf
    t = torch.from_numpy(x).cuda()
    ids, logp, lse = ll.topk_lse_noalloc(t, 4)
    ids_ref, logp_ref, lse_ref = ll.topk_lse(t, 4)
    torch.cuda.synchronize()
    lse, lse_ref = lse.cpu().numpy(), lse_ref.cpu().numpy()
    assert not np.isfinite(lse[2])
    if bad == "all_minus_inf":
        assert lse[2] == -np.inf
    else:
        assert np.isnan(lse[2])
    ok = [0, 1, 3, 4, 5]
    assert np.isfinite(lse[ok]).all()
    assert np.abs(lse[ok] - lse_ref[ok]).max() <= TOL
    assert torch.equal(ids[ok], ids_ref[ok])
