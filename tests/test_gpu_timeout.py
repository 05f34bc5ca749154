"""The failure side of the bounded waits (the LILICORR_ERR_TIMEOUT status): the
tensor-core linear layer is launched with its copies withheld, so its MMA warp waits on a
barrier that nothing arrives on. With a short wait limit the kernel must give up, record
the timeout in the status word, free its tensor memory and return; the context must stay
usable, and the same layer without the hook must then compute correctly."""
import time

import pytest
import torch

pytestmark = pytest.mark.gpu

TIMEOUT = 6        # LILICORR_ERR_TIMEOUT


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


@pytest.mark.parametrize("M,N,Kd", [(256, 512, 512), (4096, 256, 256)])
def test_withheld_copies_time_out_and_the_context_survives(M, N, Kd):
    ll = _ll()
    g = torch.Generator(device="cuda").manual_seed(M + N)
    A = torch.randn((M, Kd), generator=g, device="cuda").to(torch.bfloat16)
    W = (0.05 * torch.randn((N, Kd), generator=g, device="cuda")).to(torch.bfloat16)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    ll.test_linear_timeout(A, W, 2_000_000, status)         # ~1 ms of SM cycles per wait
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert int(status.item()) == TIMEOUT
    assert dt < 5.0, f"the timed-out launch took {dt:.2f} s"
    # the context is usable and the kernel, run normally, is correct
    status.zero_()
    C = ll.test_linear(A, W, path=3, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    want = A.float() @ W.float().T
    assert (C - want).abs().max().item() <= 2e-4 * max(1.0, want.abs().max().item()) * (Kd / 256) ** 0.5
    # twice in a row: the timeout leaves nothing behind that a second one trips over
    ll.test_linear_timeout(A, W, 2_000_000, status)
    torch.cuda.synchronize()
    assert int(status.item()) == TIMEOUT


def test_timeout_hook_rejects_unbounded_limits():
    ll = _ll()
    A = torch.zeros((128, 64), device="cuda", dtype=torch.bfloat16)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for bad in (0, 10, 10**12):
        with pytest.raises(ll.LilicorrError):
            ll.test_linear_timeout(A, A, bad, status)
