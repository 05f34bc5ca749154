"""GPU check of the scoring network's linear-layer kernels (building blocks of step 2)
against a plain PyTorch fp32 matmul of the same bf16/fp32 operands: the tensor-core
(tcgen05) kernels (tiled, and one tile of rows with whole-K copies), the tiled and the
few-row CUDA-core kernels (one, four or sixteen rows per CTA), with bias, SiLU,
residual, bf16 output, ragged M/N and long Kd."""
import pytest
import torch

pytestmark = pytest.mark.gpu


def _ll():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll


def _ref(A, W, bias, residual, act):
    y = A.float() @ W.float().T
    if bias is not None:
        y = y + bias
    if act == 1:
        y = torch.nn.functional.silu(y)
    if residual is not None:
        y = y + residual
    return y


CASES = [  # M, N, Kd
    (128, 256, 256), (128, 64, 64), (300, 768, 256), (129, 64, 4096), (512, 512, 4096),
    (256, 1536, 512), (1000, 200, 512), (4096, 512, 512), (16, 256, 4096), (1, 256, 256),
    (64, 1024, 2048), (3, 264, 4096), (4, 256, 512), (5, 104, 256), (1, 8, 4096),
]


@pytest.mark.parametrize("M,N,Kd", CASES)
@pytest.mark.parametrize("path", [0, 1, 2, 3])
def test_linear_paths(M, N, Kd, path):
    ll = _ll()
    if path == 2 and M > 64:
        pytest.skip("few-row kernel serves M <= 64")
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N + Kd)
    A = torch.randn((M, Kd), generator=g, device="cuda").to(torch.bfloat16)
    W = (0.02 * torch.randn((N, Kd), generator=g, device="cuda")).to(torch.bfloat16)
    bias = 0.1 * torch.randn(N, generator=g, device="cuda")
    res = torch.randn((M, N), generator=g, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for act, b, r, odt in [(0, None, None, torch.float32), (1, bias, None, torch.float32),
                           (0, bias, res, torch.float32), (1, bias, None, torch.bfloat16)]:
        C = ll.test_linear(A, W, odt, bias=b, residual=r, act=act, path=path, status=status)
        torch.cuda.synchronize()
        want = _ref(A, W, b, r, act)
        tol = 2e-2 if odt == torch.bfloat16 else 2e-4 * max(1.0, (Kd / 256) ** 0.5)
        err = (C.float() - want).abs().max().item()
        assert err <= tol * max(1.0, want.abs().max().item()), (path, act, odt, err)
    assert int(status.item()) == 0


def test_linear_fp32_operands_use_cuda_cores():
    ll = _ll()
    A = torch.randn((200, 96), device="cuda")
    W = torch.randn((72, 96), device="cuda")
    with pytest.raises(ll.LilicorrError):
        ll.test_linear(A, W, path=3)
    C = ll.test_linear(A, W, path=0)
    assert (C - A @ W.T).abs().max().item() < 1e-4


SMALL_CASES = [  # M, N, Kd: one tile of rows, whole-K copies
    (128, 256, 256), (128, 768, 256), (128, 512, 512), (100, 256, 512), (65, 64, 64),
    (1, 32, 128), (128, 1024, 256), (77, 192, 320),
]


@pytest.mark.parametrize("M,N,Kd", SMALL_CASES)
def test_linear_one_row_tile(M, N, Kd):
    ll = _ll()
    g = torch.Generator(device="cuda").manual_seed(M * 5 + N + Kd)
    A = torch.randn((M, Kd), generator=g, device="cuda").to(torch.bfloat16)
    W = (0.02 * torch.randn((N, Kd), generator=g, device="cuda")).to(torch.bfloat16)
    bias = 0.1 * torch.randn(N, generator=g, device="cuda")
    res = torch.randn((M, N), generator=g, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    combos = [(0, None, None, torch.float32), (1, bias, None, torch.float32),
              (0, bias, res, torch.float32)]
    if N % 64 == 0:
        combos.append((1, bias, None, torch.bfloat16))
    for act, b, r, odt in combos:
        C = ll.test_linear(A, W, odt, bias=b, residual=r, act=act, path=4, status=status)
        torch.cuda.synchronize()
        want = _ref(A, W, b, r, act)
        tol = 2e-2 if odt == torch.bfloat16 else 2e-4 * max(1.0, (Kd / 256) ** 0.5)
        err = (C.float() - want).abs().max().item()
        assert err <= tol * max(1.0, want.abs().max().item()), (act, odt, err)
    assert int(status.item()) == 0


def test_linear_one_row_tile_rejects_other_shapes():
    ll = _ll()
    A = torch.randn((129, 256), device="cuda").to(torch.bfloat16)
    W = torch.randn((256, 256), device="cuda").to(torch.bfloat16)
    with pytest.raises(ll.LilicorrError):
        ll.test_linear(A, W, path=4)                        # more than one tile of rows
    A = torch.randn((128, 1024), device="cuda").to(torch.bfloat16)
    W = torch.randn((256, 1024), device="cuda").to(torch.bfloat16)
    with pytest.raises(ll.LilicorrError):
        ll.test_linear(A, W, path=4)                        # Kd above 512


ROW_CASES = [  # M, N, Kd: fp32 activations at per-sequence row counts
    (256, 512, 512), (65, 40, 1032), (1000, 200, 512), (1024, 512, 256), (17, 8, 8),
    (300, 96, 2048),
]


@pytest.mark.parametrize("M,N,Kd", ROW_CASES)
@pytest.mark.parametrize("wdt", [torch.bfloat16, torch.float32])
def test_linear_fp32_rows(M, N, Kd, wdt):
    """The row-block kernel (path 5) and the network's own choice for fp32 activations with
    more than 64 rows, against fp32 PyTorch: bias, SiLU, residual, bf16 output, ragged M and
    N, Kd over several staged chunks."""
    ll = _ll()
    g = torch.Generator(device="cuda").manual_seed(M * 3 + N + Kd)
    A = torch.randn((M, Kd), generator=g, device="cuda")
    W = (0.05 * torch.randn((N, Kd), generator=g, device="cuda")).to(wdt)
    bias = 0.1 * torch.randn(N, generator=g, device="cuda")
    res = torch.randn((M, N), generator=g, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for path in (5, 0) if M > 64 else (5,):
        for act, b, r, odt in [(0, None, None, torch.float32), (1, bias, None, torch.float32),
                               (0, bias, res, torch.float32), (1, bias, None, torch.bfloat16)]:
            C = ll.test_linear(A, W, odt, bias=b, residual=r, act=act, path=path, status=status)
            torch.cuda.synchronize()
            want = _ref(A, W, b, r, act)
            tol = 2e-2 if odt == torch.bfloat16 else 2e-5 * max(1.0, (Kd / 256) ** 0.5)
            err = (C.float() - want).abs().max().item()
            assert err <= tol * max(1.0, want.abs().max().item()), (path, act, odt, err)
    assert int(status.item()) == 0


def test_linear_fp32_rows_rejects_unaligned():
    ll = _ll()
    W = torch.randn((32, 96), device="cuda")
    A = torch.randn((80, 102), device="cuda")[:, :96]     # row stride 102: not 16-byte rows
    with pytest.raises(ll.LilicorrError):
        ll.test_linear(A, W, path=5)
    A = torch.randn((80, 100), device="cuda")
    with pytest.raises(ll.LilicorrError):
        ll.test_linear(A, torch.randn((32, 100), device="cuda"), path=5)   # Kd not a multiple of 8
    A = torch.randn((80, 102), device="cuda")[:, :96]
    C = ll.test_linear(A, W, path=0)                      # the network's choice falls back
    torch.cuda.synchronize()
    assert (C - A @ W.T).abs().max().item() < 1e-4
