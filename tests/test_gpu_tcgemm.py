"""The tensor-core GEMM (tcgen05.mma, TMEM accumulators, 128-byte swizzled operand tiles)
through mcd_tc_gemm against torch on the same device tensors: exact on small-integer
operands (every product and partial sum is an integer below 2^24, so any misplaced
element, swizzle error or dropped k-slice changes the result), and within fp32
accumulation-order rounding on Gaussian bf16 operands at the batched path's shapes."""
import pytest
import torch

from paper_2609_37007_gb300 import mcd

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _run(M, N, K, bn, A, B):
    Y = torch.full((N, M), float("nan"), dtype=torch.float32, device=DEV)
    mcd.mcd_tc_gemm(M, N, K, bn, A.view(torch.int16), B.view(torch.int16), Y)
    return Y


@pytest.mark.parametrize("M,N,K,bn", [(128, 128, 64, 128), (128, 256, 128, 256), (256, 128, 512, 128),
                                      (1024, 512, 1024, 256)])
def test_tc_gemm_exact_on_integers(M, N, K, bn):
    g = torch.Generator(device=DEV).manual_seed(M + N + K)
    A = torch.randint(-3, 4, (M, K), generator=g, device=DEV).to(torch.bfloat16)
    B = torch.randint(-3, 4, (N, K), generator=g, device=DEV).to(torch.bfloat16)
    Y = _run(M, N, K, bn, A, B)
    ref = B.double() @ A.double().T
    assert torch.equal(Y.double(), ref)


@pytest.mark.parametrize("M,N,K,bn", [(6144, 512, 1024, 128), (4096, 512, 1024, 256), (1024, 512, 3072, 128),
                                      (2048, 128, 1024, 128), (6144, 512, 1024, 0), (1024, 3072, 1024, 0)])
def test_tc_gemm_gaussian(M, N, K, bn):
    g = torch.Generator(device=DEV).manual_seed(7 * M + N + K)
    A = (0.02 * torch.randn(M, K, generator=g, device=DEV)).to(torch.bfloat16)
    B = torch.randn(N, K, generator=g, device=DEV).to(torch.bfloat16)
    Y = _run(M, N, K, bn, A, B)
    ref = B.double() @ A.double().T
    err = (Y.double() - ref).abs().max().item()
    assert err <= 1e-5 * ref.abs().max().item() * (K / 1024) ** 0.5 * 10, err


def test_tc_gemm_rejects_shapes():
    A = torch.zeros((128, 64), dtype=torch.int16, device=DEV)
    with pytest.raises(RuntimeError):
        mcd.mcd_tc_gemm(100, 128, 64, 128, A, A, A)     # M not a multiple of 128
    with pytest.raises(RuntimeError):
        mcd.mcd_tc_gemm(128, 128, 48, 128, A, A, A)     # K not a multiple of 64
    with pytest.raises(RuntimeError):
        mcd.mcd_tc_gemm(128, 128, 64, 64, A, A, A)      # unsupported tile width


@pytest.mark.parametrize("M,N,K,bn", [(6144, 512, 1024, 128), (6144, 512, 1024, 256), (6144, 512, 1024, 0),
                                      (256, 256, 192, 256), (384, 208, 128, 0)])
def test_tc_gemm_tiled_equals_one_call_form(M, N, K, bn):
    """Tile once, multiply twice through the asynchronous entry: bit-identical to the
    one-call form and exact on small-integer operands."""
    g = torch.Generator(device=DEV).manual_seed(3 * M + N + K)
    A = torch.randint(-3, 4, (M, K), generator=g, device=DEV).to(torch.bfloat16)
    B = torch.randint(-3, 4, (N, K), generator=g, device=DEV).to(torch.bfloat16)
    ta = torch.empty(M * K * 2 + 1024, dtype=torch.uint8, device=DEV)
    tb = torch.empty(N * K * 2 + 1024, dtype=torch.uint8, device=DEV)
    ta = ta[(-ta.data_ptr()) % 1024:][:M * K * 2]
    tb = tb[(-tb.data_ptr()) % 1024:][:N * K * 2]
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    mcd.mcd_tc_tile(M, K, A.view(torch.int16), ta)
    mcd.mcd_tc_tile(N, K, B.view(torch.int16), tb)
    ys = []
    for _ in range(2):
        Y = torch.full((N, M), float("nan"), dtype=torch.float32, device=DEV)
        mcd.mcd_tc_gemm_tiled(M, N, K, bn, ta, tb, Y, err)
        ys.append(Y)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    ref = B.double() @ A.double().T
    assert torch.equal(ys[0].double(), ref) and torch.equal(ys[1], ys[0])
    assert torch.equal(ys[0], _run(M, N, K, bn, A, B))
