"""Weight-streaming GEMM (sd2_gemm): tensor-core and CUDA-core kernels against the fp32 product
of the same bf16 operands (the matmul step of the oracle's decoder), for every epilogue."""
import pytest
import torch

import parity
from oracle import model as omodel
from paper_2511_09844_gb300 import sd2

pytestmark = pytest.mark.gpu

TOL = 1e-4   # fp32 accumulation in a different order; operands are exact bf16 values


def _operands(M, N, K, seed):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(M, K, generator=g).to(torch.bfloat16)
    w = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16)
    return x, w


SHAPES = [
    (1, 128, 64), (5, 256, 128), (6, 384, 4096), (16, 128, 960), (17, 1024, 256),
    (40, 512, 2048), (144, 256, 1024), (256, 128, 192), (300, 384, 512),
    (6, 128, 14336),      # one weight tile split across every CTA
    (2, 4096, 4096),      # the 8B O projection at drafter-step M
    (144, 28672, 256),    # wide token tiles, 224 whole tiles: two CTAs per SM, one tile each
    (256, 16384, 128),    # the widest token tile (256 columns), 128 whole tiles
]


@pytest.mark.parametrize("impl", [1, 2])
@pytest.mark.parametrize("M,N,K", SHAPES)
def test_store(impl, M, N, K):
    x, w = _operands(M, N, K, M * 7 + N + K)
    ref = x.float() @ w.float().T
    y = sd2.gemm(x.cuda(), w.cuda(), epilogue=0, impl=impl)
    torch.cuda.synchronize()
    assert parity.row_rel_err(y, ref) < TOL


@pytest.mark.parametrize("impl", [1, 2])
def test_residual_add_and_strided_rows(impl):
    M, N, K = 11, 640, 448
    x, w = _operands(M, N, K, 3)
    big = torch.zeros(M, K + 64, dtype=torch.bfloat16)
    big[:, :K] = x                                     # row stride larger than K
    out0 = torch.randn(M, N + 32)                      # output row stride larger than N
    out = out0.clone().cuda()
    sd2.gemm(big.cuda()[:, :K], w.cuda(), epilogue=1, out=out[:, :N], impl=impl)
    torch.cuda.synchronize()
    ref = out0.clone()
    ref[:, :N] += x.float() @ w.float().T
    assert parity.row_rel_err(out.cpu(), ref) < TOL
    assert torch.equal(out.cpu()[:, N:], out0[:, N:])


@pytest.mark.parametrize("impl", [1, 2])
@pytest.mark.parametrize("M,N,K", [(5, 640, 448), (2, 2048, 8192), (144, 256, 1024)])
def test_residual_add_with_sequence_bias(impl, M, N, K):
    """Residual add plus a per-sequence bias (the after-MLP steering site): out += Y + bias[seq[m]]."""
    x, w = _operands(M, N, K, 5 + M)
    g = torch.Generator().manual_seed(6)
    out0 = torch.randn(M, N, generator=g)
    bias = torch.randn(3, N, generator=g)
    seq = torch.randint(0, 3, (M,), generator=g).to(torch.int32)
    out = out0.clone().cuda()
    sd2.gemm(x.cuda(), w.cuda(), epilogue=1, out=out, bias=bias.cuda(), seq=seq.cuda(), impl=impl)
    torch.cuda.synchronize()
    ref = out0 + x.float() @ w.float().T + bias[seq.long()]
    assert parity.row_rel_err(out.cpu(), ref) < TOL


@pytest.mark.parametrize("impl", [1, 2])
@pytest.mark.parametrize("M,N,K", [(3, 128, 256), (16, 2048, 2048), (150, 384, 512)])
def test_silu_bias_epilogue(impl, M, N, K):
    """Epilogue 4: bf16(SiLU(Y + bias[seq[m]])) (the conditional bias MLP's hidden layer)."""
    x, w = _operands(M, N, K, 9 + M)
    g = torch.Generator().manual_seed(10)
    bias = torch.randn(2, N, generator=g)
    seq = torch.randint(0, 2, (M,), generator=g).to(torch.int32)
    h = sd2.gemm(x.cuda(), w.cuda(), epilogue=4, bias=bias.cuda(), seq=seq.cuda(), impl=impl)
    torch.cuda.synchronize()
    y = x.float() @ w.float().T + bias[seq.long()]
    ref = omodel.silu(y)
    assert parity.row_rel_err(h.float().cpu(), ref) < 1e-2   # bf16 output


@pytest.mark.parametrize("impl", [1, 2])
@pytest.mark.parametrize("M,F,K", [(6, 256, 512), (18, 192, 2048), (1, 64, 4864), (144, 14336, 512)])
def test_steered_swiglu_epilogue(impl, M, F, K):
    g = torch.Generator().manual_seed(M + F)
    x = torch.randn(M, K, generator=g).to(torch.bfloat16)
    wg = (torch.randn(F, K, generator=g) * 0.05).to(torch.bfloat16)
    wu = (torch.randn(F, K, generator=g) * 0.05).to(torch.bfloat16)
    bias = torch.randn(3, F, generator=g)
    seq = torch.tensor([i % 3 for i in range(M)], dtype=torch.int32)
    h = sd2.gemm(x.cuda(), wg.cuda(), epilogue=2, w_up=wu.cuda(), bias=bias.cuda(), seq=seq.cuda(), impl=impl)
    torch.cuda.synchronize()
    ref = omodel.steered_swiglu(x.float(), wg, wu, torch.eye(F), bias[seq.long()])
    assert parity.row_rel_err(h.float().cpu(), ref) < 1e-2     # bf16 output


def test_implementations_agree_and_repeat():
    M, N, K = 6, 1024, 4096
    x, w = _operands(M, N, K, 11)
    a = sd2.gemm(x.cuda(), w.cuda(), impl=1)
    b = sd2.gemm(x.cuda(), w.cuda(), impl=2)
    c = sd2.gemm(x.cuda(), w.cuda(), impl=2)
    torch.cuda.synchronize()
    assert parity.row_rel_err(a, b) < TOL
    assert torch.equal(b, c)          # the split-tile reduction runs in a fixed order
