"""The tensor-core shared-memory layouts of the attention kernel, checked on
one 128 x N x 128 bf16 product against a plain fp32 matrix product.

mode 0: both operands K-major, loaded by TMA (S^T = K Q^T in the kernel)
mode 1: both operands M/N-major; A loaded by TMA, B written by threads in
        the probability-tile layout (O^T += V^T P^T in the kernel)
mode 2: as mode 1 with a 64-wide A (head dim 64): rows 64..127 repeat 0..63
mode 3: A (hi + lo) from tensor memory, B M/N-major (the row-layout kernel's PV)
"""
import pytest
import torch

pytestmark = pytest.mark.gpu


def _rand(shape, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(shape, generator=g).to(torch.bfloat16)


@pytest.mark.parametrize("N", [32, 64, 128, 256])
def test_kmajor_operands(cuda_device, N):
    from paper_2405_18628_gb300 import ppd
    a = _rand((128, 128), 1)
    b = _rand((N, 128), 2)
    d = torch.full((128, N), float("nan"), device=cuda_device)
    ppd.ppd_selftest_umma(a.to(cuda_device), b.to(cuda_device), d, 0, N)
    torch.cuda.synchronize()
    ref = a.float() @ b.float().T
    torch.testing.assert_close(d.cpu(), ref, rtol=1e-4, atol=1e-3)


@pytest.mark.parametrize("N", [32, 64, 128, 192, 256])
def test_mn_major_operands(cuda_device, N):
    from paper_2405_18628_gb300 import ppd
    a = _rand((128, 128), 3)     # [K][M]
    b = _rand((128, N), 4)       # [K][N]
    d = torch.full((128, N), float("nan"), device=cuda_device)
    ppd.ppd_selftest_umma(a.to(cuda_device), b.to(cuda_device), d, 1, N)
    torch.cuda.synchronize()
    ref = a.float().T @ b.float()
    torch.testing.assert_close(d.cpu(), ref, rtol=1e-4, atol=1e-3)


def test_mn_major_half_width(cuda_device):
    from paper_2405_18628_gb300 import ppd
    N = 64
    a = _rand((128, 64), 5)      # [K][M=64]
    b = _rand((128, N), 6)
    d = torch.full((128, N), float("nan"), device=cuda_device)
    ppd.ppd_selftest_umma(a.to(cuda_device), b.to(cuda_device), d, 2, N)
    torch.cuda.synchronize()
    ref = a.float().T @ b.float()
    torch.testing.assert_close(d.cpu()[:64], ref, rtol=1e-4, atol=1e-3)
    torch.testing.assert_close(d.cpu()[64:], ref, rtol=1e-4, atol=1e-3)



@pytest.mark.parametrize("N", [64, 128])
def test_tmem_a_operand_hi_lo(cuda_device, N):
    """mode 3: A = hi + lo from tensor memory (two products per 16 keys), B M/N-major."""
    from paper_2405_18628_gb300 import ppd
    a_hi = _rand((128, 128), 7)
    a_lo = (_rand((128, 128), 8).float() * 2.0 ** -9).to(torch.bfloat16)
    b = _rand((128, N), 9)       # [K][N]
    d = torch.full((128, N), float("nan"), device=cuda_device)
    a = torch.cat([a_hi, a_lo], dim=1).contiguous()
    ppd.ppd_selftest_umma(a.to(cuda_device), b.to(cuda_device), d, 3, N)
    torch.cuda.synchronize()
    ref = a_hi.float() @ b.float() + a_lo.float() @ b.float()
    torch.testing.assert_close(d.cpu(), ref, rtol=1e-4, atol=1e-3)
