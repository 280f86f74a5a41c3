"""The tcgen05 GEMM against a plain PyTorch fp32 matmul of the same bf16
operands (GPU).

Shapes cover one tile, ragged M (rows past the end read zero and are not
stored), several N tiles and K slices, and the three epilogues. The result is
one bf16 rounding of an fp32 sum, so the bound is a few bf16 units of the
result's magnitude plus fp32 summation-order noise.
"""

import pytest
import torch

import paper_2502_01637_gb300 as scone
from gpu_cases import DEV

pytestmark = pytest.mark.gpu


def rand(shape, seed, scale=1.0):
    g = torch.Generator(device="cpu").manual_seed(seed)
    return (torch.randn(shape, generator=g) * scale).to(torch.bfloat16).to(DEV)


def close(got, want, what):
    err = (got.float() - want).abs()
    bound = 2.0 ** -7 * want.abs() + 1e-3 * want.abs().max()
    bad = (err > bound).sum().item()
    assert bad == 0, f"{what}: {bad} elements off, max err {err.max().item():.3e}"


VARIANTS = [1, 2]      # one SM per tile, SM pairs


@pytest.mark.parametrize("variant", VARIANTS)
@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (200, 256, 128), (129, 512, 2048),
                                   (1000, 768, 512), (4099, 1024, 256)])
def test_store(M, N, K, variant):
    A, B = rand((M, K), 1), rand((N, K), 2)
    C = torch.empty((M, N), dtype=torch.bfloat16, device=DEV)
    scone.scone_gemm_bf16(A, B, C, variant=variant)
    close(C, A.float() @ B.float().T, f"store {M}x{N}x{K} variant {variant}")


@pytest.mark.parametrize("variant", VARIANTS)
@pytest.mark.parametrize("M,N,K", [(77, 256, 64), (300, 512, 1024)])
def test_residual_in_place(M, N, K, variant):
    A, B = rand((M, K), 3), rand((N, K), 4)
    R = rand((M, N), 5, scale=4.0)
    want = R.float() + A.float() @ B.float().T
    scone.scone_gemm_bf16(A, B, R, R=R, epilogue=scone.SCONE_GEMM_RESIDUAL, variant=variant)
    close(R, want, "residual")


@pytest.mark.parametrize("variant", VARIANTS)
def test_swiglu_pairs(variant):
    M, N, K = 250, 512, 256
    A, B = rand((M, K), 6, 0.5), rand((N, K), 7, 0.1)
    C = torch.empty((M, N // 2), dtype=torch.bfloat16, device=DEV)
    scone.scone_gemm_bf16(A, B, C, epilogue=scone.SCONE_GEMM_SWIGLU, variant=variant)
    P = A.float() @ B.float().T                      # [M, N]
    P = P.view(M, N // 32, 2, 16)
    g, u = P[:, :, 0, :], P[:, :, 1, :]
    want = (torch.nn.functional.silu(g) * u).reshape(M, N // 2)
    close(C, want, "swiglu")


def test_rejects_bad_shapes():
    A, B = rand((128, 64), 1), rand((200, 64), 2)     # N not a multiple of 256
    C = torch.empty((128, 200), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(scone.SconeError):
        scone.scone_gemm_bf16(A, B, C)


@pytest.mark.parametrize("variant", VARIANTS)
@pytest.mark.parametrize("epilogue", [0, 1, 2])      # store, residual, SwiGLU
def test_rows_past_m_are_not_written(variant, epilogue):
    """The epilogue stores whole 32-row boxes; rows past M must stay untouched
    (the store clips them), for every epilogue and a ragged M."""
    M, N, K = 333, 512, 128
    A, B = rand((M, K), 8), rand((N, K), 9)
    ncol = N // 2 if epilogue == scone.SCONE_GEMM_SWIGLU else N
    full = torch.full((M + 64, ncol), 7.0, dtype=torch.bfloat16, device=DEV)
    C = full[:M]
    R = None
    if epilogue == scone.SCONE_GEMM_RESIDUAL:
        C.copy_(rand((M, ncol), 10))
        R = C
    want_tail = full[M:].clone()
    scone.scone_gemm_bf16(A, B, C, R=R, epilogue=epilogue, variant=variant)
    torch.cuda.synchronize()
    assert torch.equal(full[M:], want_tail)
