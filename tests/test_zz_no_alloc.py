"""The allocation-free split-K GEMM entry point (hero_gemm_bf16_splitk_noalloc).

Callers that must not allocate device memory at call time (a host framework that
owns all device memory through its own pool, a latency-critical loop where a
cudaMalloc would synchronise the device) use this entry point: its partial sums
live in a static device array.  Its output must match the regular tensor-core
GEMM entry point, hero_gemm_bf16_check, within the GEMM tests' tolerance, on two
calls in a row (the static scratch keeps the previous call's contents), and
requests beyond the static scratch must be refused with HERO_ERR_ARG.

This file is collected last so that a failure here does not hide other tests.
"""

import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hero():
    import torch
    assert torch.cuda.is_available()
    from paper_2609_08189_gb300 import build, hero as H
    build.build()
    H.load()
    return H


def _gemm_tol(ref, K):
    return 1e-5 * K ** 0.5 * ref.abs().max().item() + 1e-6


@pytest.mark.parametrize("M,N,K,splits", [(64, 4096, 14336, 8), (333, 512, 1024, 3),
                                          (1, 256, 320, 5), (128, 264, 4096, 1),
                                          (64, 256, 320, 4)])   # 5 K blocks over 4 slices
def test_noalloc_matches_allocating_gemm_twice(hero, M, N, K, splits):
    import torch
    st = torch.cuda.current_stream().cuda_stream
    for call in range(2):   # second call sees the first call's leftovers in the static scratch
        g = torch.Generator(device="cuda").manual_seed(1000 * call + M + N + K)
        A = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
        B = torch.randn(N, K, device="cuda", generator=g).to(torch.bfloat16)
        C_ref = torch.full((M, N), float("nan"), device="cuda")
        C_na = torch.full((M, N), float("nan"), device="cuda")
        hero.hero_gemm_bf16_check(A.data_ptr(), B.data_ptr(), C_ref.data_ptr(), M, N, K, st)
        hero.hero_gemm_bf16_splitk_noalloc(A.data_ptr(), B.data_ptr(), C_na.data_ptr(), M, N, K,
                                           splits, st)
        torch.cuda.synchronize()
        exact = A.double() @ B.double().T
        tol = _gemm_tol(exact, K)
        assert torch.isfinite(C_na).all()
        assert (C_na.double() - C_ref.double()).abs().max().item() <= 2 * tol
        assert (C_na.double() - exact).abs().max().item() <= tol
    # the static error word: no wait expired and no bad index in either call
    hero.hero_gemm_bf16_splitk_noalloc_status(st)


def test_noalloc_rejects_requests_beyond_the_static_scratch(hero):
    import torch
    A = torch.zeros(4096, 128, device="cuda", dtype=torch.bfloat16)
    B = torch.zeros(1024, 128, device="cuda", dtype=torch.bfloat16)
    C = torch.zeros(4096, 1024, device="cuda")
    with pytest.raises(hero.HeroError) as e:   # 2 * 4096 * 1024 > 4,194,304 partial sums
        hero.hero_gemm_bf16_splitk_noalloc(A.data_ptr(), B.data_ptr(), C.data_ptr(), 4096, 1024,
                                           128, 2)
    assert e.value.status == hero.HERO_ERR_ARG
    assert "static scratch" in str(e.value)
    with pytest.raises(hero.HeroError) as e:   # more slices than 64-wide K blocks
        hero.hero_gemm_bf16_splitk_noalloc(A.data_ptr(), B.data_ptr(), C.data_ptr(), 16, 1024,
                                           128, 3)
    assert e.value.status == hero.HERO_ERR_ARG
    # the same shape within the limit runs
    hero.hero_gemm_bf16_splitk_noalloc(A.data_ptr(), B.data_ptr(), C.data_ptr(), 4096, 1024, 128, 1)
    torch.cuda.synchronize()
    assert (C == 0).all()
