"""Failure detection on the GPU without a fault: a bounded device wait is made to run
out, and the expiry must come back to the host as HERO_ERR_TIMEOUT while the
context stays usable.

The tensor-core GEMM's epilogue warps wait (bounded) for the accumulator of their
tile.  With a single 128 x 256 tile and K = 131072 that accumulation takes well over
a hundred microseconds, so with the wait bound lowered to 1 microsecond the wait
gives up long before the tile is ready; the kernel then lets its copies and MMAs in
flight finish (their own fixed bound), records the expiry and returns.  Every wait
of the kernel is bounded, so nothing here can wait forever.  The bound is restored
and the same GEMM must then run normally and correctly.
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


def test_expired_wait_reports_timeout_then_recovers(hero):
    import torch
    M, N, K = 128, 256, 131072
    g = torch.Generator(device="cuda").manual_seed(7)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
    B = torch.randn(N, K, device="cuda", generator=g).to(torch.bfloat16)
    C = torch.zeros(M, N, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    hero.hero_set_wait_limit_ns(1000)
    try:
        with pytest.raises(hero.HeroError) as e:
            hero.hero_gemm_bf16_check(A.data_ptr(), B.data_ptr(), C.data_ptr(), M, N, K, st)
        assert e.value.status == hero.HERO_ERR_TIMEOUT
        assert "wait" in str(e.value)
    finally:
        hero.hero_set_wait_limit_ns(0)
    torch.cuda.synchronize()          # no CUDA error: the context is intact
    C.fill_(float("nan"))
    hero.hero_gemm_bf16_check(A.data_ptr(), B.data_ptr(), C.data_ptr(), M, N, K, st)
    ref = A.double() @ B.double().T
    err = (C.double() - ref).abs().max().item()
    assert err <= 1e-5 * K ** 0.5 * ref.abs().max().item() + 1e-6, err
    # the error word was cleared by the failing call's report
    A1, B1 = A[:, :64].contiguous(), B[:, :64].contiguous()
    hero.hero_gemm_bf16_check(A1.data_ptr(), B1.data_ptr(), C.data_ptr(), M, N, 64, st)
