"""A bounded wait inside a kernel runs out without faulting or hanging the GPU (failure detection).

zl_wait_selftest runs the mbarrier wait that every tcgen05 kernel uses on a barrier that nothing
arrives at. The wait must give up after its limit (about 2 s of SM clock), report ZL_DEVERR_TIMEOUT
through the error word, and leave the device usable: a GEMM right after it gives the right result.
"""
import time

import pytest
import torch

pytestmark = pytest.mark.gpu


def test_expired_wait_reports_timeout_and_the_context_stays_usable():
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300 import binding as b
    t0 = time.perf_counter()
    bits = b.zl_wait_selftest()
    dt = time.perf_counter() - t0
    assert bits == b.ZL_DEVERR_TIMEOUT, bits
    assert 0.5 <= dt <= 60.0, dt                # the wait ran to its limit, and that limit is bounded
    a = torch.randn(256, 128, device="cuda").to(torch.bfloat16)
    w = torch.randn(192, 128, device="cuda").to(torch.bfloat16)
    c = torch.empty(256, 192, device="cuda", dtype=torch.bfloat16)
    b.zl_op_gemm(b.ZL_DTYPE_BF16, 0, 256, 192, 128, a, w, c)
    torch.cuda.synchronize()
    ref = a.double() @ w.double().T
    assert float((c.double() - ref).abs().max()) <= 8e-3 * float(ref.abs().max())
