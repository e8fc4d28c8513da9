"""Failure detection on the GPU without a fault: the bounded mbarrier wait
used by the GEMM pipelines gives up on an injected missed arrival (a barrier
nothing arrives on) after its time limit, and at once when the abort flag is
raised, and reports both through the status word."""
import time

import pytest
import torch

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_missed_arrival():
    from paper_2605_31035_gb300 import ops
    limit_ns = 20_000_000
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    bits = ops.selftest_bounded_wait(limit_ns)
    dt = time.perf_counter() - t0
    assert bits == 0xE, hex(bits)      # (a) ok, (b) timed out after the limit, (c) aborted
    assert dt >= limit_ns * 1e-9
    # the device is still usable afterwards
    x = torch.ones(1024, device="cuda")
    assert float(x.sum()) == 1024.0
