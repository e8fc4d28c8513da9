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


def test_gemm_missed_stage_reports_and_recovers(oracle):
    """The CTA-pair GEMM kernel with its first code stage withheld: its
    bounded waits run out, the status word reports the roles that gave up,
    the call returns without writing C, and a normal GEMM on the same device
    right after is correct."""
    import numpy as np
    from paper_2605_31035_gb300 import ops, synth
    dev = "cuda:0"
    # K = 1024: four 256-wide K slices, so the producer comes back to the
    # withheld stage's ring slot and its own wait runs out as well.
    x = synth.activations(256, 1024, 9901, 9902)
    w = synth.weights(512, 1024, 9903, 0.02, 0.5)
    qa, qb = ops.mixfp4_quantize(x.to(dev)), ops.mixfp4_quantize(w.to(dev))
    C = torch.full((256, 512), -7.0, dtype=torch.float32, device=dev)
    bits = ops.selftest_gemm_missed_stage(qa, qb, C, limit_ns=5_000_000)
    assert bits & 1, f"producer did not report ({bits:#x})"   # its wait on the withheld stage's slot
    assert bits & 16, f"decoders did not report ({bits:#x})"  # their wait on the withheld stage
    assert torch.all(C == -7.0)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    C2 = ops.mixfp4_gemm(qa, qb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    A = oracle.dequant_rows_f64(qa.codes.cpu().numpy(), qa.scales.cpu().numpy(), qa.tensor_scale.item(), range(256))
    B = oracle.dequant_rows_f64(qb.codes.cpu().numpy(), qb.scales.cpu().numpy(), qb.tensor_scale.item(), range(512))
    D = np.abs(A) @ np.abs(B).T
    err = np.abs(C2.cpu().numpy().astype(np.float64) - A @ B.T)
    assert np.all(err <= 1e-5 * D)
