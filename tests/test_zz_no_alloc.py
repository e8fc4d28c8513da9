"""mixfp4_quantize_noalloc: the allocation-free quantizer entry point.

Some callers cannot allocate device memory while they run -- an inference
runtime that plans its device buffers ahead of time and hands an operator only
its inputs and outputs, or a plugin whose execute call must not call
cudaMalloc.  For them the library keeps the quantizer's one scratch word (the
amax accumulator) in its own device array.  This test calls that entry point
through the C ABI twice in a row and requires the same codes, scale bytes and
tensor scale as mixfp4_quantize with a caller-provided workspace (the
quantizer's outputs are compared bit for bit, as in every quantizer test).
The file is named to be collected last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth

pytestmark = pytest.mark.gpu


def _lib():
    from paper_2605_31035_gb300 import build, ops
    build.build()
    L = ops.lib()
    P, I64, I = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    L.mixfp4_quantize_noalloc.restype = I
    L.mixfp4_quantize_noalloc.argtypes = [P, I, I64, I64, I64, P, P, P, I, P]
    return L


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


@pytest.mark.parametrize("mode", [0, 1, 2, 3])
def test_noalloc_matches_workspace_entry_point(mode):
    L = _lib()
    dev = torch.device("cuda:0")
    stream = ctypes.c_void_p(torch.cuda.current_stream(dev).cuda_stream)
    # two different tensors, so the second call must not reuse the first's amax
    xs = [synth.activations(96, 1024, 4100 + mode, 4200).to(dev),
          (synth.activations(96, 1024, 4300 + mode, None).float() * 3e-3).to(torch.bfloat16).to(dev)]
    for x in xs:
        rows, K = x.shape
        ref_c = torch.empty(rows, K // 2, dtype=torch.uint8, device=dev)
        ref_s = torch.empty(rows, K // 16, dtype=torch.uint8, device=dev)
        ref_t = torch.empty(1, dtype=torch.float32, device=dev)
        ws = torch.empty(1, dtype=torch.int32, device=dev)
        st = L.mixfp4_quantize(_ptr(x), 0, rows, K, K, _ptr(ref_c), _ptr(ref_s), _ptr(ref_t), _ptr(ws),
                               mode, 0, stream)
        assert st == 0
        c = torch.full((rows, K // 2), 0xAA, dtype=torch.uint8, device=dev)
        s = torch.full((rows, K // 16), 0xAA, dtype=torch.uint8, device=dev)
        t = torch.full((1,), -1.0, dtype=torch.float32, device=dev)
        st = L.mixfp4_quantize_noalloc(_ptr(x), 0, rows, K, K, _ptr(c), _ptr(s), _ptr(t), mode, stream)
        assert st == 0
        torch.cuda.synchronize(dev)
        assert np.array_equal(c.cpu().numpy(), ref_c.cpu().numpy())
        assert np.array_equal(s.cpu().numpy(), ref_s.cpu().numpy())
        assert t.cpu().numpy().view(np.uint32)[0] == ref_t.cpu().numpy().view(np.uint32)[0]


def test_noalloc_rejects_bad_arguments():
    L = _lib()
    fake = ctypes.c_void_p(1 << 20)
    assert L.mixfp4_quantize_noalloc(fake, 0, 4, 24, 24, fake, fake, fake, 0, None) == -2
    assert L.mixfp4_quantize_noalloc(fake, 3, 4, 32, 32, fake, fake, fake, 0, None) == -4
    assert L.mixfp4_quantize_noalloc(fake, 0, 4, 32, 32, fake, fake, None, 0, None) == -1
