"""GPU parity of stochastic rounding (reading R13): row-wise and column-wise
codes bit-exact against the CPU oracle for several seeds and offsets (the
Philox4x32-10 uniforms are drawn independently on each side from the same
published definition), with scale bytes and s32 equal to round-to-nearest
Algorithm 1.  Every call goes through the C ABI."""
import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
SEEDS = [(0, 0), (12345, 7), (0xFEDCBA9876543210, (3 << 32) + 11)]


def ops():
    from paper_2605_31035_gb300 import ops as o
    return o


def check(q, ref):
    torch.cuda.synchronize()
    c, s, t = ref
    assert np.float32(q.tensor_scale.item()).view(np.uint32) == np.float32(t).view(np.uint32)
    assert np.array_equal(q.scales.cpu().numpy(), s)
    gc = q.codes.cpu().numpy()
    assert np.array_equal(gc, c), f"{int((gc != c).sum())} code byte mismatches"


@pytest.mark.parametrize("shape", [(1, 16), (37, 80), (256, 512)])
@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("seed,offset", SEEDS)
def test_rowwise_sr_bit_exact(oracle, shape, mode, seed, offset):
    rows, K = shape
    g = synth.activations(rows, K, 9500 + rows, 9501)   # gradient-like heavy tails
    q = ops().mixfp4_quantize_sr(g.to(DEV), seed, offset, mode)
    check(q, oracle.quantize_sr(synth.bf16_bits(g), seed, offset, mode))
    rn = oracle.quantize(synth.bf16_bits(g), mode)
    assert np.array_equal(q.scales.cpu().numpy(), rn[1])


@pytest.mark.parametrize("shape", [(16, 16), (80, 272), (512, 64)])
@pytest.mark.parametrize("mode", [0, 2])
@pytest.mark.parametrize("seed,offset", SEEDS[1:])
def test_colwise_sr_bit_exact(oracle, shape, mode, seed, offset):
    R, C = shape
    g = synth.activations(R, C, 9600 + R, 9601)
    q = ops().mixfp4_quantize_sr(g.to(DEV), seed, offset, mode, colwise=True)
    check(q, oracle.quantize_colwise_sr(synth.bf16_bits(g), seed, offset, mode))


def test_sr_strided_given_scale_and_determinism(oracle):
    g = synth.activations(40, 96, 9700, 9701)
    buf = torch.zeros(40, 128, dtype=torch.bfloat16)
    buf[:, :96] = g
    xd = buf.to(DEV)[:, :96]
    s32 = 0.0123
    q1 = ops().mixfp4_quantize_sr(xd, 99, 5, tensor_scale=torch.tensor([s32], device=DEV))
    q2 = ops().mixfp4_quantize_sr(xd, 99, 5, tensor_scale=torch.tensor([s32], device=DEV))
    check(q1, oracle.quantize_sr(synth.bf16_bits(g), 99, 5, s32=float(np.float32(s32))))
    assert torch.equal(q1.codes, q2.codes)
    q3 = ops().mixfp4_quantize_sr(xd, 100, 5, tensor_scale=torch.tensor([s32], device=DEV))
    torch.cuda.synchronize()
    assert not torch.equal(q1.codes, q3.codes)     # another seed, other draws
