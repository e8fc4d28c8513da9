"""GPU parity of the fused 128-point rotation + MixFP4 quantizer
(mixfp4_quantize_rht) against the oracle's rotation (reading R11) followed by
Algorithm 1 on the fp32 result: codes, scale bytes and s32 bit-identical."""
import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def ops():
    from paper_2605_31035_gb300 import ops as o
    return o


def signs_of(seed):
    return None if seed is None else np.random.default_rng(seed).integers(0, 256, 16).astype(np.uint8)


def run_gpu(x_cpu, sg, mode=0, s32=None, ldx_pad=0):
    rows, K = x_cpu.shape
    if ldx_pad:
        buf = torch.zeros(rows, K + ldx_pad, dtype=torch.bfloat16)
        buf[:, :K] = x_cpu
        xd = buf.to(DEV)[:, :K]
    else:
        xd = x_cpu.to(DEV)
    sd = None if sg is None else torch.from_numpy(sg).to(DEV)
    ts = None if s32 is None else torch.tensor([s32], dtype=torch.float32, device=DEV)
    q = ops().mixfp4_quantize_rht(xd, sd, mode, ts)
    torch.cuda.synchronize()
    return q.codes.cpu().numpy(), q.scales.cpu().numpy(), q.tensor_scale.item()


def check(oracle, x_cpu, sg, mode=0, s32=None, ldx_pad=0):
    y = oracle.rht(synth.bf16_bits(x_cpu), sg)
    rc, rs, rt = oracle.quantize_f32(y, mode, s32)
    gc, gs, gt = run_gpu(x_cpu, sg, mode, s32, ldx_pad)
    assert np.float32(gt) == np.float32(rt)
    bad = np.argwhere(gs != rs)
    assert bad.size == 0, f"scale mismatch at {bad[:5].tolist()}"
    assert np.array_equal(gc, rc)


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("seed", [None, 5])
def test_rht_quantize_matches_oracle(oracle, mode, seed):
    x = synth.activations(64, 1024, 81, 82)
    check(oracle, x, signs_of(seed), mode)


@pytest.mark.parametrize("shape", [(1, 128), (3, 256), (33, 2048), (257, 384)])
def test_rht_ragged_rows_and_chunks(oracle, shape):
    x = synth.activations(shape[0], shape[1], 83 + shape[0], 84)
    check(oracle, x, signs_of(7))


def test_rht_strided_rows(oracle):
    check(oracle, synth.activations(40, 512, 85, 86), signs_of(9), ldx_pad=64)


@pytest.mark.parametrize("s32", [0.01, 1e-30])
def test_rht_given_scale(oracle, s32):
    x = synth.activations(16, 512, 87, 88)
    if s32 < 1e-20:
        x = (x.float() * 1e-35).to(torch.bfloat16)
    check(oracle, x, signs_of(3), s32=np.float32(s32).item())


def test_rht_zeros_and_unit_vectors(oracle):
    x = torch.zeros(8, 256, dtype=torch.bfloat16)
    check(oracle, x, None)
    x = torch.zeros(8, 256)
    for r in range(8):
        x[r, 37 * r % 256] = 2.0 ** (r - 3)
    check(oracle, x.to(torch.bfloat16), signs_of(11))


def test_rht_rejects_k_not_multiple_of_128():
    x = torch.zeros(4, 64, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(Exception):
        ops().mixfp4_quantize_rht(x)


@pytest.mark.slow
def test_rht_full_size_sampled_rows(oracle):
    """8192 x 8192 activations with outlier channels (the Hadamard-rotated
    GEMM's X before rotation): s32 from the whole rotated tensor, sampled rows
    bit-exact."""
    x = synth.activations(8192, 8192, 1005, 3005)
    sg = signs_of(13)
    gc, gs, gt = run_gpu(x, sg)
    b = synth.bf16_bits(x)
    y = oracle.rht(b, sg)
    s32 = float(np.float32(np.float32(np.abs(y).max()) / np.float32(2688.0)))
    assert np.float32(gt) == np.float32(s32)
    rows = np.unique(np.concatenate([[0, 8191], np.random.default_rng(1).integers(0, 8192, 30)]))
    rc, rs, _ = oracle.quantize_f32(y[rows], 0, s32)
    assert np.array_equal(gs[rows], rs) and np.array_equal(gc[rows], rc)
