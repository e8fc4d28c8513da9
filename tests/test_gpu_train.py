"""GPU parity of the training-flow quantizer orientations (Sec. 3.2):
column-wise blocks (WGRAD / DGRAD operands), 2D 16 x 16 weight blocks
(reading R12) and the transpose of a 2D-quantized tensor, each bit-exact
against the CPU oracle, plus the GEMMs they feed within the 1e-5 bound.
Every call goes through the C ABI."""
import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def ops():
    from paper_2605_31035_gb300 import ops as o
    return o


def on_gpu(x_cpu, pad=0):
    if not pad:
        return x_cpu.to(DEV)
    rows, K = x_cpu.shape
    buf = torch.zeros(rows, K + pad, dtype=torch.bfloat16)
    buf[:, :K] = x_cpu
    return buf.to(DEV)[:, :K]


def same(q, ref):
    torch.cuda.synchronize()
    c, s, t = ref
    assert np.float32(q.tensor_scale.item()).view(np.uint32) == np.float32(t).view(np.uint32)
    gc, gs = q.codes.cpu().numpy(), q.scales.cpu().numpy()
    bad = np.argwhere(gs != s)
    assert bad.size == 0, f"{len(bad)} scale mismatches, first at {bad[0]}"
    assert np.array_equal(gc, c), f"{int((gc != c).sum())} code byte mismatches"


@pytest.mark.parametrize("shape", [(16, 16), (64, 256), (80, 272), (208, 512), (1024, 48)])
@pytest.mark.parametrize("mode", [0, 1, 2])
def test_colwise_bit_exact(oracle, shape, mode):
    """Tiles of 64 rows x 256 columns: one tile, ragged row and column tails."""
    R, C = shape
    x = synth.activations(R, C, 9100 + R + C, 9101)
    q = ops().mixfp4_quantize_colwise(x.to(DEV), mode)
    same(q, oracle.quantize_colwise(synth.bf16_bits(x), mode))


def test_colwise_strided_and_given_scale(oracle):
    x = synth.activations(96, 160, 9102, 9103)
    q = ops().mixfp4_quantize_colwise(on_gpu(x, 32))
    same(q, oracle.quantize_colwise(synth.bf16_bits(x)))
    s32 = 0.0371
    q = ops().mixfp4_quantize_colwise(x.to(DEV), tensor_scale=torch.tensor([s32], device=DEV))
    same(q, oracle.quantize_colwise(synth.bf16_bits(x), s32=float(np.float32(s32))))


@pytest.mark.parametrize("shape", [(16, 16), (1, 64), (37, 80), (64, 512), (130, 272)])
@pytest.mark.parametrize("mode", [0, 1, 2])
def test_2d_bit_exact(oracle, shape, mode):
    """Whole and ragged row tiles, an odd number of block columns (a half-warp
    with no tile), all three modes."""
    rows, K = shape
    w = synth.weights(rows, K, 9200 + rows + K, 0.02, 0.5)
    q = ops().mixfp4_quantize_2d(w.to(DEV), mode)
    same(q, oracle.quantize_2d(synth.bf16_bits(w), mode))


def test_2d_strided_given_scale_and_activations(oracle):
    x = synth.activations(48, 96, 9201, 9202)    # heavy tails and outlier columns
    q = ops().mixfp4_quantize_2d(on_gpu(x, 16))
    same(q, oracle.quantize_2d(synth.bf16_bits(x)))
    s32 = 3.0e-4
    q = ops().mixfp4_quantize_2d(x.to(DEV), tensor_scale=torch.tensor([s32], device=DEV))
    same(q, oracle.quantize_2d(synth.bf16_bits(x), s32=float(np.float32(s32))))


@pytest.mark.parametrize("shape", [(16, 16), (48, 80), (64, 144), (128, 256), (272, 1040), (320, 1040)])
def test_transpose_2d_bit_exact(oracle, shape):
    rows, K = shape
    w = synth.weights(rows, K, 9300 + rows, 0.02, 0.5)
    q = ops().mixfp4_quantize_2d(w.to(DEV))
    t = ops().mixfp4_transpose_2d(q)
    torch.cuda.synchronize()
    ct, st = oracle.transpose_2d(q.codes.cpu().numpy(), q.scales.cpu().numpy())
    assert np.array_equal(t.codes.cpu().numpy(), ct) and np.array_equal(t.scales.cpu().numpy(), st)


def test_training_gemms(oracle):
    """FPROP, DGRAD and WGRAD of one linear layer on MixFP4 operands, each
    within the 1e-5 bound of the float64 oracle GEMM of the same operands:
    Y = X W^T (X row-wise, W 2D), dX = dY W (dY row-wise, W^T by the 2D
    transpose), dW = dY^T X (both column-wise, reducing over tokens)."""
    o = ops()
    T_, I_, O_ = 512, 256, 768      # tokens, in features, out features
    X = synth.activations(T_, I_, 9400, 9401)
    W = synth.weights(O_, I_, 9402, 0.02, 0.5)
    dY = synth.activations(T_, O_, 9403, None)
    qX, qW, qdY = o.mixfp4_quantize(X.to(DEV)), o.mixfp4_quantize_2d(W.to(DEV)), o.mixfp4_quantize(dY.to(DEV))
    qWt = o.mixfp4_transpose_2d(qW)
    qdYc, qXc = o.mixfp4_quantize_colwise(dY.to(DEV)), o.mixfp4_quantize_colwise(X.to(DEV))
    cases = [(qX, qW), (qdY, qWt), (qdYc, qXc)]
    for a, b in cases:
        C = o.mixfp4_gemm(a, b)
        torch.cuda.synchronize()
        ra = (a.codes.cpu().numpy(), a.scales.cpu().numpy(), float(a.tensor_scale.item()))
        rb = (b.codes.cpu().numpy(), b.scales.cpu().numpy(), float(b.tensor_scale.item()))
        Cref = oracle.gemm_f64(ra, rb)
        A = oracle.dequant_rows_f64(*ra, range(a.rows))
        B = oracle.dequant_rows_f64(*rb, range(b.rows))
        D = np.abs(A) @ np.abs(B).T
        err = np.abs(C.cpu().numpy().astype(np.float64) - Cref)
        assert np.all(err <= 1e-5 * D)
    # the operands themselves are the oracle's
    same(qWt, (*oracle.transpose_2d(*oracle.quantize_2d(synth.bf16_bits(W))[:2]),
               oracle.quantize_2d(synth.bf16_bits(W))[2]))
    same(qdYc, oracle.quantize_colwise(synth.bf16_bits(dY)))


@pytest.mark.slow
def test_full_size_orientations(oracle):
    """The attention-projection weight (4096 x 4096) in 2D blocks and its
    transpose, and the attention activation (2048 x 4096) column-wise, on
    sampled rows of the oracle."""
    o = ops()
    lin = synth.workloads()["attn"].linears[0]
    w, x = lin.make_w(), lin.make_x()
    q = o.mixfp4_quantize_2d(w.to(DEV))
    t = o.mixfp4_transpose_2d(q)
    qc = o.mixfp4_quantize_colwise(x.to(DEV))
    torch.cuda.synchronize()
    s32w = float(q.tensor_scale.item())
    rng = np.random.default_rng(3)
    for rt in sorted(set(rng.integers(0, 256, 6).tolist()) | {0, 255}):
        rows = slice(16 * rt, 16 * rt + 16)
        c, s, _ = oracle.quantize_2d(synth.bf16_bits(w[rows]), s32=s32w)
        assert np.array_equal(q.codes[rows].cpu().numpy(), c) and np.array_equal(q.scales[rows].cpu().numpy(), s)
    ct, st = oracle.transpose_2d(q.codes.cpu().numpy(), q.scales.cpu().numpy())
    assert np.array_equal(t.codes.cpu().numpy(), ct) and np.array_equal(t.scales.cpu().numpy(), st)
    s32x = float(qc.tensor_scale.item())
    xb = synth.bf16_bits(x)
    for col in sorted(set(rng.integers(0, 4096, 24).tolist()) | {0, 4095}):
        c, s, _ = oracle.quantize(np.ascontiguousarray(xb[:, col][None, :]), s32=s32x)
        assert np.array_equal(qc.codes[col].cpu().numpy(), c[0]) and np.array_equal(qc.scales[col].cpu().numpy(), s[0])


@pytest.mark.parametrize("shape", [(128, 16), (256, 80), (384, 272)])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("with_signs", [False, True])
def test_colwise_rht_bit_exact(oracle, shape, mode, with_signs):
    """Rotation of every 128-row chunk of each column, then column-wise
    Algorithm 1: the rotated X^T quantized bit for bit as the oracle's
    quantize_f32(rht(X^T)); one and several 64-column tiles, ragged columns."""
    R, C = shape
    x = synth.activations(R, C, 9800 + R + C, 9801)
    signs = None
    if with_signs:
        signs = np.random.default_rng(R + C).integers(0, 256, 16).astype(np.uint8)
    sg = None if signs is None else torch.from_numpy(signs).to(DEV)
    q = ops().mixfp4_quantize_colwise_rht(x.to(DEV), sg, mode)
    same(q, oracle.quantize_colwise_rht(synth.bf16_bits(x), signs, mode))


def test_colwise_rht_given_scale_and_row_wise_agreement(oracle):
    """With a given s32, and equal to the row-wise rotated quantizer applied to
    an explicitly transposed copy of X on the GPU."""
    x = synth.activations(256, 48, 9802, 9803)
    s32 = 0.021
    q = ops().mixfp4_quantize_colwise_rht(x.to(DEV), tensor_scale=torch.tensor([s32], device=DEV))
    same(q, oracle.quantize_colwise_rht(synth.bf16_bits(x), None, 0, s32=float(np.float32(s32))))
    qt = ops().mixfp4_quantize_rht(x.t().contiguous().to(DEV))
    qc = ops().mixfp4_quantize_colwise_rht(x.to(DEV))
    torch.cuda.synchronize()
    assert torch.equal(qt.codes, qc.codes) and torch.equal(qt.scales, qc.scales)
    assert qt.tensor_scale.item() == qc.tensor_scale.item()


@pytest.mark.slow
def test_colwise_rht_attention_activation(oracle):
    """The attention activation (2048 tokens x 4096) rotated along tokens,
    against the row-wise rotated quantizer on its explicit transpose."""
    x = synth.workloads()["attn"].linears[0].make_x().to(DEV)
    signs = torch.from_numpy(np.random.default_rng(7).integers(0, 256, 16).astype(np.uint8)).to(DEV)
    qc = ops().mixfp4_quantize_colwise_rht(x, signs)
    qt = ops().mixfp4_quantize_rht(x.t().contiguous(), signs)
    torch.cuda.synchronize()
    assert torch.equal(qt.codes, qc.codes) and torch.equal(qt.scales, qc.scales)
    assert qt.tensor_scale.item() == qc.tensor_scale.item()
