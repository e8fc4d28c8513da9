"""GPU parity of the candidate-set / block-size quantize-dequantize (reading
R14; Sec. 2.4 candidate sets, Sec. 4.3 Table 5 block sizes): outputs (fp32 and
bf16), per-block choices and the tensor scale bit-exact against the CPU
oracle, through the C ABI."""
import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
ALL = 15
SETS = [ALL, 1 | 4, 1 | 2 | 8, 1, 8]   # all four, {E2M1(6), E2M1(4)}, {E2M1(6), E1M2, E3M0}, NVFP4, E3M0


def ops():
    from paper_2605_31035_gb300 import ops as o
    return o


def check(x_cpu, mask, g, s32=None, out_dtype=torch.float32, pad_in=0, pad_out=0, oracle=None):
    o = ops()
    rows, K = x_cpu.shape
    if pad_in:
        buf = torch.zeros(rows, K + pad_in, dtype=torch.bfloat16)
        buf[:, :K] = x_cpu
        x = buf.to(DEV)[:, :K]
    else:
        x = x_cpu.to(DEV)
    out = None
    if pad_out:
        out = torch.empty(rows, K + pad_out, dtype=out_dtype, device=DEV)[:, :K]
    ts = None if s32 is None else torch.tensor([s32], device=DEV)
    y, ch, t = o.mixfp4_fake_quantize(x, mask, g, out_dtype, tensor_scale=ts, out=out)
    torch.cuda.synchronize()
    ref, rch, rs = oracle.fake_quantize(synth.bf16_bits(x_cpu), mask, g, s32, out_bf16=out_dtype == torch.bfloat16)
    assert np.float32(t.item()).view(np.uint32) == np.float32(rs).view(np.uint32)
    bad = np.argwhere(ch.cpu().numpy() != rch)
    assert bad.size == 0, f"{len(bad)} choice mismatches, first at {bad[0]}"
    if out_dtype == torch.bfloat16:
        got = y.cpu().view(torch.int16).numpy().view(np.uint16)
    else:
        got = y.cpu().numpy().view(np.uint32)
        ref = ref.view(np.uint32)
    mism = np.argwhere(got != ref)
    assert mism.size == 0, f"{len(mism)} output mismatches, first at {mism[0]}"


@pytest.mark.parametrize("mask", range(1, 16))
def test_every_candidate_set_g16(oracle, mask):
    check(synth.activations(40, 512, 7000 + mask, 7001), mask, 16, oracle=oracle)


@pytest.mark.parametrize("g", [8, 32, 64])
@pytest.mark.parametrize("mask", SETS)
@pytest.mark.parametrize("shape", [(1, 64), (37, 192), (96, 1024)])
def test_block_sizes(oracle, g, mask, shape):
    rows, K = shape
    check(synth.activations(rows, K, 7100 + g + rows, 7101), mask, g, oracle=oracle)


@pytest.mark.parametrize("g", [8, 16, 64])
def test_bf16_output_strided_and_given_scale(oracle, g):
    x = synth.activations(50, 320, 7200 + g, 7201)
    check(x, ALL, g, out_dtype=torch.bfloat16, oracle=oracle)
    check(x, 1 | 2 | 8, g, pad_in=32, pad_out=16, oracle=oracle)
    check(x, ALL, g, s32=float(np.float32(0.0217)), out_dtype=torch.bfloat16, pad_out=48, oracle=oracle)


def test_weights_distribution(oracle):
    w = synth.weights(64, 4096, 7300, 0.02, 0.5)
    for g in (8, 16, 32, 64):
        check(w, ALL, g, oracle=oracle)


def test_zero_tensor_ties_to_last_candidate(oracle):
    x = torch.zeros(16, 128, dtype=torch.bfloat16)
    x[3] = -0.0
    for mask, last in [(ALL, 3), (1 | 4, 2), (1 | 2, 1)]:
        check(x, mask, 32, oracle=oracle)
        _, ch, t = ops().mixfp4_fake_quantize(x.to(DEV), mask, 32)
        assert t.item() == 0.0 and bool((ch == last).all())


def test_mixfp4_pair_is_quantize_then_dequantize():
    """{E2M1(6), E1M2} at g = 16 through this entry point equals the
    dequantized output of the MixFP4 quantizer (two GPU paths, one
    definition)."""
    o = ops()
    x = synth.activations(256, 4096, 7400, 7401).to(DEV)
    y, ch, t = o.mixfp4_fake_quantize(x, 1 | 2, 16)
    q = o.mixfp4_quantize(x)
    d = o.mixfp4_dequantize(q)
    torch.cuda.synchronize()
    assert torch.equal(y.view(torch.int32), d.view(torch.int32))
    assert torch.equal(ch, (q.scales >> 7).to(torch.uint8))
    assert t.item() == q.tensor_scale.item()


@pytest.mark.slow
def test_full_size_sampled_rows(oracle):
    """The attention activation (2048 x 4096) with all four candidates at each
    block size; sampled rows against the oracle, which takes the tensor scale
    fl32(max|x| / 2688) computed here from the input."""
    o = ops()
    lin = synth.workloads()["attn"].linears[0]
    x = lin.make_x()
    s32 = float(np.float32(np.float32(x.abs().max().float().item()) / np.float32(2688.0)))
    xd = x.to(DEV)
    rows = [0, 1, 777, 1500, 2047]
    for g in (8, 16, 32, 64):
        y, ch, t = o.mixfp4_fake_quantize(xd, ALL, g)
        torch.cuda.synchronize()
        assert np.float32(t.item()) == np.float32(s32)
        ref, rch, _ = oracle.fake_quantize(synth.bf16_bits(x[rows]), ALL, g, s32)
        assert np.array_equal(y[rows].cpu().numpy().view(np.uint32), ref.view(np.uint32))
        assert np.array_equal(ch[rows].cpu().numpy(), rch)


@pytest.mark.parametrize("shape", [(1, 16), (40, 512), (37, 272)])
@pytest.mark.parametrize("given", [False, True])
def test_four_six_mode_packs_the_46_candidate_set(oracle, shape, given):
    """MIXFP4_MODE_FOUR_SIX: the codes the GPU stores decode (oracle
    dequantizer) to exactly the oracle's {E2M1(6), E2M1(4)} quantize-dequantize
    at g = 16, every type bit is 0, and each scale byte is E4M3 of B/6 or B/4
    as the oracle chose."""
    o = ops()
    rows, K = shape
    x = synth.activations(rows, K, 7500 + rows + K, 7501)
    bits = synth.bf16_bits(x)
    s32 = float(np.float32(0.0173)) if given else None
    ts = None if s32 is None else torch.tensor([s32], device=DEV)
    q = o.mixfp4_quantize(x.to(DEV), o.MODE_FOUR_SIX, tensor_scale=ts)
    torch.cuda.synchronize()
    codes, scales, t = q.codes.cpu().numpy(), q.scales.cpu().numpy(), float(q.tensor_scale.item())
    ref, choice, rs = oracle.fake_quantize(bits, 1 | 4, 16, s32)
    assert np.float32(t).view(np.uint32) == np.float32(rs).view(np.uint32)
    assert not np.any(scales & 0x80)
    deq = oracle.dequantize(codes, scales, t)
    assert np.array_equal(deq.view(np.uint32), ref.view(np.uint32))
    xf = (bits.astype(np.uint32) << 16).view(np.float32)
    a = (np.abs(xf) / np.float32(rs)).astype(np.float32) if rs > 0 else np.zeros_like(xf)
    B = a.reshape(rows, K // 16, 16).max(axis=2)
    div = np.where(choice == 2, np.float32(4.0), np.float32(6.0))
    want = np.vectorize(lambda v: oracle.e4m3_rne(float(v)))((B / div).astype(np.float32))
    assert np.array_equal(scales, want.astype(np.uint8))


def test_four_six_operands_in_both_gemms(oracle):
    """4/6 operands are plain NVFP4 bits: the decode-path GEMM and the native
    variant (one E2M1 product) take them, within the 1e-5 bound."""
    o = ops()
    X = synth.activations(256, 512, 7600, 7601)
    W = synth.weights(384, 512, 7602, 0.02, 0.5)
    qx, qw = o.mixfp4_quantize(X.to(DEV), o.MODE_FOUR_SIX), o.mixfp4_quantize(W.to(DEV), o.MODE_FOUR_SIX)
    C1 = o.mixfp4_gemm(qx, qw)
    C2 = o.mixfp4_gemm_native(o.mixfp4_split_native(qx), o.mixfp4_split_native(qw))
    torch.cuda.synchronize()
    ra = (qx.codes.cpu().numpy(), qx.scales.cpu().numpy(), float(qx.tensor_scale.item()))
    rb = (qw.codes.cpu().numpy(), qw.scales.cpu().numpy(), float(qw.tensor_scale.item()))
    Cref = oracle.gemm_f64(ra, rb)
    D = np.abs(oracle.dequant_rows_f64(*ra, range(256))) @ np.abs(oracle.dequant_rows_f64(*rb, range(384))).T
    for C in (C1, C2):
        assert np.all(np.abs(C.cpu().numpy().astype(np.float64) - Cref) <= 1e-5 * D)
