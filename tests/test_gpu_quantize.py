"""GPU parity of the MixFP4 quantizer and decoder against the CPU oracle.

Codes, scale bytes and s32 must be bit-identical to the oracle (the method's
outputs are integers and bytes); dequantized values must be bit-identical too
(one rounding of an exact product).  Every call goes through the C ABI.
"""
import math

import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def ops():
    from paper_2605_31035_gb300 import ops as o
    return o


def bits(t):
    return synth.bf16_bits(t)


def gpu_quant(x_cpu, mode=0, s32=None, ldx_pad=0):
    o = ops()
    rows, K = x_cpu.shape
    if ldx_pad:
        buf = torch.zeros(rows, K + ldx_pad, dtype=torch.bfloat16)
        buf[:, :K] = x_cpu
        xd = buf.to(DEV)[:, :K]
    else:
        xd = x_cpu.to(DEV)
    ts = None if s32 is None else torch.tensor([s32], dtype=torch.float32, device=DEV)
    q = o.mixfp4_quantize(xd, mode, ts)
    torch.cuda.synchronize()
    return q


def assert_same(q, ref, x_cpu, what=""):
    gc, gs = q.codes.cpu().numpy(), q.scales.cpu().numpy()
    gt = np.float32(q.tensor_scale.item())
    oc, os_, ot = ref
    assert gt.view(np.uint32) == np.float32(ot).view(np.uint32), (what, float(gt), ot)
    if not np.array_equal(gs, os_) or not np.array_equal(gc, oc):
        bad_s = np.argwhere(gs != os_)
        bad_c = np.argwhere(gc != oc)
        r, b = (bad_s[0] if len(bad_s) else (bad_c[0][0], bad_c[0][1] // 8))
        blk = x_cpu[r, b * 16:(b + 1) * 16].float().tolist()
        raise AssertionError(
            f"{what}: {len(bad_s)} scale / {len(bad_c)} code mismatches; first row {r} block {b}: "
            f"x={blk} gpu scale {gs[r, b]:#04x} codes {gc[r, b*8:b*8+8].tolist()} "
            f"oracle scale {os_[r, b]:#04x} codes {oc[r, b*8:b*8+8].tolist()}")


def check(oracle, x_cpu, mode=0, s32=None, ldx_pad=0, what=""):
    q = gpu_quant(x_cpu, mode, s32, ldx_pad)
    ref = oracle.quantize(bits(x_cpu), mode=mode, s32=s32)
    assert_same(q, ref, x_cpu, what)
    return q, ref


@pytest.mark.parametrize("mode", [0, 1, 2])
def test_tiny_linear_operands(oracle, mode):
    w = synth.workloads()["tiny"].linears[0]
    check(oracle, w.make_x(), mode, what="tiny X")
    check(oracle, w.make_w(), mode, what="tiny W")


def test_worked_blocks_on_gpu(oracle):
    """The hand-worked Algorithm 1 blocks reproduce on the GPU byte for byte."""
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "worked_blocks.txt")
    modes = {"mix": 0, "e2m1": 1, "e1m2": 2}
    cases, cur = [], None
    for line in open(path):
        p = line.split()
        if not p or p[0].startswith("#"):
            continue
        if p[0] == "case":
            cur = {"mode": modes[p[2]]}
            cases.append(cur)
        elif p[0] == "x":
            cur["x"] = [float(v) for v in p[1:]]
        elif p[0] in ("codes", "scales"):
            cur[p[0]] = [int(v, 16) for v in p[1:]]
    for c in cases:
        x = torch.tensor(c["x"], dtype=torch.float32).to(torch.bfloat16)[None, :]
        q = gpu_quant(x, c["mode"])
        assert q.codes.cpu().numpy()[0].tolist() == c["codes"]
        assert q.scales.cpu().numpy()[0].tolist() == c["scales"]
        assert q.tensor_scale.item() == 1.0


def _edge_tensor(kind, rng):
    rows, K = 8, 256
    if kind == "zeros":
        return torch.zeros(rows, K, dtype=torch.bfloat16)
    if kind == "negzeros":
        return -torch.zeros(rows, K, dtype=torch.bfloat16)
    x = torch.from_numpy(rng.standard_t(3, (rows, K)).astype(np.float32))
    if kind == "zero_blocks":
        x[:, 32:64] = 0
        x[3, :] = 0
    elif kind == "underflow_blocks":  # block max far below s32 * 2^-10 -> E4M3 zero scales
        x[:, 16:48] *= 1e-7
        x[0, 0] = 1000.0
    elif kind == "ties":  # dyadic grid: exact midpoints in both codebooks
        g = np.array([0, .25, .5, .75, 1, 1.25, 1.5, 1.75, 2, 2.5, 3, 3.5, 4, 5, 6, 7], np.float32)
        x = torch.from_numpy(rng.choice(g, (rows, K)) * rng.choice([-1, 1], (rows, K)).astype(np.float32))
        x[0, 0] = 2688.0
        x *= 2.0 ** int(rng.integers(-6, 6))
    elif kind == "subnormal":  # every value a bf16 subnormal -> s32 subnormal (rescaled path)
        x = torch.from_numpy(rng.integers(1, 128, (rows, K)).astype(np.float32)) * 2.0 ** -133
        x *= torch.from_numpy(rng.choice([-1.0, 1.0], (rows, K)).astype(np.float32))
    elif kind == "mixed_subnormal":
        x[:, ::3] = torch.from_numpy(rng.integers(1, 128, (rows, (K + 2) // 3)).astype(np.float32)) * 2.0 ** -133
    elif kind == "tiny_tensor":  # s32 < 2^-20: rescaled path
        x *= 1e-9
    elif kind == "huge_tensor":  # s32 > 2^100: rescaled path
        x *= 1e36
    elif kind == "wide_range":
        x *= torch.from_numpy((2.0 ** rng.integers(-60, 20, (rows, 1))).astype(np.float32))
    return x.to(torch.bfloat16)


EDGE = ["zeros", "negzeros", "zero_blocks", "underflow_blocks", "ties", "subnormal",
        "mixed_subnormal", "tiny_tensor", "huge_tensor", "wide_range"]


@pytest.mark.parametrize("kind", EDGE)
@pytest.mark.parametrize("mode", [0, 1, 2])
def test_edge_tensors(oracle, kind, mode):
    rng = np.random.default_rng(EDGE.index(kind) * 7 + mode)
    x = _edge_tensor(kind, rng)
    check(oracle, x, mode, what=kind)


def test_power_of_two_rescaling(oracle):
    x = synth.activations(16, 512, 77, 78)
    q0 = gpu_quant(x)
    for k in (-7, 5):
        qk = gpu_quant((x.float() * 2.0 ** k).to(torch.bfloat16))
        assert torch.equal(qk.codes, q0.codes) and torch.equal(qk.scales, q0.scales)
        assert qk.tensor_scale.item() == q0.tensor_scale.item() * 2.0 ** k


@pytest.mark.parametrize("s32", [1.0, 0.0123, 3.0e-4, 1e-30, 5e-45])
def test_given_scale(oracle, s32):
    """SCALE_GIVEN: s32 supplied by the caller, including values that make
    blocks saturate (a > 2688) and tiny ones that take the rescaled path."""
    x = synth.activations(8, 512, 91, 92)
    if s32 < 1e-20:
        x = (x.float() * 1e-35).to(torch.bfloat16)
    check(oracle, x, 0, s32=np.float32(s32).item(), what=f"given {s32}")


@pytest.mark.parametrize("s32", [float.fromhex("0x1.a15686p+0"), float.fromhex("0x1.f250c6p-3"),
                                 float.fromhex("0x1.000002p+0"), float.fromhex("0x1.0b06ecp+5")])
def test_given_scale_division_fallback(oracle, s32):
    """Tensor scales whose x / s32 the kernel must not take with the
    two-instruction division (it is inexact for a bf16 significand of x, or
    its correction term can leave the normal range), so the quantizer falls
    back to Markstein's correction; the block data include the significand
    that fails (0x1.8e for 0x1.a15686, 0x1.e8 for 0x1.f250c6)."""
    x = synth.activations(8, 512, 93, 94).float()
    for i, v in enumerate((float.fromhex("0x1.8ep+0"), float.fromhex("0x1.e8p+0"))):
        cols = x[::2, i::37].shape[1]
        x[::2, i::37] = torch.from_numpy(v * 2.0 ** np.arange(-3, 4).repeat(3)[:cols]).float()
        x[1::2, 5 + i::41] = -v
    check(oracle, x.to(torch.bfloat16), 0, s32=s32, what=f"given {s32!r}")


@pytest.mark.parametrize("shape", [(1, 16), (3, 48), (257, 4112), (5, 16 * 999)])
def test_ragged_shapes(oracle, shape):
    rows, K = shape
    x = synth.activations(rows, K, 1000 + rows, None)
    check(oracle, x, 0, what=str(shape))


def test_strided_rows(oracle):
    x = synth.activations(33, 512, 55, 56)
    check(oracle, x, 0, ldx_pad=48, what="ldx=K+48")
    check(oracle, x, 1, ldx_pad=16, what="ldx=K+16")


def test_empty_input():
    o = ops()
    x = torch.empty(0, 64, dtype=torch.bfloat16, device=DEV)
    q = o.mixfp4_quantize(x)
    torch.cuda.synchronize()
    assert q.tensor_scale.item() == 0.0 and q.codes.numel() == 0


def _sampled_check(oracle, x_cpu, nsample=48, seed=0):
    """Full-size tensor on the GPU; the oracle redoes sampled rows with the
    tensor scale fixed by the definition s32 = fl32(max|X| / 2688)."""
    q = gpu_quant(x_cpu)
    amax = np.float32(x_cpu.abs().max().float().item())
    s32 = np.float32(amax / np.float32(2688.0))
    assert np.float32(q.tensor_scale.item()).view(np.uint32) == s32.view(np.uint32)
    rng = np.random.default_rng(seed)
    rows = np.unique(np.concatenate([[0, x_cpu.shape[0] - 1],
                                     rng.integers(0, x_cpu.shape[0], nsample)]))
    xs = x_cpu[torch.from_numpy(rows)]
    oc, os_, _ = oracle.quantize(bits(xs), s32=float(s32))
    gc = q.codes[torch.from_numpy(rows).to(DEV)].cpu().numpy()
    gs = q.scales[torch.from_numpy(rows).to(DEV)].cpu().numpy()
    assert np.array_equal(gs, os_) and np.array_equal(gc, oc)
    return q


@pytest.mark.slow
@pytest.mark.parametrize("name", ["attn", "mlp", "decode", "hadamard"])
def test_full_size_workloads(oracle, name):
    wl = synth.workloads()[name]
    for lin in wl.linears[:2] if name == "mlp" else wl.linears:
        _sampled_check(oracle, lin.make_x(), seed=1)
        _sampled_check(oracle, lin.make_w(), seed=2)
    if name == "mlp":
        _sampled_check(oracle, wl.linears[2].make_x(), seed=3)


@pytest.mark.slow
def test_sweep_point_2_26(oracle):
    _sampled_check(oracle, synth.sweep_activation(26), seed=4)


# ---------------------------------------------------------------- dequantize
def test_dequantize_bit_exact(oracle):
    for x in (synth.activations(64, 512, 5, 6), _edge_tensor("ties", np.random.default_rng(3)),
              _edge_tensor("subnormal", np.random.default_rng(4))):
        for mode in (0, 1, 2):
            q = gpu_quant(x, mode)
            out = ops().mixfp4_dequantize(q)
            torch.cuda.synchronize()
            ref = oracle.dequantize(q.codes.cpu().numpy(), q.scales.cpu().numpy(), q.tensor_scale.item())
            assert np.array_equal(out.cpu().numpy().view(np.uint32), ref.view(np.uint32))
