"""GPU parity of the MixFP4 x MixFP4 GEMM against the float64 CPU oracle.

Criterion (spec tolerance): max |C_gpu - C_oracle| / (|A_deq| . |B_deq|^T)
<= 1e-5 elementwise, with C_oracle the float64 product of the dequantized
operands; where |A_deq| . |B_deq|^T is 0, C_gpu must be exactly 0.  The
operands are first checked to be the oracle's codes bit for bit.
"""
import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
TOL = 1e-5


def ops():
    from paper_2605_31035_gb300 import ops as o
    return o


def quant_both(oracle, t, mode=0):
    q = ops().mixfp4_quantize(t.to(DEV), mode)
    ref = oracle.quantize(synth.bf16_bits(t), mode=mode)
    torch.cuda.synchronize()
    assert np.array_equal(q.codes.cpu().numpy(), ref[0]) and np.array_equal(q.scales.cpu().numpy(), ref[1])
    return q, ref


def assert_close(Cg, Cref, A, B):
    D = np.abs(A) @ np.abs(B).T
    err = np.abs(Cg.astype(np.float64) - Cref)
    zero = D == 0
    assert np.all(Cg[zero] == 0)
    rel = err[~zero] / D[~zero]
    assert rel.size == 0 or rel.max() <= TOL, f"max rel err {rel.max():.3e}"
    return 0.0 if rel.size == 0 else float(rel.max())


def full_check(oracle, x, w, mode=0):
    qa, ra = quant_both(oracle, x, mode)
    qb, rb = quant_both(oracle, w, mode)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = ops().mixfp4_gemm(qa, qb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    Cref = oracle.gemm_f64(ra, rb)
    A = oracle.dequant_rows_f64(ra[0], ra[1], ra[2], range(x.shape[0]))
    B = oracle.dequant_rows_f64(rb[0], rb[1], rb[2], range(w.shape[0]))
    return assert_close(C.cpu().numpy(), Cref, A, B)


@pytest.mark.parametrize("mode", [0, 1, 2])
def test_tiny_linear(oracle, mode):
    lin = synth.workloads()["tiny"].linears[0]
    full_check(oracle, lin.make_x(), lin.make_w(), mode)


@pytest.mark.parametrize("M,N,K", [(200, 300, 512), (1, 1, 256), (129, 257, 768), (64, 520, 1280),
                                   (300, 16, 256), (1, 600, 512), (17, 1024, 768), (48, 700, 256),
                                   (64, 2048, 4096), (65, 512, 512)])
def test_ragged_tiles(oracle, M, N, K):
    """M and N tails (TMA zero fill, masked stores), one code stage, odd
    numbers of code stages (ring wrap), and the few-row (M <= 64) path with its
    split of weight tiles and K slices across CTAs."""
    x = synth.activations(M, K, 7000 + M, 7100 + M)
    w = synth.weights(N, K, 7200 + N, 0.02, 0.5)
    full_check(oracle, x, w)


def test_zero_operand_gives_exact_zero(oracle):
    x = torch.zeros(128, 512, dtype=torch.bfloat16)
    w = synth.weights(256, 512, 11, 0.02)
    qa, _ = quant_both(oracle, x)
    qb, _ = quant_both(oracle, w)
    C = ops().mixfp4_gemm(qa, qb)
    torch.cuda.synchronize()
    assert torch.count_nonzero(C).item() == 0


def test_empty_reduction_and_shapes():
    o = ops()
    qa = o.empty_qtensor(4, 0, DEV)
    qb = o.empty_qtensor(8, 0, DEV)
    C = torch.full((4, 8), 7.0, device=DEV)
    o.mixfp4_gemm(qa, qb, out=C)
    torch.cuda.synchronize()
    assert torch.count_nonzero(C).item() == 0
    qa = o.empty_qtensor(0, 256, DEV)
    qb = o.empty_qtensor(8, 256, DEV)
    C = o.mixfp4_gemm(qa, qb)
    assert C.shape == (0, 8)


def test_strided_output(oracle):
    x = synth.activations(130, 512, 21, 22)
    w = synth.weights(200, 512, 23, 0.02)
    qa, ra = quant_both(oracle, x)
    qb, rb = quant_both(oracle, w)
    big = torch.full((130, 260), -1.0, device=DEV)
    ops().mixfp4_gemm(qa, qb, out=big[:, :200])
    torch.cuda.synchronize()
    assert torch.all(big[:, 200:] == -1.0)
    Cref = oracle.gemm_f64(ra, rb)
    A = oracle.dequant_rows_f64(ra[0], ra[1], ra[2], range(130))
    B = oracle.dequant_rows_f64(rb[0], rb[1], rb[2], range(200))
    assert_close(big[:, :200].cpu().numpy(), Cref, A, B)


def sampled_check(oracle, qa, qb, nsample=400, seed=0):
    """Large shapes: compare sampled C entries with float64 dots of the
    oracle's dequantized rows."""
    ac, as_, at = qa.codes.cpu().numpy(), qa.scales.cpu().numpy(), qa.tensor_scale.item()
    bc, bs, bt = qb.codes.cpu().numpy(), qb.scales.cpu().numpy(), qb.tensor_scale.item()
    C = ops().mixfp4_gemm(qa, qb)
    torch.cuda.synchronize()
    rng = np.random.default_rng(seed)
    M, N = C.shape
    ms = np.unique(np.concatenate([[0, M - 1], rng.integers(0, M, 24)]))
    ns = np.unique(np.concatenate([[0, N - 1], rng.integers(0, N, nsample // 24)]))
    A = oracle.dequant_rows_f64(ac, as_, at, ms)
    B = oracle.dequant_rows_f64(bc, bs, bt, ns)
    Cg = C[torch.from_numpy(ms).to(DEV)][:, torch.from_numpy(ns).to(DEV)].cpu().numpy()
    return assert_close(Cg, A @ B.T, A, B)


@pytest.mark.slow
@pytest.mark.parametrize("name", ["attn", "mlp", "decode", "hadamard"])
def test_full_size_workloads(oracle, name):
    wl = synth.workloads()[name]
    o = ops()
    for lin in wl.linears:
        qa = o.mixfp4_quantize(lin.make_x().to(DEV))
        qb = o.mixfp4_quantize(lin.make_w().to(DEV))
        sampled_check(oracle, qa, qb, seed=sum(map(ord, lin.name)))


def test_stream_k_tail(oracle):
    """80 tiles of 256 x 256 with K = 4096: on a GPU with 76 CTA pairs the 4
    tiles past the first wave are split into K slices over all pairs, up to
    a dozen or more pairs adding into one tile of C.  Ragged M and N; whole
    rows and whole columns of C are checked."""
    M, N, K = 2000, 2500, 4096
    x = synth.activations(M, K, 7301, 7302)
    w = synth.weights(N, K, 7303, 0.02, 0.5)
    o = ops()
    qa = o.mixfp4_quantize(x.to(DEV))
    qb = o.mixfp4_quantize(w.to(DEV))
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = o.mixfp4_gemm(qa, qb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    ac, as_, at = qa.codes.cpu().numpy(), qa.scales.cpu().numpy(), qa.tensor_scale.item()
    bc, bs, bt = qb.codes.cpu().numpy(), qb.scales.cpu().numpy(), qb.tensor_scale.item()
    rng = np.random.default_rng(5)
    rows = np.unique(np.concatenate([[0, 255, 256, 1791, 1792, M - 1], rng.integers(0, M, 16)]))
    cols = np.unique(np.concatenate([[0, 255, 256, 2303, 2304, N - 1], rng.integers(0, N, 16)]))
    Cn = C.cpu().numpy()
    A_r = oracle.dequant_rows_f64(ac, as_, at, rows)
    B_c = oracle.dequant_rows_f64(bc, bs, bt, cols)
    B_all = oracle.dequant_rows_f64(bc, bs, bt, range(N))
    assert_close(Cn[rows], A_r @ B_all.T, A_r, B_all)
    A_all = oracle.dequant_rows_f64(ac, as_, at, range(M))
    assert_close(Cn[:, cols], A_all @ B_c.T, A_all, B_c)


@pytest.mark.parametrize("M,N,K", [(2048, 4000, 512), (256, 1000, 512), (300, 600, 1024)])
def test_narrow_tile_widths(oracle, M, N, K):
    """Shapes for which the launcher picks 224- or 192-wide pair tiles (so the
    last wave is full): every element of C against float64 from the oracle's
    dequantized operands."""
    x = synth.activations(M, K, 7401 + M, 7402)
    w = synth.weights(N, K, 7403 + N, 0.02, 0.5)
    o = ops()
    qa, qb = o.mixfp4_quantize(x.to(DEV)), o.mixfp4_quantize(w.to(DEV))
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = o.mixfp4_gemm(qa, qb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    A = oracle.dequant_rows_f64(qa.codes.cpu().numpy(), qa.scales.cpu().numpy(), qa.tensor_scale.item(), range(M))
    B = oracle.dequant_rows_f64(qb.codes.cpu().numpy(), qb.scales.cpu().numpy(), qb.tensor_scale.item(), range(N))
    assert_close(C.cpu().numpy(), A @ B.T, A, B)
