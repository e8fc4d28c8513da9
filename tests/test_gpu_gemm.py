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


@pytest.mark.parametrize("K", [512, 8192])
def test_unaligned_output(oracle, K):
    """C whose base and row stride are not 16-byte aligned: the epilogue
    cannot use TMA stores of C and writes element by element (stores for the
    first accumulation chunk, atomic adds for the second at K = 8192); the
    columns around the output are untouched."""
    x = synth.activations(130, K, 31 + K, 32)
    w = synth.weights(200, K, 33 + K, 0.02)
    qa, ra = quant_both(oracle, x)
    qb, rb = quant_both(oracle, w)
    big = torch.full((130, 203), -1.0, device=DEV)
    out = big[:, 1:201]  # base 4 bytes past a 16-byte boundary, ldc = 203
    ops().mixfp4_gemm(qa, qb, out=out)
    torch.cuda.synchronize()
    assert torch.all(big[:, 0] == -1.0) and torch.all(big[:, 201:] == -1.0)
    Cref = oracle.gemm_f64(ra, rb)
    A = oracle.dequant_rows_f64(ra[0], ra[1], ra[2], range(130))
    B = oracle.dequant_rows_f64(rb[0], rb[1], rb[2], range(200))
    assert_close(out.cpu().numpy(), Cref, A, B)


def rows_cols_check(oracle, qa, qb, C, rows, cols, block=2048):
    """Whole rows of C against every column and whole columns against every
    row: float64 dots of the oracle's dequantized operands, the full operand
    dequantized block by block to bound host memory."""
    ac, as_, at = qa.codes.cpu().numpy(), qa.scales.cpu().numpy(), qa.tensor_scale.item()
    bc, bs, bt = qb.codes.cpu().numpy(), qb.scales.cpu().numpy(), qb.tensor_scale.item()
    M, N = C.shape
    rows = np.unique(np.asarray(rows, dtype=np.int64).clip(0, M - 1))
    cols = np.unique(np.asarray(cols, dtype=np.int64).clip(0, N - 1))
    C_rows = C[torch.from_numpy(rows).to(C.device)].cpu().numpy()
    C_cols = C[:, torch.from_numpy(cols).to(C.device)].cpu().numpy()
    A_r = oracle.dequant_rows_f64(ac, as_, at, rows)
    B_c = oracle.dequant_rows_f64(bc, bs, bt, cols)
    worst = 0.0
    for n0 in range(0, N, block):
        B_blk = oracle.dequant_rows_f64(bc, bs, bt, range(n0, min(N, n0 + block)))
        worst = max(worst, assert_close(C_rows[:, n0:n0 + block], A_r @ B_blk.T, A_r, B_blk))
    for m0 in range(0, M, block):
        A_blk = oracle.dequant_rows_f64(ac, as_, at, range(m0, min(M, m0 + block)))
        worst = max(worst, assert_close(C_cols[m0:m0 + block], A_blk @ B_c.T, A_blk, B_c))
    return worst


def boundary_indices(n, tile_widths=(224, 192, 256), extra=16, seed=0):
    """First and last index, both sides of every candidate tile edge near the
    start and the end, plus random indices."""
    rng = np.random.default_rng(seed)
    idx = [0, n - 1]
    for w in tile_widths:
        for e in (w, 2 * w, (n // w) * w):
            idx += [e - 1, e]
    return np.concatenate([np.array(idx), rng.integers(0, n, extra)])


@pytest.mark.slow
@pytest.mark.parametrize("name", ["attn", "mlp", "decode", "hadamard"])
def test_full_size_workloads(oracle, name):
    """Every linear of the workload at full size, in the launch configuration
    the bench times: whole rows of C (every column) and whole columns (every
    row) against float64 from the oracle's dequantized operands."""
    wl = synth.workloads()[name]
    o = ops()
    for lin in wl.linears:
        qa = o.mixfp4_quantize(lin.make_x().to(DEV))
        qb = o.mixfp4_quantize(lin.make_w().to(DEV))
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        C = o.mixfp4_gemm(qa, qb, status_word=status)
        torch.cuda.synchronize()
        assert status.item() == 0
        seed = sum(map(ord, lin.name))
        rows_cols_check(oracle, qa, qb, C, boundary_indices(lin.M, seed=seed), boundary_indices(lin.N, seed=seed + 1))


def coinciding_outliers(M, N, K, seed):
    """Activations and weights whose x50 outlier channels are the same 1 % of
    K (weights without row scales): the products of two outliers dominate
    every dot product, so the accumulator runs far from the typical partial
    sum -- the case in which a long fp32 accumulation on the tensor cores
    drifts furthest (relative to |A|.|B|) from the exact result."""
    x = synth.activations(M, K, seed, 3000 + K)
    w = synth.weights(N, K, seed + 100, 0.02, None, 3000 + K)
    return x, w


@pytest.mark.parametrize("K", [14336, 28672])
@pytest.mark.parametrize("M", [256, 16, 600])
def test_long_k_accumulation_bound(oracle, M, K):
    """Long reductions on outlier-heavy operands stay within 1e-5 of |A|.|B|:
    the GEMMs cut every TMEM accumulation into chunks of at most 4096 K and
    add the chunks into C in fp32.  M = 256 and 600 take the CTA-pair kernel
    (600: ragged, several tiles), M = 16 the few-row kernel; the native FP4
    GEMM (and, for M = 16, its few-row form) on the same operands; every
    element of C is checked."""
    N = 512
    x, w = coinciding_outliers(M, N, K, 9500 + K + M)
    o = ops()
    qa, qb = o.mixfp4_quantize(x.to(DEV)), o.mixfp4_quantize(w.to(DEV))
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = o.mixfp4_gemm(qa, qb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    A = oracle.dequant_rows_f64(qa.codes.cpu().numpy(), qa.scales.cpu().numpy(), qa.tensor_scale.item(), range(M))
    B = oracle.dequant_rows_f64(qb.codes.cpu().numpy(), qb.scales.cpu().numpy(), qb.tensor_scale.item(), range(N))
    Cref = A @ B.T
    assert_close(C.cpu().numpy(), Cref, A, B)
    # The native block-scaled FP4 path accumulates on the same tensor cores.
    Cn = o.mixfp4_gemm_native(o.mixfp4_split_native(qa), o.mixfp4_split_native(qb), status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    assert_close(Cn.cpu().numpy(), Cref, A, B)
    if M <= 64:
        Cf = o.mixfp4_gemm_native_fewrows(qa, qb, status_word=status)
        torch.cuda.synchronize()
        assert status.item() == 0
        assert_close(Cf.cpu().numpy(), Cref, A, B)


@pytest.mark.slow
def test_long_k_full_size_down_projection(oracle):
    """The MLP down projection shape (4096 x 4096, K = 14336) with coinciding
    outlier channels: whole rows and columns of C, including the stream-K
    tail and the four accumulation chunks of every whole tile."""
    M = N = 4096
    K = 14336
    x, w = coinciding_outliers(M, N, K, 9700)
    o = ops()
    qa, qb = o.mixfp4_quantize(x.to(DEV)), o.mixfp4_quantize(w.to(DEV))
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = o.mixfp4_gemm(qa, qb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    rows_cols_check(oracle, qa, qb, C, boundary_indices(M, seed=3), boundary_indices(N, seed=4))


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


@pytest.mark.slow
def test_stream_k_chunked_segments(oracle):
    """126 tiles of 256 x 256 with K = 14336 (56 K slices): on 76 CTA pairs
    the 50 tiles past the first wave are shared out as about 37 K slices per
    pair, so stream-K shares cross accumulation-chunk edges (every 16 K
    slices) and are cut there; whole tiles run as four chunks.  Whole rows
    and columns are checked."""
    M, N, K = 768, 10528, 14336
    x, w = coinciding_outliers(M, N, K, 9800)
    o = ops()
    qa, qb = o.mixfp4_quantize(x.to(DEV)), o.mixfp4_quantize(w.to(DEV))
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = o.mixfp4_gemm(qa, qb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    rows_cols_check(oracle, qa, qb, C, boundary_indices(M, seed=5), boundary_indices(N, seed=6))
