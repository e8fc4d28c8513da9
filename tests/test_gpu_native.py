"""GPU parity of the native block-scaled FP4 variant (split + kind::mxf4nvf4 GEMM).

The split is byte work: main codes, residual codes and tiled scales must equal
the oracle's split bit for bit.  The GEMM computes the same C as the MixFP4
GEMM, so it is held to the same criterion against the float64 oracle of the
MixFP4 operands: max |C_gpu - C_oracle| / (|A_deq| . |B_deq|^T) <= 1e-5, and
exact zeros where that denominator is 0.  Every call goes through the C ABI.
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


@pytest.mark.parametrize("rows,K,mode", [(1, 64, 0), (37, 192, 0), (300, 512, 0), (130, 256, 1), (64, 320, 2)])
def test_split_bit_exact(oracle, rows, K, mode):
    x = synth.activations(rows, K, 8100 + rows, 8101)
    q, ref = quant_both(oracle, x, mode)
    nt = ops().mixfp4_split_native(q)
    torch.cuda.synchronize()
    main, res, sf = oracle.split_native(ref[0], ref[1])
    assert np.array_equal(nt.main.cpu().numpy(), main)
    assert np.array_equal(nt.res.cpu().numpy(), res)
    assert np.array_equal(nt.sf.cpu().numpy(), sf)


def native_check(oracle, x, w, mode_a=0, mode_b=0):
    qa, ra = quant_both(oracle, x, mode_a)
    qb, rb = quant_both(oracle, w, mode_b)
    o = ops()
    na = o.mixfp4_split_native(qa, keep_residual=mode_a != 1)
    nb = o.mixfp4_split_native(qb, keep_residual=mode_b != 1)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = o.mixfp4_gemm_native(na, nb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    Cref = oracle.gemm_f64(ra, rb)
    A = oracle.dequant_rows_f64(ra[0], ra[1], ra[2], range(x.shape[0]))
    B = oracle.dequant_rows_f64(rb[0], rb[1], rb[2], range(w.shape[0]))
    return assert_close(C.cpu().numpy(), Cref, A, B)


@pytest.mark.parametrize("M,N,K", [(256, 256, 256), (200, 300, 512), (1, 1, 256), (129, 257, 768),
                                   (64, 520, 1280), (300, 16, 256), (512, 768, 2048)])
def test_native_gemm_mix(oracle, M, N, K):
    """Both operands MixFP4 with E1M2 blocks: four products per K step.  One
    tile, ragged M and N tails, one to eight stages, ring wrap."""
    x = synth.activations(M, K, 8200 + M, 8201 + M)
    w = synth.weights(N, K, 8202 + N, 0.02, 0.5)
    native_check(oracle, x, w)


@pytest.mark.parametrize("mode_a,mode_b", [(1, 1), (0, 1), (1, 0), (2, 2), (2, 0)])
def test_native_gemm_modes(oracle, mode_a, mode_b):
    """E2M1-only operands drop their residual (one or two products per K step);
    E1M2-only operands keep it."""
    x = synth.activations(200, 768, 8300, 8301)
    w = synth.weights(330, 768, 8302, 0.02, 0.5)
    native_check(oracle, x, w, mode_a, mode_b)


def test_native_zero_operand(oracle):
    x = torch.zeros(128, 512, dtype=torch.bfloat16)
    w = synth.weights(256, 512, 8400, 0.02)
    o = ops()
    qa, _ = quant_both(oracle, x)
    qb, _ = quant_both(oracle, w)
    C = o.mixfp4_gemm_native(o.mixfp4_split_native(qa), o.mixfp4_split_native(qb))
    torch.cuda.synchronize()
    assert torch.count_nonzero(C).item() == 0


def test_native_matches_decoding_gemm(oracle):
    """Same operands through both GEMMs: each within the tolerance of the
    float64 oracle, so within twice of each other."""
    x = synth.activations(384, 1024, 8500, 8501)
    w = synth.weights(640, 1024, 8502, 0.02, 0.5)
    o = ops()
    qa, ra = quant_both(oracle, x)
    qb, rb = quant_both(oracle, w)
    C1 = o.mixfp4_gemm(qa, qb).cpu().numpy()
    C2 = o.mixfp4_gemm_native(o.mixfp4_split_native(qa), o.mixfp4_split_native(qb)).cpu().numpy()
    A = oracle.dequant_rows_f64(ra[0], ra[1], ra[2], range(384))
    B = oracle.dequant_rows_f64(rb[0], rb[1], rb[2], range(640))
    D = np.abs(A) @ np.abs(B).T
    assert np.all(np.abs(C1.astype(np.float64) - C2) <= 2 * TOL * D)


def test_native_stream_k_tail(oracle):
    """80 tiles of 256 x 256 with K = 4096 on 76 CTA pairs: the last wave is
    split into K slices added into C.  Whole rows and columns are checked."""
    M, N, K = 2000, 2500, 4096
    x = synth.activations(M, K, 8601, 8602)
    w = synth.weights(N, K, 8603, 0.02, 0.5)
    o = ops()
    qa, qb = o.mixfp4_quantize(x.to(DEV)), o.mixfp4_quantize(w.to(DEV))
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = o.mixfp4_gemm_native(o.mixfp4_split_native(qa), o.mixfp4_split_native(qb), status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    ac, as_, at = qa.codes.cpu().numpy(), qa.scales.cpu().numpy(), qa.tensor_scale.item()
    bc, bs, bt = qb.codes.cpu().numpy(), qb.scales.cpu().numpy(), qb.tensor_scale.item()
    rng = np.random.default_rng(6)
    rows = np.unique(np.concatenate([[0, 255, 256, 1791, 1792, M - 1], rng.integers(0, M, 16)]))
    cols = np.unique(np.concatenate([[0, 255, 256, 2303, 2304, N - 1], rng.integers(0, N, 16)]))
    Cn = C.cpu().numpy()
    A_r = oracle.dequant_rows_f64(ac, as_, at, rows)
    B_all = oracle.dequant_rows_f64(bc, bs, bt, range(N))
    assert_close(Cn[rows], A_r @ B_all.T, A_r, B_all)
    A_all = oracle.dequant_rows_f64(ac, as_, at, range(M))
    B_c = oracle.dequant_rows_f64(bc, bs, bt, cols)
    assert_close(Cn[:, cols], A_all @ B_c.T, A_all, B_c)


@pytest.mark.slow
@pytest.mark.parametrize("name", ["attn", "mlp", "hadamard"])
def test_native_full_size_workloads(oracle, name):
    wl = synth.workloads()[name]
    o = ops()
    for lin in wl.linears:
        qa = o.mixfp4_quantize(lin.make_x().to(DEV))
        qb = o.mixfp4_quantize(lin.make_w().to(DEV))
        C = o.mixfp4_gemm_native(o.mixfp4_split_native(qa), o.mixfp4_split_native(qb))
        torch.cuda.synchronize()
        rng = np.random.default_rng(sum(map(ord, lin.name)))
        M, N = C.shape
        ms = np.unique(np.concatenate([[0, M - 1], rng.integers(0, M, 24)]))
        ns = np.unique(np.concatenate([[0, N - 1], rng.integers(0, N, 16)]))
        A = oracle.dequant_rows_f64(qa.codes.cpu().numpy(), qa.scales.cpu().numpy(), qa.tensor_scale.item(), ms)
        B = oracle.dequant_rows_f64(qb.codes.cpu().numpy(), qb.scales.cpu().numpy(), qb.tensor_scale.item(), ns)
        Cg = C[torch.from_numpy(ms).to(DEV)][:, torch.from_numpy(ns).to(DEV)].cpu().numpy()
        assert_close(Cg, A @ B.T, A, B)


@pytest.mark.parametrize("M,N,K", [(1, 128, 256), (16, 300, 768), (33, 1000, 512), (64, 256, 2048), (7, 129, 1280),
                                   (20, 384, 1024), (32, 640, 4352)])
def test_fewrows_native_gemm(oracle, M, N, K):
    """The few-row native path splits the stored MixFP4 operands on the fly:
    one or several 128-row weight groups, a ragged last group, activation
    rows from 1 to 64 (all three activation tile heights: up to 16, 32 and 64
    rows), several K slices per CTA, a run crossing a 4096-K accumulation
    chunk."""
    x = synth.activations(M, K, 8600 + M, 8601)
    w = synth.weights(N, K, 8602 + N, 0.02, 0.5)
    qa, ra = quant_both(oracle, x)
    qb, rb = quant_both(oracle, w)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    C = ops().mixfp4_gemm_native_fewrows(qa, qb, status_word=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    Cref = oracle.gemm_f64(ra, rb)
    A = oracle.dequant_rows_f64(ra[0], ra[1], ra[2], range(M))
    B = oracle.dequant_rows_f64(rb[0], rb[1], rb[2], range(N))
    assert_close(C.cpu().numpy(), Cref, A, B)


def test_fewrows_native_modes_and_ldc(oracle):
    """E2M1-only and E1M2-only operands (all-main and all-split blocks) and a
    padded output row stride."""
    o = ops()
    for mode_a, mode_b in ((1, 1), (2, 2), (0, 2)):
        x = synth.activations(16, 512, 8700 + mode_a, 8701)
        w = synth.weights(256, 512, 8702 + mode_b, 0.02, 0.5)
        qa, ra = quant_both(oracle, x, mode_a)
        qb, rb = quant_both(oracle, w, mode_b)
        Cbuf = torch.full((16, 300), 7.0, dtype=torch.float32, device=DEV)
        C = o.mixfp4_gemm_native_fewrows(qa, qb, out=Cbuf[:, :256])
        torch.cuda.synchronize()
        assert torch.all(Cbuf[:, 256:] == 7.0)
        A = oracle.dequant_rows_f64(ra[0], ra[1], ra[2], range(16))
        B = oracle.dequant_rows_f64(rb[0], rb[1], rb[2], range(256))
        assert_close(C.cpu().numpy(), oracle.gemm_f64(ra, rb), A, B)


@pytest.mark.slow
def test_fewrows_native_decode_shape(oracle):
    """The decode-shaped linear (16 x 8192 . 28672 x 8192) against sampled
    weight rows of the float64 oracle."""
    lin = synth.workloads()["decode"].linears[0]
    x, w = lin.make_x(), lin.make_w()
    qa, ra = quant_both(oracle, x)
    qb = ops().mixfp4_quantize(w.to(DEV))
    C = ops().mixfp4_gemm_native_fewrows(qa, qb)
    torch.cuda.synchronize()
    rng = np.random.default_rng(8)
    rows = np.unique(np.concatenate([[0, 28671], rng.integers(0, 28672, 40)]))
    s32 = float(qb.tensor_scale.item())
    rb = oracle.quantize(synth.bf16_bits(w[torch.from_numpy(rows)]), s32=s32)
    assert np.array_equal(qb.codes[torch.from_numpy(rows).to(DEV)].cpu().numpy(), rb[0])
    Cref = oracle.gemm_f64(ra, rb)
    A = oracle.dequant_rows_f64(ra[0], ra[1], ra[2], range(16))
    B = oracle.dequant_rows_f64(rb[0], rb[1], rb[2], range(len(rows)))
    assert_close(C.cpu().numpy()[:, rows], Cref, A, B)
