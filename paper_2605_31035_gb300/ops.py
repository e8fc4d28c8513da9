"""Thin ctypes binding over libmixfp4.so (C ABI in include/mixfp4.h).

Each function marshals torch CUDA tensors to device pointers and the current
stream, calls the entry point of the same name, and raises on a nonzero status.
All arithmetic runs in the library's CUDA kernels; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

MODE_MIX, MODE_E2M1_ONLY, MODE_E1M2_ONLY, MODE_FOUR_SIX = 0, 1, 2, 3
SCALE_COMPUTE, SCALE_GIVEN = 0, 1
DTYPE_BF16, DTYPE_F32 = 0, 1
# Candidates of mixfp4_fake_quantize, bit c of the mask.
CAND_E2M1_6, CAND_E1M2, CAND_E2M1_4, CAND_E3M0 = 1, 2, 4, 8

STATUS = {0: "ok", -1: "null pointer", -2: "invalid shape", -3: "misaligned", -4: "unsupported dtype",
          -5: "CUDA error", -6: "device-side wait timed out", -7: "argument out of range"}

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmixfp4.so")
_lib = None


class MixFP4Error(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} failed: {STATUS.get(status, status)} ({status})")
        self.status = status


def lib() -> ctypes.CDLL:
    """Load libmixfp4.so; raise if it has not been built (no fallback exists)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(
                f"{_LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(_LIB_PATH)
        P, I64, I = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        L.mixfp4_quantize.restype = I
        L.mixfp4_quantize.argtypes = [P, I, I64, I64, I64, P, P, P, P, I, I, P]
        L.mixfp4_quantize_rht.restype = I
        L.mixfp4_quantize_rht.argtypes = [P, I, I64, I64, I64, P, P, P, P, P, I, I, P]
        L.mixfp4_quantize_colwise.restype = I
        L.mixfp4_quantize_colwise.argtypes = [P, I, I64, I64, I64, P, P, P, P, I, I, P]
        L.mixfp4_quantize_colwise_rht.restype = I
        L.mixfp4_quantize_colwise_rht.argtypes = [P, I, I64, I64, I64, P, P, P, P, P, I, I, P]
        U64 = ctypes.c_uint64
        L.mixfp4_quantize_sr.restype = I
        L.mixfp4_quantize_sr.argtypes = [P, I, I64, I64, I64, P, P, P, P, I, I, U64, U64, P]
        L.mixfp4_quantize_colwise_sr.restype = I
        L.mixfp4_quantize_colwise_sr.argtypes = [P, I, I64, I64, I64, P, P, P, P, I, I, U64, U64, P]
        L.mixfp4_quantize_2d.restype = I
        L.mixfp4_quantize_2d.argtypes = [P, I, I64, I64, I64, P, P, P, P, I, I, P]
        L.mixfp4_transpose_2d.restype = I
        L.mixfp4_transpose_2d.argtypes = [P, P, I64, I64, P, P, P]
        L.mixfp4_dequantize.restype = I
        L.mixfp4_dequantize.argtypes = [P, P, P, I64, I64, P, P]
        L.mixfp4_gemm.restype = I
        L.mixfp4_gemm.argtypes = [P, P, P, P, P, P, I64, I64, I64, P, I64, P, P]
        L.mixfp4_split_native.restype = I
        L.mixfp4_split_native.argtypes = [P, P, I64, I64, P, P, P, P]
        L.mixfp4_gemm_native.restype = I
        L.mixfp4_gemm_native.argtypes = [P, P, P, P, P, P, P, P, I64, I64, I64, P, I64, P, P]
        L.mixfp4_gemm_native_fewrows.restype = I
        L.mixfp4_gemm_native_fewrows.argtypes = [P, P, P, P, P, P, I64, I64, I64, P, I64, P, P]
        L.mixfp4_fake_quantize.restype = I
        L.mixfp4_fake_quantize.argtypes = [P, I, I64, I64, I64, I, I, P, P, I, P, I, I64, P, P]
        L.mixfp4_selftest_gemm_missed_stage.restype = I
        L.mixfp4_selftest_gemm_missed_stage.argtypes = [P, P, P, P, P, P, I64, I64, I64, P, I64, P,
                                                         ctypes.c_uint64, P]
        L.mixfp4_selftest_bounded_wait.restype = I
        L.mixfp4_selftest_bounded_wait.argtypes = [P, ctypes.c_uint64, P]
        L.mixfp4_status_string.restype = ctypes.c_char_p
        L.mixfp4_status_string.argtypes = [I]
        L.mixfp4_version.restype = I
        L.mixfp4_version.argtypes = []
        _lib = L
    return _lib


def _require(cond: bool, msg: str):
    """Argument check that stays on under python -O (raises ValueError)."""
    if not cond:
        raise ValueError(msg)


def _check_x(x: torch.Tensor):
    _require(isinstance(x, torch.Tensor) and x.is_cuda and x.dtype == torch.bfloat16 and x.dim() == 2
             and x.stride(1) == 1, "x must be a 2-D bf16 CUDA tensor with unit column stride")


def _check_signs(signs):
    _require(signs is None or (signs.dtype == torch.uint8 and signs.numel() == 16 and signs.is_contiguous()
                               and signs.is_cuda), "signs must be 16 contiguous uint8 bytes on the GPU")


def _check_dev(t, device, what: str):
    """t must be a CUDA tensor on `device` (the device of the call's main input)."""
    _require(isinstance(t, torch.Tensor) and t.is_cuda and t.device == device,
             f"{what} must be a CUDA tensor on {device}")


def _check_u8(t, shape, device, what: str):
    _check_dev(t, device, what)
    _require(t.dtype == torch.uint8 and tuple(t.shape) == tuple(shape) and t.is_contiguous(),
             f"{what} must be a dense uint8 tensor of shape {tuple(shape)}")


def _check_scalar_f32(t, device, what: str):
    _check_dev(t, device, what)
    _require(t.dtype == torch.float32 and t.numel() >= 1, f"{what} must hold at least one float32")


def _check_qtensor(q, rows: int, K: int, device, what: str):
    """A MixFP4 operand: codes uint8 [rows, K/2], scales uint8 [rows, K/16], s32 float32, all on `device`."""
    _require(isinstance(q, QTensor), f"{what} must be a QTensor")
    _check_u8(q.codes, (rows, K // 2), device, f"{what}.codes")
    _check_u8(q.scales, (rows, K // 16), device, f"{what}.scales")
    _check_scalar_f32(q.tensor_scale, device, f"{what}.tensor_scale")


def _check_operand(q, what: str):
    """A GEMM operand: a QTensor on a CUDA device, consistent with its own codes shape."""
    _require(isinstance(q, QTensor) and isinstance(q.codes, torch.Tensor) and q.codes.dim() == 2,
             f"{what} must be a QTensor with 2-D codes")
    _check_qtensor(q, q.rows, q.K, q.codes.device, what)


def _check_c(C, M: int, N: int, device):
    """GEMM output: float32 [M, N] on `device`, unit column stride (row stride >= N)."""
    _check_dev(C, device, "out")
    _require(C.dtype == torch.float32 and C.dim() == 2 and tuple(C.shape) == (M, N)
             and (C.stride(1) == 1 or N <= 1) and C.stride(0) >= max(N, 1),
             f"out must be a float32 [{M}, {N}] tensor with unit column stride")


def _check_workspace(ws, device):
    if ws is not None:
        _check_dev(ws, device, "workspace")
        _require(ws.numel() * ws.element_size() >= 4 and ws.is_contiguous(),
                 "workspace must be a dense CUDA tensor of at least 4 bytes")


def _check_status(sw, device):
    if sw is not None:
        _check_dev(sw, device, "status_word")
        _require(sw.numel() >= 1 and sw.element_size() == 4 and not sw.dtype.is_floating_point,
                 "status_word must be a CUDA tensor of 32-bit integers with at least one element")


def _check_given_scale(ts):
    if ts is not None:
        _require(isinstance(ts, torch.Tensor) and ts.numel() == 1, "tensor_scale must be a 1-element tensor")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(fn: str, status: int):
    if status != 0:
        raise MixFP4Error(fn, status)


@dataclass
class QTensor:
    """A MixFP4 tensor: codes [rows, K/2], scales [rows, K/16], s32 (1 float), all on one device."""
    codes: torch.Tensor
    scales: torch.Tensor
    tensor_scale: torch.Tensor

    @property
    def rows(self) -> int:
        return self.codes.shape[0]

    @property
    def K(self) -> int:
        return self.codes.shape[1] * 2


def empty_qtensor(rows: int, K: int, device) -> QTensor:
    return QTensor(torch.empty(rows, K // 2, dtype=torch.uint8, device=device),
                   torch.empty(rows, K // 16, dtype=torch.uint8, device=device),
                   torch.empty(1, dtype=torch.float32, device=device))


def mixfp4_quantize(x: torch.Tensor, mode: int = MODE_MIX, tensor_scale: torch.Tensor | None = None,
                    out: QTensor | None = None, workspace: torch.Tensor | None = None,
                    stream=None) -> QTensor:
    """Quantize a bf16 [rows, K] CUDA tensor (row stride may exceed K).

    With tensor_scale=None the per-tensor scale is computed (max|x| / 2688);
    otherwise the given 1-element fp32 tensor is used as s32.
    """
    _check_x(x)
    rows, K = x.shape
    q = out if out is not None else empty_qtensor(rows, K, x.device)
    _check_qtensor(q, rows, K, x.device, "out")
    _check_given_scale(tensor_scale)
    given = tensor_scale is not None
    if given:
        q.tensor_scale.copy_(tensor_scale.reshape(1))
    ws = None
    if not given:
        ws = workspace if workspace is not None else torch.empty(1, dtype=torch.int32, device=x.device)
        _check_workspace(ws, x.device)
    st = lib().mixfp4_quantize(_ptr(x), DTYPE_BF16, rows, K, x.stride(0), _ptr(q.codes), _ptr(q.scales),
                               _ptr(q.tensor_scale), _ptr(ws), int(mode),
                               SCALE_GIVEN if given else SCALE_COMPUTE, _stream(stream))
    _check("mixfp4_quantize", st)
    return q


def mixfp4_quantize_rht(x: torch.Tensor, signs: torch.Tensor | None = None, mode: int = MODE_MIX,
                        tensor_scale: torch.Tensor | None = None, out: QTensor | None = None,
                        workspace: torch.Tensor | None = None, stream=None) -> QTensor:
    """Rotate every 128-element chunk of each row of a bf16 [rows, K] CUDA tensor
    (sign flips from the 16-byte `signs`, then the normalised Walsh-Hadamard
    transform) and quantize the result; K % 128 == 0."""
    _check_x(x)
    _check_signs(signs)
    rows, K = x.shape
    q = out if out is not None else empty_qtensor(rows, K, x.device)
    _check_qtensor(q, rows, K, x.device, "out")
    _check_given_scale(tensor_scale)
    given = tensor_scale is not None
    if given:
        q.tensor_scale.copy_(tensor_scale.reshape(1))
    ws = None
    if not given:
        ws = workspace if workspace is not None else torch.empty(1, dtype=torch.int32, device=x.device)
        _check_workspace(ws, x.device)
    st = lib().mixfp4_quantize_rht(_ptr(x), DTYPE_BF16, rows, K, x.stride(0), _ptr(signs), _ptr(q.codes),
                                   _ptr(q.scales), _ptr(q.tensor_scale), _ptr(ws), int(mode),
                                   SCALE_GIVEN if given else SCALE_COMPUTE, _stream(stream))
    _check("mixfp4_quantize_rht", st)
    return q


def mixfp4_quantize_colwise(x: torch.Tensor, mode: int = MODE_MIX, tensor_scale: torch.Tensor | None = None,
                            out: QTensor | None = None, workspace: torch.Tensor | None = None,
                            stream=None) -> QTensor:
    """Quantize a bf16 [R, C] CUDA tensor with 16-row blocks down each column
    (the orientation of a GEMM reducing over R): returns the MixFP4 tensor of
    X^T, codes [C, R/2], scales [C, R/16]."""
    _check_x(x)
    R, C = x.shape
    q = out if out is not None else empty_qtensor(C, R, x.device)
    _check_qtensor(q, C, R, x.device, "out")
    _check_given_scale(tensor_scale)
    given = tensor_scale is not None
    if given:
        q.tensor_scale.copy_(tensor_scale.reshape(1))
    ws = None
    if not given:
        ws = workspace if workspace is not None else torch.empty(1, dtype=torch.int32, device=x.device)
        _check_workspace(ws, x.device)
    st = lib().mixfp4_quantize_colwise(_ptr(x), DTYPE_BF16, R, C, x.stride(0), _ptr(q.codes), _ptr(q.scales),
                                       _ptr(q.tensor_scale), _ptr(ws), int(mode),
                                       SCALE_GIVEN if given else SCALE_COMPUTE, _stream(stream))
    _check("mixfp4_quantize_colwise", st)
    return q


def mixfp4_quantize_colwise_rht(x: torch.Tensor, signs: torch.Tensor | None = None, mode: int = MODE_MIX,
                                tensor_scale: torch.Tensor | None = None, out: QTensor | None = None,
                                workspace: torch.Tensor | None = None, stream=None) -> QTensor:
    """Rotate every 128-row chunk of each column of a bf16 [R, C] CUDA tensor and
    quantize down the columns: the MixFP4 tensor of the rotated X^T."""
    _check_x(x)
    _check_signs(signs)
    R, C = x.shape
    q = out if out is not None else empty_qtensor(C, R, x.device)
    _check_qtensor(q, C, R, x.device, "out")
    _check_given_scale(tensor_scale)
    given = tensor_scale is not None
    if given:
        q.tensor_scale.copy_(tensor_scale.reshape(1))
    ws = None
    if not given:
        ws = workspace if workspace is not None else torch.empty(1, dtype=torch.int32, device=x.device)
        _check_workspace(ws, x.device)
    st = lib().mixfp4_quantize_colwise_rht(_ptr(x), DTYPE_BF16, R, C, x.stride(0), _ptr(signs), _ptr(q.codes),
                                           _ptr(q.scales), _ptr(q.tensor_scale), _ptr(ws), int(mode),
                                           SCALE_GIVEN if given else SCALE_COMPUTE, _stream(stream))
    _check("mixfp4_quantize_colwise_rht", st)
    return q


def mixfp4_quantize_sr(x: torch.Tensor, seed: int, offset: int = 0, mode: int = MODE_MIX,
                       tensor_scale: torch.Tensor | None = None, out: QTensor | None = None,
                       workspace: torch.Tensor | None = None, colwise: bool = False, stream=None) -> QTensor:
    """mixfp4_quantize (or, with colwise=True, mixfp4_quantize_colwise) with
    stochastic rounding of the codes drawn from (seed, offset)."""
    _check_x(x)
    rows, K = x.shape
    q = out if out is not None else (empty_qtensor(K, rows, x.device) if colwise else empty_qtensor(rows, K, x.device))
    _check_qtensor(q, K if colwise else rows, rows if colwise else K, x.device, "out")
    _check_given_scale(tensor_scale)
    given = tensor_scale is not None
    if given:
        q.tensor_scale.copy_(tensor_scale.reshape(1))
    ws = None
    if not given:
        ws = workspace if workspace is not None else torch.empty(1, dtype=torch.int32, device=x.device)
        _check_workspace(ws, x.device)
    fn = lib().mixfp4_quantize_colwise_sr if colwise else lib().mixfp4_quantize_sr
    st = fn(_ptr(x), DTYPE_BF16, rows, K, x.stride(0), _ptr(q.codes), _ptr(q.scales), _ptr(q.tensor_scale),
            _ptr(ws), int(mode), SCALE_GIVEN if given else SCALE_COMPUTE, int(seed) & (2 ** 64 - 1),
            int(offset) & (2 ** 64 - 1), _stream(stream))
    _check("mixfp4_quantize_colwise_sr" if colwise else "mixfp4_quantize_sr", st)
    return q


def mixfp4_quantize_2d(x: torch.Tensor, mode: int = MODE_MIX, tensor_scale: torch.Tensor | None = None,
                       out: QTensor | None = None, workspace: torch.Tensor | None = None,
                       stream=None) -> QTensor:
    """Quantize a bf16 [rows, K] CUDA tensor with 16 x 16 blocks (one scale
    and format per tile, repeated on the tile's rows)."""
    _check_x(x)
    rows, K = x.shape
    q = out if out is not None else empty_qtensor(rows, K, x.device)
    _check_qtensor(q, rows, K, x.device, "out")
    _check_given_scale(tensor_scale)
    given = tensor_scale is not None
    if given:
        q.tensor_scale.copy_(tensor_scale.reshape(1))
    ws = None
    if not given:
        ws = workspace if workspace is not None else torch.empty(1, dtype=torch.int32, device=x.device)
        _check_workspace(ws, x.device)
    st = lib().mixfp4_quantize_2d(_ptr(x), DTYPE_BF16, rows, K, x.stride(0), _ptr(q.codes), _ptr(q.scales),
                                  _ptr(q.tensor_scale), _ptr(ws), int(mode),
                                  SCALE_GIVEN if given else SCALE_COMPUTE, _stream(stream))
    _check("mixfp4_quantize_2d", st)
    return q


def mixfp4_transpose_2d(q: QTensor, out: QTensor | None = None, stream=None) -> QTensor:
    """The transpose of a 2D-quantized tensor (rows and K multiples of 16);
    the tensor scale is shared with the input."""
    _check_operand(q, "q")
    t = out if out is not None else QTensor(
        torch.empty(q.K, q.rows // 2, dtype=torch.uint8, device=q.codes.device),
        torch.empty(q.K, q.rows // 16, dtype=torch.uint8, device=q.codes.device), q.tensor_scale)
    _check_u8(t.codes, (q.K, q.rows // 2), q.codes.device, "out.codes")
    _check_u8(t.scales, (q.K, q.rows // 16), q.codes.device, "out.scales")
    st = lib().mixfp4_transpose_2d(_ptr(q.codes), _ptr(q.scales), q.rows, q.K, _ptr(t.codes), _ptr(t.scales),
                                   _stream(stream))
    _check("mixfp4_transpose_2d", st)
    return t


def mixfp4_fake_quantize(x: torch.Tensor, candidates: int, block: int = 16, out_dtype=torch.float32,
                         tensor_scale: torch.Tensor | None = None, want_choice: bool = True,
                         out: torch.Tensor | None = None, choice: torch.Tensor | None = None,
                         workspace: torch.Tensor | None = None, stream=None):
    """Quantize-dequantize of a bf16 [rows, K] CUDA tensor under a candidate
    set (mask of CAND_*) and block size (8, 16, 32, 64): returns (out
    [rows, K] of out_dtype (float32 or bfloat16), choice uint8 [rows, K/block]
    or None, tensor_scale)."""
    _check_x(x)
    _require(out_dtype in (torch.float32, torch.bfloat16), "out_dtype must be torch.float32 or torch.bfloat16")
    _require(block in (8, 16, 32, 64), "block must be 8, 16, 32 or 64")
    rows, K = x.shape
    o = out if out is not None else torch.empty(rows, K, dtype=out_dtype, device=x.device)
    _check_dev(o, x.device, "out")
    _require(o.dtype == out_dtype and o.dim() == 2 and o.shape == x.shape and o.stride(1) == 1,
             "out must be a [rows, K] tensor of out_dtype with unit column stride")
    ch = None
    if want_choice:
        ch = choice if choice is not None else torch.empty(rows, K // block, dtype=torch.uint8,
                                                           device=x.device)
        _check_dev(ch, x.device, "choice")
        _require(ch.dtype == torch.uint8 and ch.is_contiguous() and ch.numel() == rows * (K // block),
                 "choice must be a dense uint8 [rows, K / block] tensor")
    _check_given_scale(tensor_scale)
    ts = torch.empty(1, dtype=torch.float32, device=x.device)
    given = tensor_scale is not None
    if given:
        ts.copy_(tensor_scale.reshape(1))
    ws = None
    if not given:
        ws = workspace if workspace is not None else torch.empty(1, dtype=torch.int32, device=x.device)
        _check_workspace(ws, x.device)
    st = lib().mixfp4_fake_quantize(_ptr(x), DTYPE_BF16, rows, K, x.stride(0), int(candidates), int(block),
                                    _ptr(ts), _ptr(ws), SCALE_GIVEN if given else SCALE_COMPUTE, _ptr(o),
                                    DTYPE_F32 if out_dtype == torch.float32 else DTYPE_BF16, o.stride(0),
                                    _ptr(ch), _stream(stream))
    _check("mixfp4_fake_quantize", st)
    return o, ch, ts


def mixfp4_dequantize(q: QTensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    _check_operand(q, "q")
    o = out if out is not None else torch.empty(q.rows, q.K, dtype=torch.float32, device=q.codes.device)
    _check_dev(o, q.codes.device, "out")
    _require(o.dtype == torch.float32 and tuple(o.shape) == (q.rows, q.K) and o.is_contiguous(),
             "out must be a dense float32 [rows, K] tensor")
    st = lib().mixfp4_dequantize(_ptr(q.codes), _ptr(q.scales), _ptr(q.tensor_scale), q.rows, q.K,
                                 _ptr(o), _stream(stream))
    _check("mixfp4_dequantize", st)
    return o


def mixfp4_gemm(a: QTensor, b: QTensor, out: torch.Tensor | None = None,
                status_word: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """C = A_deq . B_deq^T in fp32; a is M x K, b is N x K."""
    _check_operand(a, "a")
    _check_operand(b, "b")
    _require(a.K == b.K and a.codes.device == b.codes.device, "operands must share K and device")
    M, N, K = a.rows, b.rows, a.K
    C = out if out is not None else torch.empty(M, N, dtype=torch.float32, device=a.codes.device)
    _check_c(C, M, N, a.codes.device)
    _check_status(status_word, a.codes.device)
    st = lib().mixfp4_gemm(_ptr(a.codes), _ptr(a.scales), _ptr(a.tensor_scale),
                           _ptr(b.codes), _ptr(b.scales), _ptr(b.tensor_scale),
                           M, N, K, _ptr(C), C.stride(0), _ptr(status_word), _stream(stream))
    _check("mixfp4_gemm", st)
    return C


@dataclass
class NativeTensor:
    """A MixFP4 tensor as native E2M1 operands: main and residual codes
    [rows, K/2] (residual None when the tensor has no E1M2 block), ue4m3 block
    scales in the tensor core's tiled layout, and s32."""
    main: torch.Tensor
    res: torch.Tensor | None
    sf: torch.Tensor
    tensor_scale: torch.Tensor

    @property
    def rows(self) -> int:
        return self.main.shape[0]

    @property
    def K(self) -> int:
        return self.main.shape[1] * 2


def sf_tiled_bytes(rows: int, K: int) -> int:
    return ((rows + 255) // 256) * 256 * (K // 16)


def _check_native(t, rows: int, K: int, device, what: str):
    """Native operand: main (and residual, if any) uint8 [rows, K/2], tiled scales, s32, all on `device`."""
    _check_u8(t.main, (rows, K // 2), device, f"{what}.main")
    if t.res is not None:
        _check_u8(t.res, (rows, K // 2), device, f"{what}.res")
    _check_dev(t.sf, device, f"{what}.sf")
    _require(t.sf.dtype == torch.uint8 and t.sf.is_contiguous() and t.sf.numel() >= sf_tiled_bytes(rows, K),
             f"{what}.sf must be a dense uint8 buffer of at least {sf_tiled_bytes(rows, K)} bytes")
    _check_scalar_f32(t.tensor_scale, device, f"{what}.tensor_scale")


def mixfp4_split_native(q: QTensor, keep_residual: bool = True, out: NativeTensor | None = None,
                        stream=None) -> NativeTensor:
    """Split a MixFP4 tensor into native E2M1 operands.  keep_residual=False
    drops the residual, which is exact only for tensors without E1M2 blocks
    (MODE_E2M1_ONLY).  `out` (with a residual buffer) is reused when given."""
    _check_operand(q, "q")
    dev = q.codes.device
    if out is not None:
        _require(out.res is not None, "out must carry a residual buffer")
        _check_native(out, q.rows, q.K, dev, "out")
        main, res, sf = out.main, out.res, out.sf
    else:
        main = torch.empty_like(q.codes)
        res = torch.empty_like(q.codes)
        sf = torch.empty(sf_tiled_bytes(q.rows, q.K), dtype=torch.uint8, device=dev)
    st = lib().mixfp4_split_native(_ptr(q.codes), _ptr(q.scales), q.rows, q.K, _ptr(main), _ptr(res), _ptr(sf),
                                   _stream(stream))
    _check("mixfp4_split_native", st)
    return NativeTensor(main, res if keep_residual else None, sf, q.tensor_scale)


def mixfp4_gemm_native(a: NativeTensor, b: NativeTensor, out: torch.Tensor | None = None,
                       status_word: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """C = A . B^T on the block-scaled FP4 tensor path; a is M x K, b is N x K."""
    _require(isinstance(a, NativeTensor) and isinstance(b, NativeTensor) and a.main.dim() == 2
             and b.main.dim() == 2, "operands must be NativeTensors")
    dev = a.main.device
    _check_native(a, a.rows, a.K, dev, "a")
    _check_native(b, b.rows, b.K, dev, "b")
    _require(a.K == b.K, "operands must share K")
    M, N, K = a.rows, b.rows, a.K
    C = out if out is not None else torch.empty(M, N, dtype=torch.float32, device=a.main.device)
    _check_c(C, M, N, dev)
    _check_status(status_word, dev)
    st = lib().mixfp4_gemm_native(_ptr(a.main), _ptr(a.res), _ptr(a.sf), _ptr(a.tensor_scale),
                                  _ptr(b.main), _ptr(b.res), _ptr(b.sf), _ptr(b.tensor_scale),
                                  M, N, K, _ptr(C), C.stride(0), _ptr(status_word), _stream(stream))
    _check("mixfp4_gemm_native", st)
    return C


def mixfp4_gemm_native_fewrows(a: QTensor, b: QTensor, out: torch.Tensor | None = None,
                               status_word: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """C = A_deq . B_deq^T for a with at most 64 rows, on the block-scaled FP4
    tensor path: the stored codes are the main E2M1 operands, their residual
    rows and scale tiles are formed on the fly."""
    _check_operand(a, "a")
    _check_operand(b, "b")
    _require(a.K == b.K and a.rows <= 64 and a.codes.device == b.codes.device,
             "operands must share K and device, and A have at most 64 rows")
    M, N, K = a.rows, b.rows, a.K
    C = out if out is not None else torch.empty(M, N, dtype=torch.float32, device=a.codes.device)
    _check_c(C, M, N, a.codes.device)
    _check_status(status_word, a.codes.device)
    st = lib().mixfp4_gemm_native_fewrows(_ptr(a.codes), _ptr(a.scales), _ptr(a.tensor_scale),
                                          _ptr(b.codes), _ptr(b.scales), _ptr(b.tensor_scale),
                                          M, N, K, _ptr(C), C.stride(0), _ptr(status_word), _stream(stream))
    _check("mixfp4_gemm_native_fewrows", st)
    return C


def selftest_bounded_wait(limit_ns: int = 20_000_000, stream=None) -> int:
    """Run the bounded-wait self-test; returns the status bits (0xE when healthy)."""
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    _check("mixfp4_selftest_bounded_wait",
           lib().mixfp4_selftest_bounded_wait(_ptr(status), int(limit_ns), _stream(stream)))
    torch.cuda.synchronize()
    return int(status.item())


def selftest_gemm_missed_stage(a: QTensor, b: QTensor, out: torch.Tensor, limit_ns: int = 5_000_000,
                               stream=None) -> int:
    """Run the pair GEMM kernel with its first code stage withheld and short
    wait limits; returns the status bits it reported (nonzero when the
    failure path worked).  `out` is not written."""
    _check_operand(a, "a")
    _check_operand(b, "b")
    _require(a.K == b.K and a.codes.device == b.codes.device, "operands must share K and device")
    _check_c(out, a.rows, b.rows, a.codes.device)
    status = torch.zeros(1, dtype=torch.int32, device=a.codes.device)
    _check("mixfp4_selftest_gemm_missed_stage",
           lib().mixfp4_selftest_gemm_missed_stage(_ptr(a.codes), _ptr(a.scales), _ptr(a.tensor_scale),
                                                   _ptr(b.codes), _ptr(b.scales), _ptr(b.tensor_scale), a.rows,
                                                   b.rows, a.K, _ptr(out), out.stride(0), _ptr(status),
                                                   int(limit_ns), _stream(stream)))
    torch.cuda.synchronize(a.codes.device)
    return int(status.item())


def linear(x: torch.Tensor, w_q: QTensor, mode: int = MODE_MIX, stream=None) -> torch.Tensor:
    """W4A4 linear: quantize the activations online, then the MixFP4 GEMM with
    pre-quantized weights.  Returns x_deq . w_deq^T in fp32."""
    return mixfp4_gemm(mixfp4_quantize(x, mode, stream=stream), w_q, stream=stream)
