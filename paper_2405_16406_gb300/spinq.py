"""Python binding of the C ABI in include/spinq.h (libspinq.so, sm_103a).

Argument marshalling only: every step of the hot path runs in the library's
CUDA kernels.  PyTorch supplies device memory and the current stream.  There
is no fallback: importing this module raises if libspinq.so is missing, and
every call raises ``SpinqError`` on a non-OK status.

Low-level names mirror the C entry points (``spinq_rotate_quant_act`` ...) and
take raw pointers; the tensor-level helpers below them (``rotate_quant_act``
...) allocate the outputs with torch and call the same entry points.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libspinq.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(
        f"libspinq.so not found at {LIB_PATH}; build it with "
        "`python -m paper_2405_16406_gb300.build` (the CUDA path has no fallback)")

_lib = ctypes.CDLL(LIB_PATH)

SPINQ_OK, SPINQ_EINVAL, SPINQ_EUNSUPPORTED, SPINQ_ECUDA, SPINQ_ETIMEOUT, SPINQ_ESCRATCH = range(6)
SPINQ_NOALLOC_SCRATCH_BYTES = 8 << 20   # include/spinq.h
SPINQ_PER_TOKEN, SPINQ_PER_CHANNEL, SPINQ_PER_GROUP = range(3)
SPINQ_GEMM_AUTO, SPINQ_GEMM_TILE128, SPINQ_GEMM_TILE256, SPINQ_GEMM_PAIR, SPINQ_GEMM_GEMV, SPINQ_GEMM_SPLITK, SPINQ_GEMM_TCGEMV = range(7)

EXPORTED = (
    "spinq_rotate_quant_act", "spinq_quant_weight", "spinq_w4a4_gemm", "spinq_rotate_quant_kv",
    "spinq_status_string", "spinq_device_status", "spinq_version", "spinq_w4a4_gemm_workspace_bytes",
    "spinq_w4a4_gemm_splitk", "spinq_w4a4_gemm_noalloc", "spinq_gemm_select_kernel", "spinq_gemm_split_k",
    "spinq_w4a4_gemm_plan", "spinq_w4a4_gemm_splitk_plan", "spinq_cayley_step",
    "spinq_rotate_quant_act8", "spinq_quant_weight8", "spinq_fp8_gemm", "spinq_w4a8_gemm",
    "spinq_rope_rotate_quant_kv", "spinq_decode_attention_workspace_bytes", "spinq_decode_attention_kv4",
    "spinq_rotate_quant_act_signed", "spinq_quant_weight_signed", "spinq_rotated_linear_workspace_bytes",
    "spinq_rotated_linear", "spinq_debug_set_wait_limit_ns", "spinq_debug_fail_launches",
    "spinq_debug_stall_launches",
)
SPINQ_FMT_INT8_PLANES, SPINQ_FMT_E4M3, SPINQ_FMT_INT4_BYTES = 1, 2, 3


class QuantCfg(ctypes.Structure):
    _fields_ = [("bits", ctypes.c_int32), ("symmetric", ctypes.c_int32),
                ("granularity", ctypes.c_int32), ("group_size", ctypes.c_int32),
                ("clip_ratio", ctypes.c_float)]


class HadCfg(ctypes.Structure):
    _fields_ = [("n_small", ctypes.c_int32), ("n_pow2", ctypes.c_int32)]


class SpinqError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {_lib.spinq_status_string(status).decode()}")


_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_lib.spinq_status_string.restype = ctypes.c_char_p
_lib.spinq_status_string.argtypes = [ctypes.c_int]
_lib.spinq_version.restype = ctypes.c_char_p
_lib.spinq_version.argtypes = []
_lib.spinq_device_status.restype = ctypes.c_int
_lib.spinq_device_status.argtypes = [ctypes.POINTER(ctypes.c_int32)]
_lib.spinq_rotate_quant_act.restype = ctypes.c_int
_lib.spinq_rotate_quant_act.argtypes = [_P, _I64, _I64, _I64, ctypes.POINTER(HadCfg),
                                        ctypes.POINTER(QuantCfg), _P, _P, _P, _P]
_lib.spinq_quant_weight.restype = ctypes.c_int
_lib.spinq_quant_weight.argtypes = [_P, _I64, _I64, ctypes.POINTER(HadCfg), ctypes.POINTER(QuantCfg),
                                    _P, _P, _P, _P]
_lib.spinq_w4a4_gemm.restype = ctypes.c_int
_lib.spinq_w4a4_gemm.argtypes = [_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _P, _P, _P]
_lib.spinq_w4a4_gemm_workspace_bytes.restype = ctypes.c_int64
_lib.spinq_w4a4_gemm_workspace_bytes.argtypes = [_I64, _I64, _I64]
_lib.spinq_w4a4_gemm_splitk.restype = ctypes.c_int
_lib.spinq_w4a4_gemm_splitk.argtypes = [_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _P, _P, _P, _I64, _P]
_lib.spinq_w4a4_gemm_noalloc.restype = ctypes.c_int
_lib.spinq_w4a4_gemm_noalloc.argtypes = [_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _P, _P, _P]
_lib.spinq_gemm_select_kernel.restype = ctypes.c_int
_lib.spinq_gemm_select_kernel.argtypes = [ctypes.c_int]
_lib.spinq_gemm_split_k.restype = ctypes.c_int
_lib.spinq_gemm_split_k.argtypes = [ctypes.c_int]
_lib.spinq_w4a4_gemm_plan.restype = ctypes.c_int
_lib.spinq_w4a4_gemm_plan.argtypes = [_I64, _I64, _I64]
_lib.spinq_w4a4_gemm_splitk_plan.restype = ctypes.c_int
_lib.spinq_w4a4_gemm_splitk_plan.argtypes = [_I64, _I64, _I64, ctypes.POINTER(ctypes.c_int)]
_lib.spinq_rotate_quant_act8.restype = ctypes.c_int
_lib.spinq_rotate_quant_act8.argtypes = [_P, _I64, _I64, _I64, ctypes.POINTER(HadCfg), ctypes.POINTER(QuantCfg),
                                         ctypes.c_int32, _P, _P, _P, _P]
_lib.spinq_quant_weight8.restype = ctypes.c_int
_lib.spinq_quant_weight8.argtypes = [_P, _I64, _I64, ctypes.POINTER(HadCfg), ctypes.POINTER(QuantCfg), ctypes.c_int32,
                                     _P, _P, _P, _P]
_lib.spinq_fp8_gemm.restype = ctypes.c_int
_lib.spinq_fp8_gemm.argtypes = [_P, _P, _P, _P, _I64, _I64, _I64, _P, _P]
_lib.spinq_w4a8_gemm.restype = ctypes.c_int
_lib.spinq_w4a8_gemm.argtypes = [_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _P, _P, _P]
_lib.spinq_rope_rotate_quant_kv.restype = ctypes.c_int
_lib.spinq_rope_rotate_quant_kv.argtypes = [_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _I64, _I64, _I64,
                                            ctypes.POINTER(HadCfg), ctypes.POINTER(QuantCfg),
                                            _P, _P, _P, _P, _P, _P, _P]
_lib.spinq_decode_attention_workspace_bytes.restype = ctypes.c_int64
_lib.spinq_decode_attention_workspace_bytes.argtypes = [_I64, _I64, _I64, _I64, _I64]
_lib.spinq_decode_attention_kv4.restype = ctypes.c_int
_lib.spinq_decode_attention_kv4.argtypes = [_P, _P, _P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _I64, _I64,
                                            ctypes.c_float, _P, _P, _I64, _P]
_lib.spinq_rotate_quant_act_signed.restype = ctypes.c_int
_lib.spinq_rotate_quant_act_signed.argtypes = [_P, _I64, _I64, _I64, ctypes.POINTER(HadCfg), _P,
                                               ctypes.POINTER(QuantCfg), _P, _P, _P, _P]
_lib.spinq_quant_weight_signed.restype = ctypes.c_int
_lib.spinq_quant_weight_signed.argtypes = [_P, _I64, _I64, ctypes.POINTER(HadCfg), _P, ctypes.POINTER(QuantCfg),
                                           _P, _P, _P, _P]
_lib.spinq_rotated_linear_workspace_bytes.restype = ctypes.c_int64
_lib.spinq_rotated_linear_workspace_bytes.argtypes = [_I64, _I64]
_lib.spinq_rotated_linear.restype = ctypes.c_int
_lib.spinq_rotated_linear.argtypes = [_P, _I64, _I64, _I64, ctypes.POINTER(HadCfg), _P, ctypes.POINTER(QuantCfg),
                                      _P, _P, _P, _I64, _P, _P, _I64, _P]
_lib.spinq_debug_set_wait_limit_ns.restype = ctypes.c_int
_lib.spinq_debug_set_wait_limit_ns.argtypes = [_I64]
_lib.spinq_debug_stall_launches.restype = ctypes.c_int
_lib.spinq_debug_stall_launches.argtypes = [ctypes.c_int]
_lib.spinq_debug_fail_launches.restype = ctypes.c_int
_lib.spinq_debug_fail_launches.argtypes = [ctypes.c_int]
_lib.spinq_cayley_step.restype = ctypes.c_int
_lib.spinq_cayley_step.argtypes = [_P, _P, _I64, _I64, ctypes.c_float, ctypes.c_int32, _P, _P, _P]
_lib.spinq_rotate_quant_kv.restype = ctypes.c_int
_lib.spinq_rotate_quant_kv.argtypes = [_P, _P, _P, _P, _I64, _I64, _I64, _I64, _I64,
                                       ctypes.POINTER(HadCfg), ctypes.POINTER(QuantCfg),
                                       _P, _P, _P, _P, _P, _P, _P]


def _check(st: int, where: str) -> None:
    if st != SPINQ_OK:
        raise SpinqError(st, where)


# ------------------------------------------------------------------ raw ABI
def spinq_rotate_quant_act(x, M, K, ldx, had, q, codes, scale, zero, stream) -> int:
    return _lib.spinq_rotate_quant_act(x, M, K, ldx, had, q, codes, scale, zero, stream)


def spinq_quant_weight(w, N, K, had, q, codes, scale, rowsum, stream) -> int:
    return _lib.spinq_quant_weight(w, N, K, had, q, codes, scale, rowsum, stream)


def spinq_w4a4_gemm(a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y, acc, stream) -> int:
    return _lib.spinq_w4a4_gemm(a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y, acc,
                                stream)


def spinq_w4a4_gemm_workspace_bytes(M, N, K) -> int:
    return int(_lib.spinq_w4a4_gemm_workspace_bytes(M, N, K))


def spinq_w4a4_gemm_splitk(a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y, acc, ws,
                           ws_bytes, stream) -> int:
    return _lib.spinq_w4a4_gemm_splitk(a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y, acc,
                                       ws, ws_bytes, stream)


def spinq_w4a4_gemm_noalloc(a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y, acc,
                            stream) -> int:
    return _lib.spinq_w4a4_gemm_noalloc(a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y,
                                        acc, stream)


def spinq_rotate_quant_kv(q_in, q_out, k_in, v_in, B, S, Hq, Hkv, D, had, kvq, k_codes, k_scale,
                          k_zero, v_codes, v_scale, v_zero, stream) -> int:
    return _lib.spinq_rotate_quant_kv(q_in, q_out, k_in, v_in, B, S, Hq, Hkv, D, had, kvq, k_codes,
                                      k_scale, k_zero, v_codes, v_scale, v_zero, stream)


def spinq_rotate_quant_act8(x, M, K, ldx, had, q, fmt, codes, scale, zero, stream) -> int:
    return _lib.spinq_rotate_quant_act8(x, M, K, ldx, had, q, fmt, codes, scale, zero, stream)


def spinq_quant_weight8(w, N, K, had, q, fmt, codes, scale, rowsum, stream) -> int:
    return _lib.spinq_quant_weight8(w, N, K, had, q, fmt, codes, scale, rowsum, stream)


def spinq_fp8_gemm(a_codes, a_scale, w_codes, w_scale, M, N, K, y, stream) -> int:
    return _lib.spinq_fp8_gemm(a_codes, a_scale, w_codes, w_scale, M, N, K, y, stream)


def spinq_w4a8_gemm(a_planes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y, acc, stream) -> int:
    return _lib.spinq_w4a8_gemm(a_planes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y, acc, stream)


def spinq_rope_rotate_quant_kv(q_in, q_out, k_in, v_in, positions, cos_sin, max_pos, B, S, Hq, Hkv, D, had, kvq,
                               k_codes, k_scale, k_zero, v_codes, v_scale, v_zero, stream) -> int:
    return _lib.spinq_rope_rotate_quant_kv(q_in, q_out, k_in, v_in, positions, cos_sin, max_pos, B, S, Hq, Hkv, D,
                                           had, kvq, k_codes, k_scale, k_zero, v_codes, v_scale, v_zero, stream)


def spinq_decode_attention_workspace_bytes(B, S, Hq, Hkv, D) -> int:
    return int(_lib.spinq_decode_attention_workspace_bytes(B, S, Hq, Hkv, D))


def spinq_decode_attention_kv4(q, k_codes, k_scale, k_zero, v_codes, v_scale, v_zero, lens, B, S, Hq, Hkv, D,
                               scale, out, ws, ws_bytes, stream) -> int:
    return _lib.spinq_decode_attention_kv4(q, k_codes, k_scale, k_zero, v_codes, v_scale, v_zero, lens, B, S, Hq,
                                           Hkv, D, scale, out, ws, ws_bytes, stream)


def spinq_rotate_quant_act_signed(x, M, K, ldx, had, signs, q, codes, scale, zero, stream) -> int:
    return _lib.spinq_rotate_quant_act_signed(x, M, K, ldx, had, signs, q, codes, scale, zero, stream)


def spinq_quant_weight_signed(w, N, K, had, signs, q, codes, scale, rowsum, stream) -> int:
    return _lib.spinq_quant_weight_signed(w, N, K, had, signs, q, codes, scale, rowsum, stream)


def spinq_rotated_linear_workspace_bytes(M, K) -> int:
    return int(_lib.spinq_rotated_linear_workspace_bytes(M, K))


def spinq_rotated_linear(x, M, K, ldx, had, signs, q, w_codes, w_scale, w_rowsum, N, y, ws, ws_bytes, stream) -> int:
    return _lib.spinq_rotated_linear(x, M, K, ldx, had, signs, q, w_codes, w_scale, w_rowsum, N, y, ws, ws_bytes,
                                     stream)


def spinq_debug_set_wait_limit_ns(ns: int) -> int:
    return int(_lib.spinq_debug_set_wait_limit_ns(ns))


def spinq_debug_stall_launches(n: int) -> int:
    return int(_lib.spinq_debug_stall_launches(n))


def spinq_debug_fail_launches(n: int) -> int:
    return int(_lib.spinq_debug_fail_launches(n))


def spinq_cayley_step(R, grad, batch, n, alpha, iters, R_out, Y_out, stream) -> int:
    return _lib.spinq_cayley_step(R, grad, batch, n, alpha, iters, R_out, Y_out, stream)


def spinq_gemm_select_kernel(kernel: int) -> int:
    return int(_lib.spinq_gemm_select_kernel(kernel))


def spinq_gemm_split_k(n: int) -> int:
    return int(_lib.spinq_gemm_split_k(n))


def spinq_w4a4_gemm_plan(M: int, N: int, K: int) -> int:
    return int(_lib.spinq_w4a4_gemm_plan(M, N, K))


def spinq_w4a4_gemm_splitk_plan(M: int, N: int, K: int) -> tuple:
    """(kernel, K slices) of spinq_w4a4_gemm_splitk for an M x N x K call."""
    ns = ctypes.c_int(0)
    kind = int(_lib.spinq_w4a4_gemm_splitk_plan(M, N, K, ctypes.byref(ns)))
    return kind, int(ns.value)


def spinq_status_string(st: int) -> str:
    return _lib.spinq_status_string(st).decode()


def spinq_version() -> str:
    return _lib.spinq_version().decode()


def spinq_device_status() -> Tuple[int, int]:
    d = ctypes.c_int32(0)
    st = _lib.spinq_device_status(ctypes.byref(d))
    return st, d.value


# ------------------------------------------------------------------ helpers
def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream: Optional[torch.cuda.Stream]):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _had(had: Optional[Tuple[int, int]]):
    return None if had is None else ctypes.byref(HadCfg(int(had[0]), int(had[1])))


def quant_cfg(bits=4, symmetric=True, granularity=SPINQ_PER_TOKEN, group_size=0, clip=1.0) -> QuantCfg:
    return QuantCfg(bits, int(bool(symmetric)), granularity, group_size, float(clip))


@dataclass
class ActCodes:
    codes: torch.Tensor            # uint8 [M, K/2]
    scale: torch.Tensor            # f32 [M]
    zero: Optional[torch.Tensor]   # f32 [M] or None (symmetric)


@dataclass
class WeightCodes:
    codes: torch.Tensor   # uint8 [N, K/2]
    scale: torch.Tensor   # f32 [N]
    rowsum: torch.Tensor  # int32 [N]


def rotate_quant_act(x: torch.Tensor, had: Optional[Tuple[int, int]], symmetric: bool = True,
                     clip: float = 1.0, out: Optional[ActCodes] = None,
                     stream: Optional[torch.cuda.Stream] = None) -> ActCodes:
    assert x.dtype == torch.float16 and x.dim() == 2 and x.stride(1) == 1
    M, K = x.shape
    if out is None:
        out = ActCodes(torch.empty((M, K // 2), dtype=torch.uint8, device=x.device),
                       torch.empty(M, dtype=torch.float32, device=x.device),
                       None if symmetric else torch.empty(M, dtype=torch.float32, device=x.device))
    q = quant_cfg(4, symmetric, SPINQ_PER_TOKEN, 0, clip)
    _check(_lib.spinq_rotate_quant_act(_ptr(x), M, K, x.stride(0), _had(had), ctypes.byref(q),
                                       _ptr(out.codes), _ptr(out.scale), _ptr(out.zero), _stream(stream)),
           "spinq_rotate_quant_act")
    return out


def quant_weight(w: torch.Tensor, had: Optional[Tuple[int, int]], clip: float = 1.0,
                 stream: Optional[torch.cuda.Stream] = None) -> WeightCodes:
    assert w.dtype == torch.float16 and w.is_contiguous()
    N, K = w.shape
    out = WeightCodes(torch.empty((N, K // 2), dtype=torch.uint8, device=w.device),
                      torch.empty(N, dtype=torch.float32, device=w.device),
                      torch.empty(N, dtype=torch.int32, device=w.device))
    q = quant_cfg(4, True, SPINQ_PER_CHANNEL, 0, clip)
    _check(_lib.spinq_quant_weight(_ptr(w), N, K, _had(had), ctypes.byref(q), _ptr(out.codes),
                                   _ptr(out.scale), _ptr(out.rowsum), _stream(stream)),
           "spinq_quant_weight")
    return out


def w4a4_gemm(a: ActCodes, w: WeightCodes, want_acc: bool = False, y: Optional[torch.Tensor] = None,
              stream: Optional[torch.cuda.Stream] = None):
    M = a.codes.shape[0]
    N, Kh = w.codes.shape
    K = Kh * 2
    if y is None:
        y = torch.empty((M, N), dtype=torch.float16, device=a.codes.device)
    acc = torch.empty((M, N), dtype=torch.int32, device=a.codes.device) if want_acc else None
    _check(_lib.spinq_w4a4_gemm(_ptr(a.codes), _ptr(a.scale), _ptr(a.zero), _ptr(w.codes), _ptr(w.scale),
                                _ptr(w.rowsum), M, N, K, _ptr(y), _ptr(acc), _stream(stream)),
           "spinq_w4a4_gemm")
    return (y, acc) if want_acc else y


def gemm_workspace(M: int, N: int, K: int, device=None) -> Optional[torch.Tensor]:
    """Zeroed workspace for w4a4_gemm_splitk (None when the shape needs none)."""
    nbytes = spinq_w4a4_gemm_workspace_bytes(M, N, K)
    if nbytes == 0:
        return None
    return torch.zeros((nbytes + 15) // 16 * 16, dtype=torch.uint8, device=device or "cuda")


def w4a4_gemm_splitk(a: ActCodes, w: WeightCodes, workspace: Optional[torch.Tensor] = None,
                     want_acc: bool = False, y: Optional[torch.Tensor] = None,
                     stream: Optional[torch.cuda.Stream] = None):
    M = a.codes.shape[0]
    N, Kh = w.codes.shape
    K = Kh * 2
    if workspace is None:
        workspace = gemm_workspace(M, N, K, a.codes.device)
    if y is None:
        y = torch.empty((M, N), dtype=torch.float16, device=a.codes.device)
    acc = torch.empty((M, N), dtype=torch.int32, device=a.codes.device) if want_acc else None
    ws_bytes = 0 if workspace is None else workspace.numel()
    _check(_lib.spinq_w4a4_gemm_splitk(_ptr(a.codes), _ptr(a.scale), _ptr(a.zero), _ptr(w.codes), _ptr(w.scale),
                                       _ptr(w.rowsum), M, N, K, _ptr(y), _ptr(acc), _ptr(workspace), ws_bytes,
                                       _stream(stream)),
           "spinq_w4a4_gemm_splitk")
    return (y, acc) if want_acc else y


@dataclass
class KVCodes:
    q_out: torch.Tensor
    k_codes: torch.Tensor
    k_scale: torch.Tensor
    k_zero: torch.Tensor
    v_codes: torch.Tensor
    v_scale: torch.Tensor
    v_zero: torch.Tensor


def rotate_quant_kv(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, clip: float = 1.0,
                    in_place_q: bool = False, out: Optional[KVCodes] = None,
                    stream: Optional[torch.cuda.Stream] = None) -> KVCodes:
    B, S, Hq, D = q.shape
    Hkv = k.shape[2]
    dev = q.device
    if out is None:
        out = KVCodes(q if in_place_q else torch.empty_like(q),
                      torch.empty((B, S, Hkv, D // 2), dtype=torch.uint8, device=dev),
                      torch.empty((B, S, Hkv), dtype=torch.float32, device=dev),
                      torch.empty((B, S, Hkv), dtype=torch.float32, device=dev),
                      torch.empty((B, S, Hkv, D // 2), dtype=torch.uint8, device=dev),
                      torch.empty((B, S, Hkv), dtype=torch.float32, device=dev),
                      torch.empty((B, S, Hkv), dtype=torch.float32, device=dev))
    kvq = quant_cfg(4, False, SPINQ_PER_GROUP, D, clip)
    had = HadCfg(1, D)
    _check(_lib.spinq_rotate_quant_kv(_ptr(q), _ptr(out.q_out), _ptr(k), _ptr(v), B, S, Hq, Hkv, D,
                                      ctypes.byref(had), ctypes.byref(kvq), _ptr(out.k_codes),
                                      _ptr(out.k_scale), _ptr(out.k_zero), _ptr(out.v_codes),
                                      _ptr(out.v_scale), _ptr(out.v_zero), _stream(stream)),
           "spinq_rotate_quant_kv")
    return out


def cayley_step(R: torch.Tensor, grad: torch.Tensor, alpha: float, iters: int = 2, out: Optional[torch.Tensor] = None,
                want_y: bool = False, stream: Optional[torch.cuda.Stream] = None):
    """One Cayley SGD update of rotations R [B, n, n] (or [n, n]) with loss
    gradient ``grad`` (fp32, device); returns R' (and Y when ``want_y``)."""
    assert R.dtype == torch.float32 and grad.dtype == torch.float32 and R.is_contiguous() and grad.is_contiguous()
    n = R.shape[-1]
    batch = R.numel() // (n * n)
    if out is None:
        out = torch.empty_like(R)
    y = torch.empty_like(R) if want_y else None
    _check(_lib.spinq_cayley_step(_ptr(R), _ptr(grad), batch, n, float(alpha), int(iters), _ptr(out), _ptr(y),
                                  _stream(stream)), "spinq_cayley_step")
    return (out, y) if want_y else out


def rotate_quant_act8(x: torch.Tensor, had: Optional[Tuple[int, int]], fmt: int, symmetric: bool = True,
                      clip: float = 1.0, out: Optional[ActCodes] = None,
                      stream: Optional[torch.cuda.Stream] = None) -> ActCodes:
    """8-bit activation codes: SPINQ_FMT_INT8_PLANES ([M, 2K]) or SPINQ_FMT_E4M3 ([M, K])."""
    assert x.dtype == torch.float16 and x.dim() == 2 and x.stride(1) == 1
    M, K = x.shape
    width = 2 * K if fmt == SPINQ_FMT_INT8_PLANES else K
    if out is None:
        out = ActCodes(torch.empty((M, width), dtype=torch.uint8, device=x.device),
                       torch.empty(M, dtype=torch.float32, device=x.device),
                       None if symmetric else torch.empty(M, dtype=torch.float32, device=x.device))
    q = quant_cfg(8, symmetric, SPINQ_PER_TOKEN, 0, clip)
    _check(_lib.spinq_rotate_quant_act8(_ptr(x), M, K, x.stride(0), _had(had), ctypes.byref(q), fmt, _ptr(out.codes),
                                        _ptr(out.scale), _ptr(out.zero), _stream(stream)), "spinq_rotate_quant_act8")
    return out


def quant_weight8(w: torch.Tensor, had: Optional[Tuple[int, int]], fmt: int, clip: float = 1.0,
                  stream: Optional[torch.cuda.Stream] = None) -> WeightCodes:
    """Weights of the 8-bit linears: SPINQ_FMT_E4M3 (FP8) or SPINQ_FMT_INT4_BYTES (W4A8)."""
    assert w.dtype == torch.float16 and w.is_contiguous()
    N, K = w.shape
    out = WeightCodes(torch.empty((N, K), dtype=torch.uint8, device=w.device),
                      torch.empty(N, dtype=torch.float32, device=w.device),
                      torch.empty(N, dtype=torch.int32, device=w.device))
    q = quant_cfg(4 if fmt == SPINQ_FMT_INT4_BYTES else 8, True, SPINQ_PER_CHANNEL, 0, clip)
    _check(_lib.spinq_quant_weight8(_ptr(w), N, K, _had(had), ctypes.byref(q), fmt, _ptr(out.codes), _ptr(out.scale),
                                    _ptr(out.rowsum), _stream(stream)), "spinq_quant_weight8")
    return out


def fp8_gemm(a: ActCodes, w: WeightCodes, y: Optional[torch.Tensor] = None,
             stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    M, K = a.codes.shape
    N = w.codes.shape[0]
    if y is None:
        y = torch.empty((M, N), dtype=torch.float16, device=a.codes.device)
    _check(_lib.spinq_fp8_gemm(_ptr(a.codes), _ptr(a.scale), _ptr(w.codes), _ptr(w.scale), M, N, K, _ptr(y),
                               _stream(stream)), "spinq_fp8_gemm")
    return y


def w4a8_gemm(a: ActCodes, w: WeightCodes, want_acc: bool = False, y: Optional[torch.Tensor] = None,
              stream: Optional[torch.cuda.Stream] = None):
    M = a.codes.shape[0]
    N, K = w.codes.shape
    if y is None:
        y = torch.empty((M, N), dtype=torch.float16, device=a.codes.device)
    acc = torch.empty((M, N), dtype=torch.int32, device=a.codes.device) if want_acc else None
    _check(_lib.spinq_w4a8_gemm(_ptr(a.codes), _ptr(a.scale), _ptr(a.zero), _ptr(w.codes), _ptr(w.scale),
                                _ptr(w.rowsum), M, N, K, _ptr(y), _ptr(acc), _stream(stream)), "spinq_w4a8_gemm")
    return (y, acc) if want_acc else y


def rope_rotate_quant_kv(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, positions: torch.Tensor,
                         cos_sin: torch.Tensor, clip: float = 1.0, in_place_q: bool = False,
                         out: Optional[KVCodes] = None, stream: Optional[torch.cuda.Stream] = None) -> KVCodes:
    """RoPE at ``positions`` [B, S] (int32) from ``cos_sin`` [max_pos, D/2, 2]
    (fp32), then R3 and the 4-bit KV quantizer."""
    B, S, Hq, D = q.shape
    Hkv = k.shape[2]
    dev = q.device
    if out is None:
        out = KVCodes(q if in_place_q else torch.empty_like(q),
                      torch.empty((B, S, Hkv, D // 2), dtype=torch.uint8, device=dev),
                      torch.empty((B, S, Hkv), dtype=torch.float32, device=dev),
                      torch.empty((B, S, Hkv), dtype=torch.float32, device=dev),
                      torch.empty((B, S, Hkv, D // 2), dtype=torch.uint8, device=dev),
                      torch.empty((B, S, Hkv), dtype=torch.float32, device=dev),
                      torch.empty((B, S, Hkv), dtype=torch.float32, device=dev))
    kvq = quant_cfg(4, False, SPINQ_PER_GROUP, D, clip)
    had = HadCfg(1, D)
    _check(_lib.spinq_rope_rotate_quant_kv(_ptr(q), _ptr(out.q_out), _ptr(k), _ptr(v), _ptr(positions),
                                           _ptr(cos_sin), cos_sin.shape[0], B, S, Hq, Hkv, D, ctypes.byref(had),
                                           ctypes.byref(kvq), _ptr(out.k_codes), _ptr(out.k_scale),
                                           _ptr(out.k_zero), _ptr(out.v_codes), _ptr(out.v_scale), _ptr(out.v_zero),
                                           _stream(stream)), "spinq_rope_rotate_quant_kv")
    return out


def decode_attention_kv4(q: torch.Tensor, kv: KVCodes, lens: Optional[torch.Tensor] = None,
                         scale: Optional[float] = None, out: Optional[torch.Tensor] = None,
                         workspace: Optional[torch.Tensor] = None,
                         stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """Decode attention of q [B, Hq, D] (fp16, rotated) over the 4-bit cache ``kv``."""
    B, Hq, D = q.shape
    S, Hkv = kv.k_codes.shape[1], kv.k_codes.shape[2]
    if out is None:
        out = torch.empty_like(q)
    need = spinq_decode_attention_workspace_bytes(B, S, Hq, Hkv, D)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=q.device)
    sc = 1.0 / (D ** 0.5) if scale is None else float(scale)
    _check(_lib.spinq_decode_attention_kv4(_ptr(q), _ptr(kv.k_codes), _ptr(kv.k_scale), _ptr(kv.k_zero),
                                           _ptr(kv.v_codes), _ptr(kv.v_scale), _ptr(kv.v_zero), _ptr(lens), B, S, Hq,
                                           Hkv, D, sc, _ptr(out), _ptr(workspace), workspace.numel(),
                                           _stream(stream)), "spinq_decode_attention_kv4")
    return out


def sign_mask(signs) -> torch.Tensor:
    """+-1 per input index -> the [K/8] byte bit mask of the signed entry
    points (bit k % 8 of byte k / 8 set for s_k = -1), on the device."""
    s = torch.as_tensor(signs).reshape(-1)
    neg = (s < 0).to(torch.uint8).reshape(-1, 8)
    bits = torch.zeros(neg.shape[0], dtype=torch.uint8)
    for e in range(8):
        bits |= neg[:, e].cpu() << e
    return bits.cuda()


def rotate_quant_act_signed(x: torch.Tensor, had: Tuple[int, int], signs: torch.Tensor, symmetric: bool = True,
                            clip: float = 1.0, out: Optional[ActCodes] = None,
                            stream: Optional[torch.cuda.Stream] = None) -> ActCodes:
    """rotate_quant_act with R = S H / sqrt(K); ``signs`` is the device bit mask."""
    M, K = x.shape
    if out is None:
        out = ActCodes(torch.empty((M, K // 2), dtype=torch.uint8, device=x.device),
                       torch.empty(M, dtype=torch.float32, device=x.device),
                       None if symmetric else torch.empty(M, dtype=torch.float32, device=x.device))
    q = quant_cfg(4, symmetric, SPINQ_PER_TOKEN, 0, clip)
    _check(_lib.spinq_rotate_quant_act_signed(_ptr(x), M, K, x.stride(0), _had(had), _ptr(signs), ctypes.byref(q),
                                              _ptr(out.codes), _ptr(out.scale), _ptr(out.zero), _stream(stream)),
           "spinq_rotate_quant_act_signed")
    return out


def quant_weight_signed(w: torch.Tensor, had: Tuple[int, int], signs: torch.Tensor, clip: float = 1.0,
                        stream: Optional[torch.cuda.Stream] = None) -> WeightCodes:
    N, K = w.shape
    out = WeightCodes(torch.empty((N, K // 2), dtype=torch.uint8, device=w.device),
                      torch.empty(N, dtype=torch.float32, device=w.device),
                      torch.empty(N, dtype=torch.int32, device=w.device))
    q = quant_cfg(4, True, SPINQ_PER_CHANNEL, 0, clip)
    _check(_lib.spinq_quant_weight_signed(_ptr(w), N, K, _had(had), _ptr(signs), ctypes.byref(q), _ptr(out.codes),
                                          _ptr(out.scale), _ptr(out.rowsum), _stream(stream)),
           "spinq_quant_weight_signed")
    return out


def rotated_linear(x: torch.Tensor, had: Tuple[int, int], w: WeightCodes, signs: Optional[torch.Tensor] = None,
                   symmetric: bool = True, clip: float = 1.0, y: Optional[torch.Tensor] = None,
                   workspace: Optional[torch.Tensor] = None, stream: Optional[torch.cuda.Stream] = None):
    """Online R4 (+ random signs) + act quant + W4A4 GEMM in one call."""
    M, K = x.shape
    N = w.codes.shape[0]
    if y is None:
        y = torch.empty((M, N), dtype=torch.float16, device=x.device)
    if workspace is None:
        workspace = torch.empty(spinq_rotated_linear_workspace_bytes(M, K), dtype=torch.uint8, device=x.device)
    q = quant_cfg(4, symmetric, SPINQ_PER_TOKEN, 0, clip)
    _check(_lib.spinq_rotated_linear(_ptr(x), M, K, x.stride(0), _had(had), _ptr(signs), ctypes.byref(q),
                                     _ptr(w.codes), _ptr(w.scale), _ptr(w.rowsum), N, _ptr(y), _ptr(workspace),
                                     workspace.numel(), _stream(stream)), "spinq_rotated_linear")
    return y
