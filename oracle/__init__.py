"""CPU oracle for the SpinQuant rotated W4A4 hot path (arXiv 2405.16406).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  It shares no code with the CUDA library in
``paper_2405_16406_gb300`` and neither side imports the other.

The arithmetic lives in ``spinq_oracle.c`` (plain C, double precision, one
definition per function, each citing the paper passage it follows).  This
module only marshals numpy arrays into it and composes the steps in the
paper's order:

* ``rotate_quant_act``  -- Sec. 3.1 (R4 online Hadamard) then Eq. 1 per token.
* ``quant_weight``      -- Sec. 3.1 rotational invariance (W' = W R) then
  Eq. 1 per output channel (RTN, as in the appendix ablation on RTN vs GPTQ).
* ``w4a4_linear``       -- the dequantized product of Eq. 1 codes, with the
  integer accumulator that a W4A4 GEMM computes.
* ``rotate_quant_kv``   -- Sec. 3.1 (R3 on Q and K over head_dim) then Eq. 1
  asymmetric per (token, kv-head) group for K and V.

Parity status: every function here is pinned by a ``-m "not gpu"`` test in
``tests/test_oracle_*.py`` (closed forms, library special cases, invariants,
brute force); none is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass
from typing import Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "spinq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libspinq_oracle.so")

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, no fast-math, OpenMP over rows)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-fno-fast-math", "-ffp-contract=off", "-fopenmp", "-fPIC", "-shared",
           "-std=c11", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    P = ctypes.c_void_p
    i64 = ctypes.c_int64
    i32 = ctypes.c_int
    dbl = ctypes.c_double
    sig = {
        "oracle_set_threads": (i32, [i32]),
        "oracle_f16_to_double": (dbl, [ctypes.c_uint16]),
        "oracle_double_to_f16": (ctypes.c_uint16, [dbl]),
        "oracle_f16_array_to_double": (None, [P, P, i64]),
        "oracle_double_array_to_f16": (None, [P, P, i64]),
        "oracle_sylvester": (i32, [i64, P]),
        "oracle_paley1": (i32, [i32, P]),
        "oracle_small_hadamard": (i32, [i32, P]),
        "oracle_fwht": (None, [P, i64]),
        "oracle_rotate": (i32, [P, P, i64, i32, i64]),
        "oracle_quantize_rows": (i32, [P, i64, i64, i32, i32, dbl, P, P, P]),
        "oracle_dequantize_rows": (None, [P, P, P, i64, i64, P]),
        "oracle_pack4": (None, [P, i64, P]),
        "oracle_unpack4": (None, [P, i64, i32, P]),
        "oracle_w4a4_gemm": (i32, [P, P, P, P, P, i64, i64, i64, P, P]),
        "oracle_w4a4_gemm_sampled": (i32, [P, P, P, P, P, i64, P, P, i64, P, P]),
        "oracle_rowsum": (None, [P, i64, i64, P]),
        "oracle_cayley_y": (i32, [P, P, i64, P]),
        "oracle_rope": (i32, [P, P, i64, i64, dbl, P]),
        "oracle_decode_attention": (i32, [P, P, P, P, i64, i64, i64, i64, i64, dbl, P]),
        "oracle_e4m3_to_double": (dbl, [ctypes.c_uint8]),
        "oracle_double_to_e4m3": (ctypes.c_uint8, [dbl]),
        "oracle_e4m3_array_to_double": (None, [P, P, i64]),
        "oracle_quantize_rows_e4m3": (i32, [P, i64, i64, dbl, P, P]),
        "oracle_w4a8_gemm": (i32, [P, P, P, P, P, i64, i64, i64, P, P]),
        "oracle_fp8_gemm": (i32, [P, P, P, P, i64, i64, i64, P]),
        "oracle_cayley_step": (i32, [P, P, i64, i64, dbl, i32, P, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a: np.ndarray, dtype) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=dtype)


def _check(rc: int, what: str) -> None:
    if rc != 0:
        raise ValueError(f"oracle: {what} rejected its arguments (rc={rc})")


def set_threads(n: int = 0) -> int:
    """Set the OpenMP thread count (0 keeps the current one); returns it."""
    return int(_load().oracle_set_threads(int(n)))


# --------------------------------------------------------------------------
# fp16 <-> double (the oracle's own IEEE binary16 conversion)
# --------------------------------------------------------------------------
def f16_to_f64(x: np.ndarray) -> np.ndarray:
    """Decode IEEE binary16 values (np.float16 or raw uint16 bits) to double."""
    h = _c(np.asarray(x).view(np.uint16), np.uint16)
    out = np.empty(h.shape, dtype=np.float64)
    _load().oracle_f16_array_to_double(_ptr(h), _ptr(out), h.size)
    return out


def f64_to_f16(x: np.ndarray) -> np.ndarray:
    """Round doubles to binary16 (round-half-to-even); returns np.float16."""
    d = _c(x, np.float64)
    out = np.empty(d.shape, dtype=np.uint16)
    _load().oracle_double_array_to_f16(_ptr(d), _ptr(out), d.size)
    return out.view(np.float16)


# --------------------------------------------------------------------------
# Hadamard matrices and the rotation (Sec. 2.2 footnote, Sec. 3.1 R3/R4)
# --------------------------------------------------------------------------
def sylvester(n: int) -> np.ndarray:
    H = np.empty((n, n), dtype=np.int8)
    _check(_load().oracle_sylvester(n, _ptr(H)), f"sylvester({n})")
    return H


def paley1(q: int) -> np.ndarray:
    H = np.empty((q + 1, q + 1), dtype=np.int8)
    _check(_load().oracle_paley1(q, _ptr(H)), f"paley1({q})")
    return H


def small_hadamard(n_s: int) -> np.ndarray:
    H = np.empty((n_s, n_s), dtype=np.int8)
    _check(_load().oracle_small_hadamard(n_s, _ptr(H)), f"small_hadamard({n_s})")
    return H


def fwht(v: np.ndarray) -> np.ndarray:
    """H_n v for one vector (natural-order Sylvester), unnormalised."""
    out = _c(v, np.float64).copy()
    _load().oracle_fwht(_ptr(out), out.size)
    return out


def rotate(x: np.ndarray, n_small: int, n_pow2: int) -> np.ndarray:
    """Rows of ``x`` (double) times (H_s (x) H_P) / sqrt(K)."""
    x = _c(x, np.float64)
    rows = x.size // (n_small * n_pow2)
    assert x.shape[-1] == n_small * n_pow2
    y = np.empty_like(x)
    _check(_load().oracle_rotate(_ptr(x), _ptr(y), rows, n_small, n_pow2), "rotate")
    return y


# --------------------------------------------------------------------------
# Eq. 1 quantizer and 4-bit packing
# --------------------------------------------------------------------------
def quantize_rows(x: np.ndarray, bits: int, symmetric: bool, clip: float = 1.0
                  ) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Per-row Eq. 1: returns (codes int32, alpha f64, beta f64)."""
    x = _c(x, np.float64)
    K = x.shape[-1]
    rows = x.size // K
    codes = np.empty(x.shape, dtype=np.int32)
    alpha = np.empty(rows, dtype=np.float64)
    beta = np.empty(rows, dtype=np.float64)
    _check(_load().oracle_quantize_rows(_ptr(x), rows, K, bits, int(bool(symmetric)), float(clip),
                                        _ptr(codes), _ptr(alpha), _ptr(beta)), "quantize_rows")
    return codes, alpha, beta


def dequantize_rows(codes: np.ndarray, alpha: np.ndarray, beta: Optional[np.ndarray]) -> np.ndarray:
    codes = _c(codes, np.int32)
    K = codes.shape[-1]
    rows = codes.size // K
    out = np.empty(codes.shape, dtype=np.float64)
    a = _c(alpha, np.float64)
    b = None if beta is None else _c(beta, np.float64)
    _load().oracle_dequantize_rows(_ptr(codes), _ptr(a), _ptr(b), rows, K, _ptr(out))
    return out


def pack4(codes: np.ndarray) -> np.ndarray:
    codes = _c(codes, np.int32)
    assert codes.shape[-1] % 2 == 0
    out = np.empty(codes.shape[:-1] + (codes.shape[-1] // 2,), dtype=np.uint8)
    _load().oracle_pack4(_ptr(codes), codes.size, _ptr(out))
    return out


def unpack4(packed: np.ndarray, signed: bool) -> np.ndarray:
    packed = _c(packed, np.uint8)
    out = np.empty(packed.shape[:-1] + (packed.shape[-1] * 2,), dtype=np.int32)
    _load().oracle_unpack4(_ptr(packed), out.size, int(bool(signed)), _ptr(out))
    return out


def rowsum(codes: np.ndarray) -> np.ndarray:
    codes = _c(codes, np.int32)
    K = codes.shape[-1]
    out = np.empty(codes.size // K, dtype=np.int32)
    _load().oracle_rowsum(_ptr(codes), codes.size // K, K, _ptr(out))
    return out


# --------------------------------------------------------------------------
# The hot-path steps, composed in the paper's order
# --------------------------------------------------------------------------
@dataclass
class QuantAct:
    codes: np.ndarray       # int32 [M, K]   (q for symmetric, u for asymmetric)
    packed: np.ndarray      # uint8 [M, K/2]
    alpha: np.ndarray       # f64 [M]
    beta: Optional[np.ndarray]  # f64 [M] (asymmetric) or None
    rotated: np.ndarray     # f64 [M, K], the rotated activation before rounding


def rotate_quant_act(x_f16: np.ndarray, had: Optional[Tuple[int, int]], bits: int = 4,
                     symmetric: bool = True, clip: float = 1.0, signs: Optional[np.ndarray] = None) -> QuantAct:
    """Sec. 3.1 R4: x' = x (H_s (x) H_P)/sqrt(K) (skipped if ``had`` is None),
    then Eq. 1 per token (row).  ``signs`` (+-1 per input index, or None)
    makes the rotation the random Hadamard S H of the Sec. 2.2 footnote:
    x' = (x S) (H_s (x) H_P)/sqrt(K)."""
    x = f16_to_f64(x_f16)
    if signs is not None:
        x = x * _sign_vector(signs, x.shape[-1])
    xr = rotate(x, had[0], had[1]) if had is not None else x
    codes, alpha, beta = quantize_rows(xr, bits, symmetric, clip)
    return QuantAct(codes, pack4(codes) if bits == 4 else None, alpha,
                    None if symmetric else beta, xr)


def _sign_vector(signs: np.ndarray, K: int) -> np.ndarray:
    s = np.asarray(signs, dtype=np.float64).reshape(-1)
    assert s.size == K and np.all(np.abs(s) == 1.0), "signs: one +-1 per input index"
    return s


@dataclass
class QuantWeight:
    codes: np.ndarray    # int32 [N, K] symmetric codes
    packed: np.ndarray   # uint8 [N, K/2]
    scale: np.ndarray    # f64 [N]
    rowsum: np.ndarray   # int32 [N]
    rotated: np.ndarray  # f64 [N, K]


def quant_weight(w_f16: np.ndarray, had: Optional[Tuple[int, int]], bits: int = 4,
                 clip: float = 1.0, signs: Optional[np.ndarray] = None) -> QuantWeight:
    """Sec. 3.1 invariance: W' = W R (each output row rotated like an
    activation row), then Eq. 1 symmetric per output channel (RTN).  With
    ``signs``, R = S H / sqrt(K) as for the activations (W' = W S H)."""
    w = f16_to_f64(w_f16)
    if signs is not None:
        w = w * _sign_vector(signs, w.shape[-1])
    wr = rotate(w, had[0], had[1]) if had is not None else w
    codes, scale, _ = quantize_rows(wr, bits, True, clip)
    return QuantWeight(codes, pack4(codes), scale, rowsum(codes), wr)


@dataclass
class Linear:
    acc: np.ndarray    # int32 [M, N]
    y: np.ndarray      # f64 [M, N]
    y_f16: np.ndarray  # float16 [M, N]


def w4a4_linear(a: QuantAct, w: QuantWeight) -> Linear:
    """Integer accumulator and dequantized product of the two Eq. 1 codes."""
    M, K = a.codes.shape
    N = w.codes.shape[0]
    acc = np.empty((M, N), dtype=np.int32)
    y = np.empty((M, N), dtype=np.float64)
    ac = _c(a.codes, np.int32)
    wc = _c(w.codes, np.int32)
    al = _c(a.alpha, np.float64)
    be = None if a.beta is None else _c(a.beta, np.float64)
    sc = _c(w.scale, np.float64)
    _check(_load().oracle_w4a4_gemm(_ptr(ac), _ptr(al), _ptr(be), _ptr(wc), _ptr(sc), M, N, K,
                                    _ptr(acc), _ptr(y)), "w4a4_gemm")
    return Linear(acc, y, f64_to_f16(y))


def w4a4_linear_sampled(a_codes: np.ndarray, a_alpha: np.ndarray, a_beta: Optional[np.ndarray],
                        w_codes: np.ndarray, w_scale: np.ndarray, ms: np.ndarray, ns: np.ndarray
                        ) -> Tuple[np.ndarray, np.ndarray]:
    """The same definition at the listed (m, n) outputs; returns (acc, y)."""
    K = a_codes.shape[-1]
    ms = _c(ms, np.int64)
    ns = _c(ns, np.int64)
    acc = np.empty(ms.size, dtype=np.int32)
    y = np.empty(ms.size, dtype=np.float64)
    ac = _c(a_codes, np.int32)
    wc = _c(w_codes, np.int32)
    al = _c(a_alpha, np.float64)
    be = None if a_beta is None else _c(a_beta, np.float64)
    sc = _c(w_scale, np.float64)
    _check(_load().oracle_w4a4_gemm_sampled(_ptr(ac), _ptr(al), _ptr(be), _ptr(wc), _ptr(sc), K,
                                            _ptr(ms), _ptr(ns), ms.size, _ptr(acc), _ptr(y)),
           "w4a4_gemm_sampled")
    return acc, y


@dataclass
class QuantKV:
    q_out: np.ndarray    # float16 [B, S, Hq, D]
    q_rot: np.ndarray    # f64 [B, S, Hq, D] rotated Q before fp16 rounding
    k_codes: np.ndarray  # int32 [B, S, Hkv, D]
    k_alpha: np.ndarray  # f64 [B, S, Hkv, D/group]
    k_beta: np.ndarray
    v_codes: np.ndarray
    v_alpha: np.ndarray
    v_beta: np.ndarray
    k_rot: np.ndarray    # f64 rotated K


def rotate_quant_kv(q_f16: np.ndarray, k_f16: np.ndarray, v_f16: np.ndarray,
                    had: Optional[Tuple[int, int]], bits: int = 4, clip: float = 1.0,
                    group: Optional[int] = None) -> QuantKV:
    """Sec. 3.1 R3: Q' = Q R, K' = K R over head_dim (R = H/sqrt(D)); then
    Eq. 1 asymmetric on K' and V per (token, kv-head) group (appendix
    "Quantization choice": asymmetric is the better choice for the KV cache)."""
    B, S, Hq, D = q_f16.shape
    Hkv = k_f16.shape[2]
    g = D if group is None else group
    assert D % g == 0
    q = f16_to_f64(q_f16).reshape(-1, D)
    k = f16_to_f64(k_f16).reshape(-1, D)
    v = f16_to_f64(v_f16).reshape(-1, D)
    qr = rotate(q, had[0], had[1]) if had is not None else q
    kr = rotate(k, had[0], had[1]) if had is not None else k
    kc, ka, kb = quantize_rows(kr.reshape(-1, g), bits, False, clip)
    vc, va, vb = quantize_rows(v.reshape(-1, g), bits, False, clip)
    sh = (B, S, Hkv, D // g)
    return QuantKV(f64_to_f16(qr).reshape(B, S, Hq, D), qr.reshape(B, S, Hq, D),
                   kc.reshape(B, S, Hkv, D), ka.reshape(sh), kb.reshape(sh),
                   vc.reshape(B, S, Hkv, D), va.reshape(sh), vb.reshape(sh),
                   kr.reshape(B, S, Hkv, D))


# --------------------------------------------------------------------------
# Cayley SGD step (Sec. 3.2)
# --------------------------------------------------------------------------
def cayley_y(R: np.ndarray, G: np.ndarray) -> np.ndarray:
    """Y = G_hat - G_hat^T with G_hat = G R^T - 1/2 R R^T G R^T (Sec. 3.2)."""
    R = _c(R, np.float64)
    G = _c(G, np.float64)
    n = R.shape[-1]
    Y = np.empty((n, n), dtype=np.float64)
    _check(_load().oracle_cayley_y(_ptr(R), _ptr(G), n, _ptr(Y)), "cayley_y")
    return Y


def cayley_step(R: np.ndarray, G: np.ndarray, alpha: float, iters: int = 2
                ) -> Tuple[np.ndarray, np.ndarray]:
    """One Cayley SGD update of each rotation in a batch [B, n, n] (or one
    [n, n]) by the fixed-point iteration: R'_0 = R + a Y R, then
    R'_{k+1} = R + (a/2) Y (R + R'_k), ``iters`` times.  ``G`` is the loss
    gradient; Y is built from -G (the descent reading of the printed update:
    the cited Cayley SGD forms G_hat from the negative gradient).  Returns
    (R', Y)."""
    R = _c(R, np.float64)
    G = _c(G, np.float64)
    single = R.ndim == 2
    Rb = R[None] if single else R
    Gb = G[None] if single else G
    B, n = Rb.shape[0], Rb.shape[-1]
    out = np.empty_like(Rb)
    Y = np.empty_like(Rb)
    _check(_load().oracle_cayley_step(_ptr(Rb), _ptr(Gb), B, n, float(alpha), int(iters), _ptr(out), _ptr(Y)),
           "cayley_step")
    return (out[0], Y[0]) if single else (out, Y)


def cayley_exact(R: np.ndarray, G: np.ndarray, alpha: float) -> np.ndarray:
    """The Cayley update by its definition, R' = (I - a/2 Y)^-1 (I + a/2 Y) R
    with Y built from -G, through a library linear solve (the fixed point of
    ``cayley_step``)."""
    R = np.asarray(R, dtype=np.float64)
    n = R.shape[-1]
    Y = cayley_y(R, -np.asarray(G, dtype=np.float64))
    eye = np.eye(n)
    return np.linalg.solve(eye - 0.5 * alpha * Y, (eye + 0.5 * alpha * Y) @ R)


# --------------------------------------------------------------------------
# 8-bit variants: W4A8 and W-fp8-A-fp8 (main results table, 4-8-x rows;
# appendix "Latency measurement on GPU", FP8 GEMM setting)
# --------------------------------------------------------------------------
def e4m3_to_f64(b: np.ndarray) -> np.ndarray:
    """Decode E4M3 bytes (finite-only FP8: bias 7, 3 mantissa bits, max 448)."""
    b = _c(b, np.uint8)
    out = np.empty(b.shape, dtype=np.float64)
    _load().oracle_e4m3_array_to_double(_ptr(b), _ptr(out), b.size)
    return out


def f64_to_e4m3(x: np.ndarray) -> np.ndarray:
    """Round to the nearest E4M3 value (ties to even), saturating at +-448."""
    lib = _load()
    x = np.asarray(x, dtype=np.float64)
    return np.array([lib.oracle_double_to_e4m3(float(v)) for v in x.reshape(-1)], dtype=np.uint8).reshape(x.shape)


@dataclass
class QuantActFP8:
    codes: np.ndarray    # uint8 E4M3 [M, K]
    alpha: np.ndarray    # f64 [M]
    rotated: np.ndarray  # f64 [M, K]


def rotate_quant_act_fp8(x_f16: np.ndarray, had: Optional[Tuple[int, int]], clip: float = 1.0) -> QuantActFP8:
    """Sec. 3.1 rotation (skipped when ``had`` is None), then per-token FP8:
    alpha = clip max|x'| / 448, code = E4M3(x' / alpha)."""
    x = f16_to_f64(x_f16)
    xr = rotate(x, had[0], had[1]) if had is not None else x
    xr = _c(xr, np.float64)
    K = xr.shape[-1]
    rows = xr.size // K
    codes = np.empty(xr.shape, dtype=np.uint8)
    alpha = np.empty(rows, dtype=np.float64)
    _check(_load().oracle_quantize_rows_e4m3(_ptr(xr), rows, K, float(clip), _ptr(codes), _ptr(alpha)),
           "quantize_rows_e4m3")
    return QuantActFP8(codes, alpha, xr)


def quant_weight_fp8(w_f16: np.ndarray, had: Optional[Tuple[int, int]], clip: float = 1.0) -> QuantActFP8:
    """W' = W R (Sec. 3.1), then per-output-channel FP8 (same rule as the
    activations, one scale per row of W')."""
    return rotate_quant_act_fp8(w_f16, had, clip)


def w4a8_linear(a: QuantAct, w: QuantWeight) -> Linear:
    """Integer accumulator and dequantized product of 8-bit activation codes
    (q, or u with the 128 offset) and 4-bit weight codes."""
    M, K = a.codes.shape
    N = w.codes.shape[0]
    acc = np.empty((M, N), dtype=np.int32)
    y = np.empty((M, N), dtype=np.float64)
    ac = _c(a.codes, np.int32)
    wc = _c(w.codes, np.int32)
    al = _c(a.alpha, np.float64)
    be = None if a.beta is None else _c(a.beta, np.float64)
    sc = _c(w.scale, np.float64)
    _check(_load().oracle_w4a8_gemm(_ptr(ac), _ptr(al), _ptr(be), _ptr(wc), _ptr(sc), M, N, K, _ptr(acc), _ptr(y)),
           "w4a8_gemm")
    return Linear(acc, y, f64_to_f16(y))


def fp8_linear(a_codes: np.ndarray, a_alpha: np.ndarray, w_codes: np.ndarray, w_scale: np.ndarray) -> np.ndarray:
    """y = sum_k (alpha_m a_mk)(s_n w_nk) over decoded E4M3 codes (double)."""
    ac = _c(a_codes, np.uint8)
    wc = _c(w_codes, np.uint8)
    M, K = ac.shape
    N = wc.shape[0]
    y = np.empty((M, N), dtype=np.float64)
    _check(_load().oracle_fp8_gemm(_ptr(ac), _ptr(_c(a_alpha, np.float64)), _ptr(wc), _ptr(_c(w_scale, np.float64)),
                                   M, N, K, _ptr(y)), "fp8_gemm")
    return y


# --------------------------------------------------------------------------
# RoPE in front of R3, and decode attention over the 4-bit KV cache
# (Sec. 3.1 R3; appendix "Latency measurement on GPU")
# --------------------------------------------------------------------------
def rope(x: np.ndarray, pos: np.ndarray, base: float = 500000.0) -> np.ndarray:
    """Rotary embedding (rotate-half form) of rows [..., D] at positions
    ``pos`` (one per row of the flattened leading dimensions), in double."""
    x = _c(x, np.float64)
    D = x.shape[-1]
    rows = x.size // D
    p = _c(np.asarray(pos, dtype=np.int64).reshape(-1), np.int64)
    assert p.size == rows, "one position per row"
    y = np.empty_like(x)
    _check(_load().oracle_rope(_ptr(x), _ptr(p), rows, D, float(base), _ptr(y)), "rope")
    return y


def rope_rotate_quant_kv(q_f16: np.ndarray, k_f16: np.ndarray, v_f16: np.ndarray, positions: np.ndarray,
                         had: Tuple[int, int], base: float = 500000.0, bits: int = 4, clip: float = 1.0) -> QuantKV:
    """RoPE on Q and K at their tokens' positions, rounded to fp16 (the
    model's activations), then R3 and the KV quantizer as rotate_quant_kv."""
    B, S, Hq, D = q_f16.shape
    Hkv = k_f16.shape[2]
    pos = np.asarray(positions, dtype=np.int64).reshape(B, S)
    qp = rope(f16_to_f64(q_f16).reshape(-1, D), np.repeat(pos.reshape(-1), Hq), base)
    kp = rope(f16_to_f64(k_f16).reshape(-1, D), np.repeat(pos.reshape(-1), Hkv), base)
    return rotate_quant_kv(f64_to_f16(qp).reshape(B, S, Hq, D), f64_to_f16(kp).reshape(B, S, Hkv, D), v_f16, had,
                           bits, clip)


def decode_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, lens: Optional[np.ndarray] = None,
                     scale: Optional[float] = None) -> np.ndarray:
    """o[b, h] = sum_t softmax_t(scale q[b, h] . k[b, t, h / G]) v[b, t, h / G]
    over t < lens[b] (double); q [B, Hq, D], k, v [B, S, Hkv, D]."""
    q = _c(q, np.float64)
    k = _c(k, np.float64)
    v = _c(v, np.float64)
    B, Hq, D = q.shape
    S, Hkv = k.shape[1], k.shape[2]
    sc = 1.0 / np.sqrt(D) if scale is None else float(scale)
    L = None if lens is None else _c(lens, np.int64)
    o = np.empty((B, Hq, D), dtype=np.float64)
    _check(_load().oracle_decode_attention(_ptr(q), _ptr(k), _ptr(v), _ptr(L), B, S, Hq, Hkv, D, sc, _ptr(o)),
           "decode_attention")
    return o


def dequant_kv(codes: np.ndarray, alpha: np.ndarray, beta: np.ndarray) -> np.ndarray:
    """alpha u + beta per (token, kv head) group of Eq. 1 asymmetric codes."""
    return dequantize_rows(codes.reshape(-1, codes.shape[-1]), alpha.reshape(-1), beta.reshape(-1)).reshape(codes.shape)
