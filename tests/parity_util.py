"""Comparison helpers for GPU-vs-oracle parity tests (no arithmetic of the
method lives here: only unpacking of stored codes and error statistics)."""
import numpy as np

import oracle

# Acceptance bars for the rotated W4A4 path.
CODE_FLIP_FRAC = 1e-4      # codes may differ by +-1 on at most this fraction (ties)
Y_REL_FROB = 1e-2          # fp16 output: ||y_gpu - y_oracle||_F / ||y_oracle||_F
SCALE_REL = 1e-5           # fp32 alpha (and beta relative to alpha) vs the double oracle


def gpu_codes(packed_u8, signed):
    return oracle.unpack4(np.ascontiguousarray(packed_u8), signed)


def code_stats(got, ref):
    d = np.abs(got.astype(np.int64) - ref.astype(np.int64))
    return int(d.max(initial=0)), float(np.count_nonzero(d) / max(d.size, 1))


def assert_codes_close(got, ref, what=""):
    mx, frac = code_stats(got, ref)
    assert mx <= 1, f"{what}: code difference {mx} > 1"
    assert frac <= CODE_FLIP_FRAC, f"{what}: {frac:.2e} of codes differ (> {CODE_FLIP_FRAC})"
    return frac


def assert_scale_close(got, ref, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = np.abs(got - ref)
    tol = SCALE_REL * np.maximum(np.abs(ref), 1e-30)
    bad = err > tol
    assert not bad.any(), f"{what}: {bad.sum()} scales off, worst {np.max(err / np.maximum(np.abs(ref), 1e-30)):.2e}"


def assert_zero_close(got, ref, alpha, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = np.abs(got - ref)
    tol = SCALE_REL * (np.abs(ref) + np.asarray(alpha, dtype=np.float64)) + 1e-30
    assert np.all(err <= tol), f"{what}: zero points off (worst {np.max(err - tol):.2e})"


def rel_frob(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))
