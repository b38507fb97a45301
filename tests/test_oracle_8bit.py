"""Pins of the oracle's 8-bit variants (W4A8 and W-fp8-A-fp8; main results
table 4-8-x rows, appendix "Latency measurement on GPU"): the E4M3 codec
against PyTorch's float8_e4m3fn on every bit pattern, every grid value and
every tie; the FP8 quantizer's invariants (the row maximum maps to 448, the
error stays within half a quantum, zero rows, clipping saturates); the W4A8
accumulator and output against numpy integer and float matmuls, including
extreme codes; the FP8 GEMM against a numpy matmul of the decoded codes."""
import numpy as np
import pytest
import torch

import oracle


def _torch_e4m3(v):
    return torch.from_numpy(np.asarray(v, dtype=np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()


def test_e4m3_decode_every_pattern():
    b = np.arange(256, dtype=np.uint8)
    d = oracle.e4m3_to_f64(b)
    t = torch.from_numpy(b).view(torch.float8_e4m3fn).double().numpy()
    assert np.array_equal(np.isnan(d), np.isnan(t))
    assert np.array_equal(d[~np.isnan(d)], t[~np.isnan(t)])
    assert d[0x7E] == 448.0 and d[0x01] == 2.0 ** -9 and d[0x08] == 2.0 ** -6


def test_e4m3_encode_grid_ties_and_random():
    grid = oracle.e4m3_to_f64(np.arange(256, dtype=np.uint8))
    grid = np.unique(grid[np.isfinite(grid)])
    mids = (grid[:-1] + grid[1:]) / 2                        # exact ties, representable in fp32
    rng = np.random.default_rng(0)
    rnd = np.concatenate([rng.uniform(-448, 448, 20000), rng.uniform(-0.02, 0.02, 20000)])
    for v in (grid, mids, rnd.astype(np.float32).astype(np.float64)):
        got = oracle.f64_to_e4m3(v)
        want = _torch_e4m3(v)
        assert np.array_equal(oracle.e4m3_to_f64(got), oracle.e4m3_to_f64(want))
    assert oracle.f64_to_e4m3(np.array([1e6, -1e6, 448.0, 460.0])).tolist() == [0x7E, 0xFE, 0x7E, 0x7E]


def test_fp8_quantizer_invariants():
    rng = np.random.default_rng(1)
    x = (rng.standard_normal((6, 512)) * 3).astype(np.float16)
    x[2] = 0
    q = oracle.rotate_quant_act_fp8(x, None)
    xd = x.astype(np.float64)
    dec = oracle.e4m3_to_f64(q.codes)
    assert q.alpha[2] == 0 and not q.codes[2].any()
    for r in (0, 1, 3, 4, 5):
        a = q.alpha[r]
        assert a == np.abs(xd[r]).max() / 448
        assert np.abs(dec[r]).max() == 448.0
        v = xd[r] / a
        # half a quantum of the E4M3 grid at |v| (2^-10 below 2^-6)
        e = np.maximum(np.floor(np.log2(np.maximum(np.abs(v), 2.0 ** -6))), -6)
        assert np.all(np.abs(dec[r] - v) <= 2.0 ** (e - 4) + 1e-12)
    qc = oracle.rotate_quant_act_fp8(x, None, clip=0.5)
    assert np.abs(oracle.e4m3_to_f64(qc.codes)).max() == 448.0       # saturated
    np.testing.assert_allclose(qc.alpha, 0.5 * q.alpha)


@pytest.mark.parametrize("sym", [True, False])
def test_w4a8_gemm_against_numpy(sym):
    rng = np.random.default_rng(2)
    M, N, K = 5, 7, 256
    a = rng.integers(-128, 128, (M, K)) if sym else rng.integers(0, 256, (M, K))
    w = rng.integers(-8, 8, (N, K))
    al = rng.uniform(0.1, 1, M)
    be = None if sym else rng.uniform(-3, 0, M)
    ws = rng.uniform(0.001, 0.01, N)
    qa = oracle.QuantAct(a.astype(np.int32), None, al, be, None)
    qw = oracle.QuantWeight(w.astype(np.int32), None, ws, w.sum(1).astype(np.int32), None)
    lin = oracle.w4a8_linear(qa, qw)
    ai = a if sym else a - 128
    assert np.array_equal(lin.acc, ai @ w.T)
    deq_a = al[:, None] * a + (0 if sym else be[:, None])
    np.testing.assert_allclose(lin.y, deq_a @ (ws[:, None] * w).T, rtol=1e-12, atol=1e-12)


def test_w4a8_extreme_codes_fit_int32():
    K = 14336
    qa = oracle.QuantAct(np.full((1, K), -128, np.int32), None, np.ones(1), None, None)
    qw = oracle.QuantWeight(np.full((2, K), -8, np.int32), None, np.ones(2), None, None)
    assert oracle.w4a8_linear(qa, qw).acc.tolist() == [[1024 * K, 1024 * K]]


def test_fp8_gemm_against_numpy_on_decoded_codes():
    rng = np.random.default_rng(3)
    M, N, K = 4, 6, 384
    ac = rng.integers(0, 256, (M, K)).astype(np.uint8)
    wc = rng.integers(0, 256, (N, K)).astype(np.uint8)
    ac[(ac & 0x7F) == 0x7F] = 0   # no NaN patterns
    wc[(wc & 0x7F) == 0x7F] = 0
    al = rng.uniform(0.1, 1, M)
    ws = rng.uniform(0.01, 0.1, N)
    y = oracle.fp8_linear(ac, al, wc, ws)
    want = (al[:, None] * oracle.e4m3_to_f64(ac)) @ (ws[:, None] * oracle.e4m3_to_f64(wc)).T
    np.testing.assert_allclose(y, want, rtol=1e-12, atol=1e-9)
