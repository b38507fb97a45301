"""Pins for the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a library
routine (numpy / scipy), a closed form, a hand-computed example, or an
invariant the paper states.  A plausible mistake anywhere in the oracle (a
dropped term, a wrong sign or index, a transposed Hadamard factor, a wrong
rounding rule) fails at least one of them.
"""
import json
import os

import numpy as np
import pytest
import scipy.linalg

import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- fp16 codec
def test_f16_decode_all_bit_patterns_match_numpy():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ours = oracle.f16_to_f64(bits)
    ref = bits.view(np.float16).astype(np.float64)
    finite = np.isfinite(ref)
    assert np.array_equal(ours[finite], ref[finite])
    assert np.array_equal(np.isnan(ours), np.isnan(ref))
    assert np.array_equal(ours[np.isinf(ref)], ref[np.isinf(ref)])


def test_f16_encode_round_half_even_matches_numpy():
    rng = np.random.default_rng(1)
    vals = np.concatenate([
        rng.standard_normal(200000) * 10.0,
        rng.standard_normal(20000) * 1e-6,        # subnormal range
        rng.uniform(60000, 70000, 2000),          # overflow edge
        # exact ties between two binary16 neighbours
        (np.arange(1, 2048, dtype=np.float64) + 0.5) * 2.0 ** -10,
        (np.arange(1, 1024, dtype=np.float64) + 0.5) * 2.0 ** -24,
        np.array([65504.0, 65519.99, 65520.0, -65520.0, 0.0, -0.0, 2.0 ** -25, 3 * 2.0 ** -26]),
    ])
    ours = oracle.f64_to_f16(vals).view(np.uint16)
    with np.errstate(over="ignore"):
        ref = vals.astype(np.float16).view(np.uint16)
    assert np.array_equal(ours, ref)


# ---------------------------------------------------------- Hadamard matrices
@pytest.mark.parametrize("n", [1, 2, 4, 8, 16, 128, 1024])
def test_sylvester_equals_scipy(n):
    assert np.array_equal(oracle.sylvester(n), scipy.linalg.hadamard(n))


@pytest.mark.parametrize("q", [11, 19, 27, 43, 59])
def test_paley1_is_skew_hadamard(q):
    H = oracle.paley1(q).astype(np.int64)
    n = q + 1
    assert set(np.unique(H)) == {-1, 1}
    assert np.array_equal(H @ H.T, n * np.eye(n, dtype=np.int64))   # Hadamard: H H^T = n I
    assert np.array_equal(H + H.T, 2 * np.eye(n, dtype=np.int64))   # Paley I is skew: S^T = -S
    assert np.all(H[0] == 1)                                        # border row of ones
    assert np.all(H[1:, 0] == -1)                                   # border column of -1


def test_paley_core_uses_textbook_quadratic_residues():
    gold = json.load(open(os.path.join(GOLD, "quadratic_residues.json")))
    for q in (11, 19):
        qr = set(gold[str(q)])
        H = oracle.paley1(q)
        for i in range(q):
            for j in range(q):
                if i == j:
                    continue
                expect = 1 if ((i - j) % q) in qr else -1
                assert H[i + 1, j + 1] == expect


def test_paley_gf27_polynomial_is_irreducible_and_matrix_is_not_symmetric():
    # t^3 + 2t + 1 has no root in GF(3), so it is irreducible (degree 3)
    assert all((t ** 3 + 2 * t + 1) % 3 != 0 for t in range(3))
    H = oracle.small_hadamard(28)
    assert not np.array_equal(H, H.T)


def test_unsupported_orders_rejected():
    for q in (7 * 3, 13, 25):  # 21 not prime power, 13 = 1 mod 4, 25 = 1 mod 4
        with pytest.raises(ValueError):
            oracle.paley1(q)
    with pytest.raises(ValueError):
        oracle.sylvester(12)


# ----------------------------------------------------------------- FWHT / R
@pytest.mark.parametrize("n", [2, 16, 256, 4096])
def test_fwht_equals_dense_sylvester(n):
    rng = np.random.default_rng(n)
    v = rng.standard_normal(n)
    ref = scipy.linalg.hadamard(n).astype(np.float64) @ v
    assert np.allclose(oracle.fwht(v), ref, rtol=0, atol=1e-9 * np.sqrt(n))


@pytest.mark.parametrize("n_s,P", [(1, 256), (1, 2048), (12, 64), (12, 256), (20, 32), (28, 32), (28, 128)])
def test_rotate_equals_explicit_kronecker_row_vector_product(n_s, P):
    rng = np.random.default_rng(n_s * 1000 + P)
    K = n_s * P
    x = rng.standard_normal((5, K))
    Hs = oracle.small_hadamard(n_s).astype(np.float64)
    Hp = scipy.linalg.hadamard(P).astype(np.float64)
    R = np.kron(Hs, Hp) / np.sqrt(K)          # small factor on the slow index
    ref = x @ R                                # row-vector product x R
    assert np.allclose(oracle.rotate(x, n_s, P), ref, rtol=0, atol=1e-10)
    if n_s > 1:
        # the transposed convention must give a different answer (Paley H is not symmetric)
        assert not np.allclose(oracle.rotate(x, n_s, P), x @ R.T, atol=1e-6)


@pytest.mark.parametrize("n_s,P", [(1, 128), (12, 16), (28, 16)])
def test_rotation_is_orthonormal(n_s, P):
    K = n_s * P
    R = oracle.rotate(np.eye(K), n_s, P)      # rows of I times R = R
    assert np.allclose(R @ R.T, np.eye(K), atol=1e-12)


@pytest.mark.parametrize("n_s,P", [(1, 256), (28, 16)])
def test_rotational_invariance_sec31(n_s, P):
    # Sec. 3.1: with no quantization the rotated layer equals the original one.
    rng = np.random.default_rng(7)
    K = n_s * P
    x = rng.standard_normal((9, K))
    W = rng.standard_normal((13, K)) * 0.02
    ref = x @ W.T
    rot = oracle.rotate(x, n_s, P) @ oracle.rotate(W, n_s, P).T
    assert np.linalg.norm(rot - ref) / np.linalg.norm(ref) < 1e-12
    # the same check in fp32 arithmetic on the rotated operands (spec bar 1e-3)
    r32 = oracle.rotate(x, n_s, P).astype(np.float32) @ oracle.rotate(W, n_s, P).astype(np.float32).T
    assert np.linalg.norm(r32 - ref) / np.linalg.norm(ref) < 1e-3


def test_rotation_removes_outliers_kurtosis():
    # Sec. 2.1 / Fig. 2: outlier channels give large kurtosis; after a
    # Hadamard rotation the distribution is close to Gaussian (kappa ~ 3).
    from paper_2405_16406_gb300 import synth
    rng = np.random.default_rng(3)
    x = synth.activations(rng, 64, 4096, outlier_frac=0.01, factor=30.0)
    xd = oracle.f16_to_f64(x)

    def kurt(a):
        a = a - a.mean()
        return float(np.mean(a ** 4) / np.mean(a ** 2) ** 2)

    assert kurt(xd) > 20.0
    assert abs(kurt(oracle.rotate(xd, 1, 4096)) - 3.0) < 0.3


def test_two_d_example_45_degrees():
    # Sec. 4 illustrative analysis: a 45-degree rotation (H_2 / sqrt 2) equalises
    # the range of a 2-D activation dominated by one axis.
    y = oracle.rotate(np.array([[2.0, 0.0]]), 1, 2)[0]
    assert np.allclose(y, [np.sqrt(2.0), np.sqrt(2.0)])


# ----------------------------------------------------------------- Eq. 1
def test_eq1_hand_computed_examples():
    gold = json.load(open(os.path.join(GOLD, "eq1_worked_examples.json")))
    for case in gold["cases"]:
        x = np.array([case["x"]], dtype=np.float64)
        codes, a, b = oracle.quantize_rows(x, case["bits"], case["symmetric"], case["clip"])
        assert codes[0].tolist() == case["codes"], case["why"]
        assert a[0] == pytest.approx(case["alpha"], rel=1e-15, abs=0)
        assert b[0] == pytest.approx(case["beta"], rel=1e-15, abs=0)


@pytest.mark.parametrize("symmetric", [True, False])
def test_eq1_properties_random(symmetric):
    rng = np.random.default_rng(11)
    x = rng.standard_normal((200, 257)) * rng.uniform(0.1, 10, (200, 1))
    codes, a, b = oracle.quantize_rows(x, 4, symmetric, 1.0)
    deq = oracle.dequantize_rows(codes, a, None if symmetric else b)
    assert np.all(np.abs(x - deq) <= a[:, None] / 2 * (1 + 1e-12))   # unclipped error <= alpha/2
    if symmetric:
        assert codes.min() >= -7 and codes.max() <= 7                 # -8 unreachable unclipped
        am = np.argmax(np.abs(x), axis=1)
        assert np.all(np.abs(codes[np.arange(200), am]) == 7)         # max maps to +-7
        assert np.allclose(a, np.abs(x).max(1) / 7)
    else:
        assert codes.min() >= 0 and codes.max() <= 15
        assert np.all(codes[np.arange(200), np.argmin(x, 1)] == 0)   # min -> 0
        assert np.all(codes[np.arange(200), np.argmax(x, 1)] == 15)  # max -> 15
        assert np.allclose(b, x.min(1))
        assert np.allclose(a, (x.max(1) - x.min(1)) / 15)


def test_eq1_clipping_saturates():
    rng = np.random.default_rng(5)
    x = rng.standard_normal((50, 128))
    codes, a, _ = oracle.quantize_rows(x, 4, True, 0.9)
    assert codes.min() >= -8 and codes.max() <= 7
    assert np.allclose(a, 0.9 * np.abs(x).max(1) / 7)
    codes, a, b = oracle.quantize_rows(x, 4, False, 0.95)
    assert np.allclose(b, 0.95 * x.min(1)) and np.allclose(a, 0.95 * (x.max(1) - x.min(1)) / 15)


def test_pack4_nibble_order_and_roundtrip():
    codes = np.array([[1, -2, 7, -8, 0, 5]], dtype=np.int32)
    p = oracle.pack4(codes)
    assert p.tolist() == [[0xE1, 0x87, 0x50]]        # even index in the low nibble
    assert np.array_equal(oracle.unpack4(p, True), codes)
    u = np.array([[0, 15, 8, 3]], dtype=np.int32)
    assert np.array_equal(oracle.unpack4(oracle.pack4(u), False), u)


# ----------------------------------------------------------------- GEMM
@pytest.mark.parametrize("symmetric", [True, False])
def test_gemm_acc_equals_numpy_int64(symmetric):
    rng = np.random.default_rng(2)
    M, N, K = 7, 9, 64
    ac = rng.integers(-8, 8, (M, K)) if symmetric else rng.integers(0, 16, (M, K))
    wc = rng.integers(-8, 8, (N, K))
    al = rng.uniform(0.1, 1, M)
    be = None if symmetric else rng.uniform(-2, 0, M)
    ws = rng.uniform(0.001, 0.01, N)
    a = oracle.QuantAct(ac.astype(np.int32), None, al, be, None)
    w = oracle.QuantWeight(wc.astype(np.int32), None, ws, wc.sum(1).astype(np.int32), None)
    out = oracle.w4a4_linear(a, w)
    a_int = ac if symmetric else ac - 8
    assert np.array_equal(out.acc, (a_int.astype(np.int64) @ wc.T.astype(np.int64)))
    # y is the dequantized product (Eq. 1 on both operands)
    deq_a = al[:, None] * ac + (0 if symmetric else be[:, None])
    deq_w = ws[:, None] * wc
    assert np.allclose(out.y, deq_a @ deq_w.T, rtol=1e-12, atol=1e-15)
    # epilogue identity used by the kernels: y = a s acc + b' s rowsum, b' = beta + 8 alpha (asym)
    bp = 0 if symmetric else (be + 8 * al)[:, None]
    ident = al[:, None] * ws[None, :] * out.acc + bp * ws[None, :] * wc.sum(1)[None, :]
    assert np.allclose(out.y, ident, rtol=1e-12, atol=1e-15)
    # fp16 output is y rounded once
    assert np.array_equal(out.y_f16, out.y.astype(np.float16))


def test_gemm_extreme_codes_long_k():
    K = 14336
    ac = np.full((2, K), -8, dtype=np.int32)
    wc = np.full((3, K), -8, dtype=np.int32)
    a = oracle.QuantAct(ac, None, np.ones(2), None, None)
    w = oracle.QuantWeight(wc, None, np.ones(3), wc.sum(1).astype(np.int32), None)
    out = oracle.w4a4_linear(a, w)
    assert np.all(out.acc == 64 * K)
    # asymmetric u = 0 is a zero-centred code of -8 as well
    a2 = oracle.QuantAct(np.zeros((2, K), np.int32), None, np.ones(2), np.zeros(2), None)
    assert np.all(oracle.w4a4_linear(a2, w).acc == 64 * K)


def test_gemm_sampled_matches_full():
    rng = np.random.default_rng(4)
    M, N, K = 11, 13, 96
    ac = rng.integers(0, 16, (M, K)).astype(np.int32)
    wc = rng.integers(-8, 8, (N, K)).astype(np.int32)
    al, be, ws = rng.uniform(0.1, 1, M), rng.uniform(-1, 0, M), rng.uniform(0.01, 0.1, N)
    full = oracle.w4a4_linear(oracle.QuantAct(ac, None, al, be, None),
                              oracle.QuantWeight(wc, None, ws, wc.sum(1).astype(np.int32), None))
    ms = rng.integers(0, M, 40)
    ns = rng.integers(0, N, 40)
    acc, y = oracle.w4a4_linear_sampled(ac, al, be, wc, ws, ms, ns)
    assert np.array_equal(acc, full.acc[ms, ns])
    assert np.array_equal(y, full.y[ms, ns])


# ----------------------------------------------------------------- composites
def test_rotate_quant_act_composition():
    from paper_2405_16406_gb300 import synth
    c = synth.tiny_linear()
    out = oracle.rotate_quant_act(c.x, c.had, 4, c.act_symmetric, c.clip)
    xd = c.x.astype(np.float64)
    ref = xd @ (scipy.linalg.hadamard(256) / 16.0)
    assert np.allclose(out.rotated, ref, atol=1e-12)
    assert np.all(np.abs(out.codes).max(1) == 7)
    assert np.allclose(out.alpha, np.abs(ref).max(1) / 7)


def test_quant_weight_merge_keeps_linear_invariant():
    from paper_2405_16406_gb300 import synth
    c = synth.tiny_linear()
    qw = oracle.quant_weight(c.w, c.had)
    xd, wd = c.x.astype(np.float64), c.w.astype(np.float64)
    xr = oracle.rotate(xd, *c.had)
    assert np.allclose(xr @ qw.rotated.T, xd @ wd.T, atol=1e-10)
    assert np.array_equal(qw.rowsum, qw.codes.sum(1))


def test_kv_composition():
    from paper_2405_16406_gb300 import synth
    c = synth.kv_case(B=1, S=3, Hq=4, Hkv=2, D=128)
    out = oracle.rotate_quant_kv(c.q, c.k, c.v, c.had)
    H = scipy.linalg.hadamard(128) / np.sqrt(128)
    qref = c.q.astype(np.float64) @ H
    assert np.array_equal(out.q_out, qref.astype(np.float16))
    kref = c.k.astype(np.float64) @ H
    assert np.allclose(out.k_rot, kref, atol=1e-12)
    assert out.k_codes.min() >= 0 and out.k_codes.max() <= 15
    kk = kref.reshape(-1, 128)
    assert np.allclose(out.k_beta.reshape(-1), kk.min(1))
    assert np.allclose(out.k_alpha.reshape(-1), (kk.max(1) - kk.min(1)) / 15)
    vv = c.v.astype(np.float64).reshape(-1, 128)
    assert np.allclose(out.v_beta.reshape(-1), vv.min(1))
