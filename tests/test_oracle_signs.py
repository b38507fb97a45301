"""Pins of the random-sign rotation R = S H / sqrt(K) (Sec. 2.2 footnote: a
Hadamard matrix times a random +-1 diagonal S is again a rotation): the
oracle's rotated rows against an explicit numpy product with diag(s) and the
Kronecker factors, orthonormality of S H, the invariance x' W'^T = x W^T
with W' = W S H (Sec. 3.1), and all-plus signs reducing to the plain path."""
import numpy as np
import pytest

import oracle
from paper_2405_16406_gb300 import synth


@pytest.mark.parametrize("had", [(1, 256), (28, 64), (12, 32)])
def test_signed_rotation_against_explicit_product(had):
    rng = np.random.default_rng(sum(had))
    K = had[0] * had[1]
    s = rng.choice([-1.0, 1.0], K)
    x = synth.activations(rng, 6, K, outlier_count=3, factor=20.0)
    q = oracle.rotate_quant_act(x, had, 4, True, 1.0, signs=s)
    H = np.kron(oracle.small_hadamard(had[0]), oracle.sylvester(had[1])).astype(np.float64)
    R = np.diag(s) @ H / np.sqrt(K)
    np.testing.assert_allclose(q.rotated, x.astype(np.float64) @ R, atol=1e-11)
    np.testing.assert_allclose(R @ R.T, np.eye(K), atol=1e-12)
    # unsigned differs (the signs act on the input index)
    assert np.abs(oracle.rotate_quant_act(x, had, 4, True, 1.0).rotated - q.rotated).max() > 1e-3


def test_signed_invariance_and_all_plus():
    rng = np.random.default_rng(5)
    had, K = (28, 64), 28 * 64
    s = rng.choice([-1.0, 1.0], K)
    x = synth.activations(rng, 4, K, outlier_count=2, factor=10.0)
    w = synth.weights(rng, 8, K)
    xr = oracle.rotate_quant_act(x, had, 8, True, 1.0, signs=s).rotated
    wr = oracle.quant_weight(w, had, 8, 1.0, signs=s).rotated
    np.testing.assert_allclose(xr @ wr.T, x.astype(np.float64) @ w.astype(np.float64).T, atol=1e-10)
    plus = np.ones(K)
    a = oracle.rotate_quant_act(x, had, 4, True, 1.0, signs=plus)
    b = oracle.rotate_quant_act(x, had, 4, True, 1.0)
    assert np.array_equal(a.codes, b.codes) and np.array_equal(a.rotated, b.rotated)
