"""Pins of the oracle's Cayley SGD step (Sec. 3.2) against what the
mathematics fixes: Y is skew-symmetric and, for an orthonormal R, equals
(G R^T - R G^T)/2; the Cayley transform of a skew matrix is orthonormal; the
2 x 2 case is a plane rotation by 2 atan(alpha t / 2) (textbook closed form);
the fixed-point iteration converges to the linear-solve definition, with an
error that shrinks geometrically; a zero gradient leaves R unchanged; and a
small step decreases a quadratic loss."""
import numpy as np
import pytest

import oracle


def _rot(rng, n):
    q, r = np.linalg.qr(rng.standard_normal((n, n)))
    return q * np.sign(np.diag(r))


@pytest.mark.parametrize("n", [2, 7, 16, 64])
def test_y_is_skew_and_matches_the_orthonormal_closed_form(n):
    rng = np.random.default_rng(n)
    R = _rot(rng, n)
    G = rng.standard_normal((n, n))
    Y = oracle.cayley_y(R, G)
    assert np.array_equal(Y, -Y.T)
    # R R^T = I reduces G_hat to G R^T / 2
    np.testing.assert_allclose(Y, 0.5 * (G @ R.T - R @ G.T), atol=1e-12)


def test_y_keeps_the_projection_for_a_non_orthonormal_r():
    """A dropped 1/2 R R^T G R^T term shows only when R R^T != I."""
    rng = np.random.default_rng(3)
    n = 6
    R = rng.standard_normal((n, n))
    G = rng.standard_normal((n, n))
    Gh = G @ R.T - 0.5 * R @ R.T @ G @ R.T
    np.testing.assert_allclose(oracle.cayley_y(R, G), Gh - Gh.T, atol=1e-10)
    assert np.abs(oracle.cayley_y(R, G) - 0.5 * (G @ R.T - R @ G.T)).max() > 1e-3


@pytest.mark.parametrize("t,alpha", [(0.3, 0.5), (-1.2, 0.1), (2.0, 1.5)])
def test_two_by_two_is_a_plane_rotation(t, alpha):
    # R = I, G = [[0, -2t], [0, 0]] gives Y = [[0, -t], [t, 0]]
    G = np.array([[0.0, -2.0 * t], [0.0, 0.0]])
    Y = oracle.cayley_y(np.eye(2), G)
    np.testing.assert_allclose(Y, [[0.0, -t], [t, 0.0]], atol=1e-15)
    # the step uses the Y of -G: a rotation by -2 atan(alpha t / 2)
    th = -2.0 * np.arctan(alpha * t / 2.0)
    want = np.array([[np.cos(th), -np.sin(th)], [np.sin(th), np.cos(th)]])
    np.testing.assert_allclose(oracle.cayley_exact(np.eye(2), G, alpha), want, atol=1e-14)
    if abs(alpha * t / 2.0) < 0.5:   # the fixed-point iteration contracts only for |a Y / 2| < 1
        np.testing.assert_allclose(oracle.cayley_step(np.eye(2), G, alpha, 80)[0], want, atol=1e-13)


@pytest.mark.parametrize("n", [8, 32, 128])
def test_cayley_transform_is_orthonormal(n):
    rng = np.random.default_rng(10 + n)
    R = _rot(rng, n)
    G = rng.standard_normal((n, n))
    alpha = 0.5 / np.abs(oracle.cayley_y(R, G)).sum(axis=1).max()
    Rp = oracle.cayley_exact(R, G, alpha)
    np.testing.assert_allclose(Rp.T @ Rp, np.eye(n), atol=1e-12)


def test_fixed_point_iteration_converges_to_the_solve():
    rng = np.random.default_rng(1)
    n = 32
    R = _rot(rng, n)
    G = rng.standard_normal((n, n))
    alpha = 0.5 / np.linalg.norm(oracle.cayley_y(R, G), 2)   # contraction factor 1/4
    exact = oracle.cayley_exact(R, G, alpha)
    errs = [np.abs(oracle.cayley_step(R, G, alpha, k)[0] - exact).max() for k in range(8)]
    assert errs[-1] < 1e-5
    for a, b in zip(errs, errs[2:]):
        assert b <= 0.25 * a          # the contraction factor 1/4 per step, over two steps
    assert np.abs(oracle.cayley_step(R, G, alpha, 60)[0] - exact).max() < 1e-13
    # iters = 0 is the explicit first step R + a Y R, with Y of -G
    Y = oracle.cayley_y(R, -G)
    np.testing.assert_allclose(oracle.cayley_step(R, G, alpha, 0)[0], R + alpha * Y @ R, atol=1e-13)


def test_zero_gradient_and_batches():
    rng = np.random.default_rng(2)
    R = np.stack([_rot(rng, 16) for _ in range(3)])
    G = rng.standard_normal((3, 16, 16))
    G[1] = 0.0
    out, Y = oracle.cayley_step(R, G, 0.05, 3)
    assert np.array_equal(out[1], R[1]) and not Y[1].any()
    for b in (0, 2):
        np.testing.assert_allclose(out[b], oracle.cayley_step(R[b], G[b], 0.05, 3)[0], atol=0)


def test_small_step_decreases_a_quadratic_loss():
    """L(R) = |R - T|^2 / 2 with gradient G = R - T: one Cayley step with a
    small learning rate lowers L and stays on the orthonormal matrices."""
    rng = np.random.default_rng(4)
    n = 24
    R = _rot(rng, n)
    T = _rot(rng, n)
    G = R - T
    Rp = oracle.cayley_step(R, G, 0.05, 6)[0]
    assert np.linalg.norm(Rp - T) < np.linalg.norm(R - T)
    np.testing.assert_allclose(Rp.T @ Rp, np.eye(n), atol=1e-7)
