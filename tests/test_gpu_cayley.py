"""Cayley SGD step on the GPU (spinq_cayley_step) against the oracle
(Sec. 3.2): the same fixed-point iterate R'_iters and the same Y, for every
supported n, several iteration counts, a batch of 32 head-dim rotations (one
R2 per layer of a 32-layer model) and the in-place form.

Tolerance: fp32 products of length n <= 128 against the double oracle.  Each
entry of R' is R plus a handful of chained n-term products whose terms are
bounded by the inputs' magnitudes (|R| <= 1, |alpha Y| <= ~0.5), so the
accumulated rounding stays below ~n * 2^-24 * 4 ~ 3e-5; the test uses 5e-5
absolute on R' and 1e-5 relative to max|Y| on Y."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _case(seed, batch, n):
    rng = np.random.default_rng(seed)
    R = np.empty((batch, n, n))
    for b in range(batch):
        q, r = np.linalg.qr(rng.standard_normal((n, n)))
        R[b] = q * np.sign(np.diag(r))
    grad = 0.5 * rng.standard_normal((batch, n, n))
    R32 = R.astype(np.float32)
    g32 = grad.astype(np.float32)
    Y = np.stack([oracle.cayley_y(R32[b].astype(np.float64), -g32[b].astype(np.float64)) for b in range(batch)])
    alpha = 0.4 / max(np.linalg.norm(Y[b], 2) for b in range(batch))   # |alpha Y / 2| <= 0.2
    return R32, g32, np.float32(alpha)


@pytest.mark.parametrize("n", [16, 32, 64, 128])
@pytest.mark.parametrize("iters", [0, 2, 5])
def test_cayley_step_matches_oracle(n, iters):
    from paper_2405_16406_gb300 import spinq
    R, g, alpha = _case(100 + n + iters, 3, n)
    out, y = spinq.cayley_step(torch.from_numpy(R).cuda(), torch.from_numpy(g).cuda(), float(alpha), iters,
                               want_y=True)
    torch.cuda.synchronize()
    ref, yref = oracle.cayley_step(R.astype(np.float64), g.astype(np.float64), float(alpha), iters)
    got = out.cpu().numpy().astype(np.float64)
    assert np.abs(got - ref).max() <= 5e-5
    yg = y.cpu().numpy().astype(np.float64)
    assert np.abs(yg - yref).max() <= 1e-5 * np.abs(yref).max()
    assert np.array_equal(yg, -np.swapaxes(yg, 1, 2))     # Y is formed as G_hat - G_hat^T


def test_cayley_step_batch_of_32_head_rotations_stays_orthonormal():
    from paper_2405_16406_gb300 import spinq
    R, g, alpha = _case(7, 32, 128)
    out = spinq.cayley_step(torch.from_numpy(R).cuda(), torch.from_numpy(g).cuda(), float(alpha), 6)
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.float64)
    ref, _ = oracle.cayley_step(R.astype(np.float64), g.astype(np.float64), float(alpha), 6)
    assert np.abs(got - ref).max() <= 5e-5
    eye = np.eye(128)
    for b in range(32):
        exact = oracle.cayley_exact(R[b].astype(np.float64), g[b].astype(np.float64), float(alpha))
        assert np.abs(got[b] - exact).max() <= 1e-4             # 6 iterations of a 0.2 contraction
        assert np.abs(got[b].T @ got[b] - eye).max() <= 2e-4


def test_cayley_step_in_place_and_empty():
    from paper_2405_16406_gb300 import spinq
    R, g, alpha = _case(9, 2, 64)
    Rt = torch.from_numpy(R).cuda()
    ref = spinq.cayley_step(Rt, torch.from_numpy(g).cuda(), float(alpha), 3)
    spinq.cayley_step(Rt, torch.from_numpy(g).cuda(), float(alpha), 3, out=Rt)
    torch.cuda.synchronize()
    assert torch.equal(Rt, ref)
    empty = torch.empty((0, 64, 64), device="cuda")
    assert spinq.cayley_step(empty, empty, 0.1, 2).shape == (0, 64, 64)
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK
