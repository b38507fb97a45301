"""The down_proj of Sec. 3.1 in one call (spinq_rotated_linear) and the
random-sign rotation R = S H / sqrt(K) (Sec. 2.2 footnote) on the GPU,
against the oracle.  Bars as the rest of the 4-bit path: codes +-1 on at most
1e-4 of the elements, scales within 1e-5, fp16 outputs within 1e-2 relative
Frobenius and 2e-3 relative + 1e-3 of max|y| elementwise."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_16406_gb300 import synth
from parity_util import assert_codes_close, assert_scale_close, assert_zero_close, gpu_codes, rel_frob

pytestmark = pytest.mark.gpu


def _signs(K, seed):
    return np.random.default_rng(seed).choice([-1.0, 1.0], K)


@pytest.mark.parametrize("had,sym,clip", [
    ((28, 512), True, 1.0),     # Paley kernel
    ((12, 256), False, 1.0),    # Paley kernel through the H24 (x) H128 regrouping
    ((1, 8192), False, 1.0),    # power-of-two kernel
    ((1, 2048), True, 1.0),
    ((1, 256), True, 1.0),      # generic kernel
    ((28, 512), True, 0.9),     # clipped: generic kernel
])
def test_signed_rotate_quant_act(had, sym, clip):
    from paper_2405_16406_gb300 import spinq
    K = had[0] * had[1]
    rng = np.random.default_rng(K + sym)
    x = synth.activations(rng, 45, K, outlier_frac=0.01, factor=30.0)
    s = _signs(K, K)
    out = spinq.rotate_quant_act_signed(torch.from_numpy(x).cuda(), had, spinq.sign_mask(s), sym, clip)
    torch.cuda.synchronize()
    ref = oracle.rotate_quant_act(x, had, 4, sym, clip, signs=s)
    assert_codes_close(gpu_codes(out.codes.cpu().numpy(), sym), ref.codes, f"signed {had}")
    assert_scale_close(out.scale.cpu().numpy(), ref.alpha, "alpha")
    if not sym:
        assert_zero_close(out.zero.cpu().numpy(), ref.beta, ref.alpha, "beta")


def test_signed_weights():
    from paper_2405_16406_gb300 import spinq
    had, K = (28, 512), 14336
    rng = np.random.default_rng(3)
    w = synth.weights(rng, 64, K)
    s = _signs(K, 9)
    q = spinq.quant_weight_signed(torch.from_numpy(w).cuda(), had, spinq.sign_mask(s))
    torch.cuda.synchronize()
    ref = oracle.quant_weight(w, had, signs=s)
    g = gpu_codes(q.codes.cpu().numpy(), True)
    assert_codes_close(g, ref.codes, "signed weights")
    assert np.array_equal(q.rowsum.cpu().numpy(), g.sum(axis=1))
    assert_scale_close(q.scale.cpu().numpy(), ref.scale, "s")


@pytest.mark.parametrize("signed", [False, True])
def test_rotated_linear_config3_full_size(signed):
    """Config 3 (2048 x 14336 -> 4096, online H28 (x) H512) through the one-call
    down_proj: the handed-over codes on sampled rows and the outputs of those
    rows against the oracle chain (oracle codes, oracle weights)."""
    from paper_2405_16406_gb300 import spinq
    c = synth.llama3_8b_down_proj()
    s = _signs(c.K, 17) if signed else None
    mask = spinq.sign_mask(s) if signed else None
    xt, wt = torch.from_numpy(c.x).cuda(), torch.from_numpy(c.w).cuda()
    qw = spinq.quant_weight_signed(wt, c.had, mask) if signed else spinq.quant_weight(wt, c.had)
    ws = torch.empty(spinq.spinq_rotated_linear_workspace_bytes(c.M, c.K), dtype=torch.uint8, device="cuda")
    y = spinq.rotated_linear(xt, c.had, qw, signs=mask, workspace=ws)
    # the same two steps as separate calls give the same bits
    qa = (spinq.rotate_quant_act_signed(xt, c.had, mask) if signed else spinq.rotate_quant_act(xt, c.had))
    y2 = spinq.w4a4_gemm(qa, qw)
    torch.cuda.synchronize()
    assert torch.equal(y, y2)
    codes_ws = ws[: c.M * c.K // 2].view(c.M, c.K // 2)
    assert torch.equal(codes_ws, qa.codes)
    rows = np.array([0, 1, 700, 1403, 2047])
    ra = oracle.rotate_quant_act(c.x[rows], c.had, 4, True, 1.0, signs=s)
    assert_codes_close(gpu_codes(codes_ws.cpu().numpy()[rows], True), ra.codes, "handed-over codes")
    rw = oracle.quant_weight(c.w, c.had, signs=s)
    yn = y.cpu().numpy()[rows].astype(np.float64)
    # the whole chain against the oracle's own codes (independent tie flips
    # on both operands): the task's Frobenius bar
    assert rel_frob(yn, oracle.w4a4_linear(ra, rw).y) <= 1e-2
    # the GEMM on the handed-over codes: the oracle's product of the same codes
    ga = gpu_codes(codes_ws.cpu().numpy()[rows], True)
    gw = gpu_codes(qw.codes.cpu().numpy(), True)
    same = oracle.w4a4_linear(
        oracle.QuantAct(ga, None, qa.scale.double().cpu().numpy()[rows], None, None),
        oracle.QuantWeight(gw, None, qw.scale.double().cpu().numpy(), gw.sum(axis=1), None))
    assert np.allclose(yn, same.y, rtol=2e-3, atol=1e-3 * np.abs(same.y).max())
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK
