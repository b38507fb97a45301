"""GPU parity: spinq_rotate_quant_act and spinq_quant_weight vs the oracle.

Bars: codes within +-1 on at most 1e-4 of elements (ties at rounding
boundaries); alpha (and beta) within 1e-5 relative.  Every configuration of
the rotated-linear workloads runs at full size; ragged, tiny, clipped and
degenerate rows are covered separately.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_16406_gb300 import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def S():
    from paper_2405_16406_gb300 import spinq
    return spinq


def run_act(S, x16, had, symmetric, clip):
    x = torch.from_numpy(x16).cuda()
    out = S.rotate_quant_act(x, had, symmetric, clip)
    torch.cuda.synchronize()
    return (out.codes.cpu().numpy(), out.scale.cpu().numpy(),
            None if out.zero is None else out.zero.cpu().numpy())


def check_act(S, x16, had, symmetric, clip, what):
    codes, scale, zero = run_act(S, x16, had, symmetric, clip)
    ref = oracle.rotate_quant_act(x16, had, 4, symmetric, clip)
    got = pu.gpu_codes(codes, symmetric)
    frac = pu.assert_codes_close(got, ref.codes, what)
    pu.assert_scale_close(scale, ref.alpha, what + " alpha")
    if not symmetric:
        pu.assert_zero_close(zero, ref.beta, ref.alpha, what + " beta")
    return frac


CASES = [
    ("tiny", synth.tiny_linear, {}),
    ("gate_up", synth.llama3_8b_gate_up, {}),
    ("down_proj", synth.llama3_8b_down_proj, {}),
    ("l32_up_M1", synth.llama32_3b_up, {"M": 1}),
    ("l32_up_M16", synth.llama32_3b_up, {"M": 16}),
    ("l32_up_M128", synth.llama32_3b_up, {"M": 128}),
    ("l32_up_M8192", synth.llama32_3b_up, {"M": 8192}),
    ("l32_down_M1", synth.llama32_3b_down, {"M": 1}),
    ("l32_down_M16", synth.llama32_3b_down, {"M": 16}),
    ("l32_down_M128", synth.llama32_3b_down, {"M": 128}),
    ("l32_down_M8192", synth.llama32_3b_down, {"M": 8192}),
]


@pytest.mark.parametrize("name,builder,kw", CASES, ids=[c[0] for c in CASES])
def test_act_full_configs(S, name, builder, kw):
    c = builder(**kw)
    check_act(S, c.x, c.had, c.act_symmetric, c.clip, name)


@pytest.mark.parametrize("had", [None, (1, 32), (1, 256), (1, 512), (1, 1024), (1, 2048), (1, 4096), (1, 8192),
                                 (1, 16384), (12, 64), (12, 128), (12, 256), (12, 512), (20, 128), (20, 256),
                                 (20, 512), (28, 64), (28, 128), (28, 256), (28, 512)])
@pytest.mark.parametrize("symmetric", [True, False])
def test_act_shapes_and_modes(S, had, symmetric):
    K = 4096 if had is None else had[0] * had[1]
    rng = np.random.default_rng(K + symmetric)
    x = synth.activations(rng, 37, K, outlier_frac=0.02, factor=25.0)
    check_act(S, x, had, symmetric, 1.0, f"had={had} sym={symmetric}")


@pytest.mark.parametrize("had,rows", [((1, 8192), 306), ((1, 8192), 2), ((1, 16384), 153), ((12, 512), 306),
                                      ((12, 512), 305), ((20, 512), 160), ((12, 256), 612), ((12, 256), 610)])
@pytest.mark.parametrize("symmetric", [True, False])
def test_act_tensor_core_rotation_shapes(S, had, rows, symmetric):
    """The tcgen05 rotate+quant kernel (at least one MMA per SM): Sylvester
    8192 (two rows per MMA) and 16384, Paley factors with few and many lanes
    (H_12 (x) H_512: two rows per MMA sharing warps); odd and small row
    counts take the other kernels."""
    K = had[0] * had[1]
    rng = np.random.default_rng(K + rows + symmetric)
    x = synth.activations(rng, rows, K, outlier_frac=0.02, factor=25.0)
    check_act(S, x, had, symmetric, 1.0, f"had={had} rows={rows} sym={symmetric}")


@pytest.mark.parametrize("had,rows", [((12, 256), 64), ((28, 512), 64), ((28, 512), 160), ((1, 8192), 320)])
@pytest.mark.parametrize("symmetric,clip", [(True, 0.9), (False, 0.9), (False, 0.5)])
def test_act_clipping(S, had, rows, symmetric, clip):
    rng = np.random.default_rng(9)
    x = synth.activations(rng, rows, had[0] * had[1], outlier_frac=0.01, factor=30.0)
    check_act(S, x, had, symmetric, clip, f"had={had} clip={clip}")


def test_act_degenerate_rows(S):
    x = np.zeros((6, 256), dtype=np.float16)
    x[1] = 3.0                                   # constant row
    x[2, 7] = -2.0                               # one nonzero
    x[3] = np.float16(65504.0)                   # largest fp16
    x[4, ::2] = 1.0
    x[4, 1::2] = -1.0
    for sym in (True, False):
        for had in (None, (1, 256)):
            check_act(S, x, had, sym, 1.0, f"degenerate sym={sym} had={had}")


@pytest.mark.parametrize("had", [None, (1, 512), (12, 256)])
def test_act_strided_rows(S, had):
    K = 4096 if had is None else had[0] * had[1]
    rng = np.random.default_rng(1)
    big = synth.activations(rng, 19, K + 64, outlier_frac=0.01, factor=10.0)
    x = torch.from_numpy(big).cuda()[:, :K]
    out = S.rotate_quant_act(x, had, True, 1.0)
    ref = oracle.rotate_quant_act(np.ascontiguousarray(big[:, :K]), had, 4, True, 1.0)
    pu.assert_codes_close(pu.gpu_codes(out.codes.cpu().numpy(), True), ref.codes, "strided")


def test_act_empty(S):
    x = torch.empty((0, 256), dtype=torch.float16, device="cuda")
    out = S.rotate_quant_act(x, (1, 256), True, 1.0)
    assert out.codes.shape == (0, 128)


WCASES = [
    ("tiny", synth.tiny_linear, {}),
    ("gate_up", synth.llama3_8b_gate_up, {"M": 1}),
    ("down_proj", synth.llama3_8b_down_proj, {"M": 1}),
    ("l32_up", synth.llama32_3b_up, {"M": 1}),
    ("l32_down", synth.llama32_3b_down, {"M": 1}),
]


@pytest.mark.parametrize("name,builder,kw", WCASES, ids=[c[0] for c in WCASES])
def test_weight_full_configs(S, name, builder, kw):
    c = builder(**kw)
    w = torch.from_numpy(c.w).cuda()
    out = S.quant_weight(w, c.had, 1.0)
    torch.cuda.synchronize()
    ref = oracle.quant_weight(c.w, c.had)
    got = pu.gpu_codes(out.codes.cpu().numpy(), True)
    pu.assert_codes_close(got, ref.codes, name)
    pu.assert_scale_close(out.scale.cpu().numpy(), ref.scale, name + " scale")
    # the row sum is the sum of the codes the GPU produced, exactly
    assert np.array_equal(out.rowsum.cpu().numpy(), got.sum(1))


def test_weight_clip(S):
    rng = np.random.default_rng(4)
    w = synth.weights(rng, 96, 1024)
    out = S.quant_weight(torch.from_numpy(w).cuda(), (1, 1024), 0.9)
    ref = oracle.quant_weight(w, (1, 1024), 4, 0.9)
    got = pu.gpu_codes(out.codes.cpu().numpy(), True)
    pu.assert_codes_close(got, ref.codes, "weight clip")
    assert got.min() >= -8
