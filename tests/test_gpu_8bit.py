"""8-bit variants on the GPU against the oracle: W4A8 (8-bit activation
codes, 4-bit weights, exact integer accumulator) and W-fp8-A-fp8 (E4M3 codes
on both sides), from the rotated quantizers to the fp16 output.

Bars: integer codes within +-1 on at most 1e-4 of the elements, E4M3 codes
within one step of the E4M3 grid on at most 1e-4 (ties of the fp32 quotient
only); scales within 1e-5; the W4A8 accumulator bit-exact given identical
codes; fp16 outputs within 1e-2 relative Frobenius (and elementwise 2e-3
relative + 1e-3 of the largest |y|).  The FP8 output adds fp32 summation
rounding of K terms (|err| <= K 2^-24 sum|a w|); it is held to the same bars."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_16406_gb300 import synth
from parity_util import assert_codes_close, assert_scale_close, assert_zero_close, rel_frob

pytestmark = pytest.mark.gpu


def _planes_to_codes(planes, K):
    p = planes.cpu().numpy()
    c = oracle.e4m3_to_f64(p[:, :K]) + oracle.e4m3_to_f64(p[:, K:])
    return c.astype(np.int64)


def _grid_index(codes_u8):
    """Position of each E4M3 value on the ordered grid (adjacent = one step)."""
    v = oracle.e4m3_to_f64(np.arange(256, dtype=np.uint8))
    grid = np.unique(v[np.isfinite(v)])
    return np.searchsorted(grid, oracle.e4m3_to_f64(codes_u8))


def _assert_e4m3_close(got, ref, what):
    d = np.abs(_grid_index(got).astype(np.int64) - _grid_index(ref))
    assert d.max(initial=0) <= 1, what
    assert np.count_nonzero(d) <= max(1e-4 * d.size, 1), f"{what}: {np.count_nonzero(d)} of {d.size} codes differ"


ACT_CASES = [
    ("none_4096", None, 4096),
    ("h28x512", (28, 512), 14336),
    ("h8192", (1, 8192), 8192),
    ("h12x256", (12, 256), 3072),
    ("h20x256", (20, 256), 5120),
    ("h28x128", (28, 128), 3584),
    ("h256", (1, 256), 256),
]


@pytest.mark.parametrize("name,had,K", ACT_CASES)
@pytest.mark.parametrize("sym", [True, False])
def test_int8_planes_quantizer(name, had, K, sym):
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(K + sym)
    x = synth.activations(rng, 37, K, outlier_frac=0.01, factor=30.0)
    out = spinq.rotate_quant_act8(torch.from_numpy(x).cuda(), had, spinq.SPINQ_FMT_INT8_PLANES, sym)
    torch.cuda.synchronize()
    ref = oracle.rotate_quant_act(x, had, 8, sym, 1.0)
    c = _planes_to_codes(out.codes, K)
    assert_codes_close(c if sym else c + 128, ref.codes, f"int8 {name}")
    assert_scale_close(out.scale.cpu().numpy(), ref.alpha, "alpha")
    if not sym:
        assert_zero_close(out.zero.cpu().numpy(), ref.beta, ref.alpha, "beta")


@pytest.mark.parametrize("name,had,K", ACT_CASES)
def test_fp8_quantizer(name, had, K):
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(K)
    x = synth.activations(rng, 29, K, outlier_frac=0.01, factor=30.0)
    x[3] = 0
    out = spinq.rotate_quant_act8(torch.from_numpy(x).cuda(), had, spinq.SPINQ_FMT_E4M3, True)
    torch.cuda.synchronize()
    ref = oracle.rotate_quant_act_fp8(x, had)
    _assert_e4m3_close(out.codes.cpu().numpy(), ref.codes, f"fp8 {name}")
    assert_scale_close(out.scale.cpu().numpy(), ref.alpha, "alpha")


@pytest.mark.parametrize("fmt,sym", [("e4m3", True), ("planes", True), ("planes", False)])
def test_8bit_quantizers_on_the_tensor_core_rotation(fmt, sym):
    """H28 (x) H512 with at least one row per SM: the FP8 quantizer runs on
    the tcgen05 rotate+quant kernel, the int8 planes on the Paley kernel;
    160 rows (more than the 152 SMs, not a multiple), every row against the
    oracle."""
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(160 + sym)
    x = synth.activations(rng, 160, 14336, outlier_frac=0.01, factor=30.0)
    x[7] = 0
    xt = torch.from_numpy(x).cuda()
    if fmt == "e4m3":
        out = spinq.rotate_quant_act8(xt, (28, 512), spinq.SPINQ_FMT_E4M3, True)
        torch.cuda.synchronize()
        ref = oracle.rotate_quant_act_fp8(x, (28, 512))
        _assert_e4m3_close(out.codes.cpu().numpy(), ref.codes, "fp8 tcgen05")
    else:
        out = spinq.rotate_quant_act8(xt, (28, 512), spinq.SPINQ_FMT_INT8_PLANES, sym)
        torch.cuda.synchronize()
        ref = oracle.rotate_quant_act(x, (28, 512), 8, sym, 1.0)
        c = _planes_to_codes(out.codes, 14336)
        assert_codes_close(c if sym else c + 128, ref.codes, "int8 tcgen05")
        if not sym:
            assert_zero_close(out.zero.cpu().numpy(), ref.beta, ref.alpha, "beta")
    assert_scale_close(out.scale.cpu().numpy(), ref.alpha, "alpha")
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK


def test_clipped_quantizers_saturate_like_the_oracle():
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(5)
    x = synth.activations(rng, 16, 4096, outlier_frac=0.01, factor=30.0)
    xt = torch.from_numpy(x).cuda()
    o8 = spinq.rotate_quant_act8(xt, None, spinq.SPINQ_FMT_INT8_PLANES, False, clip=0.9)
    of = spinq.rotate_quant_act8(xt, None, spinq.SPINQ_FMT_E4M3, True, clip=0.5)
    torch.cuda.synchronize()
    r8 = oracle.rotate_quant_act(x, None, 8, False, 0.9)
    assert_codes_close(_planes_to_codes(o8.codes, 4096) + 128, r8.codes, "int8 clip")
    rf = oracle.rotate_quant_act_fp8(x, None, 0.5)
    _assert_e4m3_close(of.codes.cpu().numpy(), rf.codes, "fp8 clip")


@pytest.mark.parametrize("had,K", [(None, 4096), ((28, 512), 14336), ((1, 8192), 8192)])
def test_weight_quantizers(had, K):
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(K + 1)
    w = synth.weights(rng, 48, K)
    wt = torch.from_numpy(w).cuda()
    q4 = spinq.quant_weight8(wt, had, spinq.SPINQ_FMT_INT4_BYTES)
    q8 = spinq.quant_weight8(wt, had, spinq.SPINQ_FMT_E4M3)
    torch.cuda.synchronize()
    r4 = oracle.quant_weight(w, had)
    g4 = oracle.e4m3_to_f64(q4.codes.cpu().numpy()).astype(np.int64)
    assert_codes_close(g4, r4.codes, "int4 bytes")
    assert np.array_equal(q4.rowsum.cpu().numpy(), g4.sum(axis=1))
    assert_scale_close(q4.scale.cpu().numpy(), r4.scale, "s")
    r8 = oracle.quant_weight_fp8(w, had)
    _assert_e4m3_close(q8.codes.cpu().numpy(), r8.codes, "fp8 weights")
    assert_scale_close(q8.scale.cpu().numpy(), r8.alpha, "s fp8")


def _w4a8_ref(out, wq, K, sym):
    c = _planes_to_codes(out.codes, K)
    codes = c if sym else c + 128
    qa = oracle.QuantAct(codes.astype(np.int32), None, out.scale.double().cpu().numpy(),
                         None if sym else out.zero.double().cpu().numpy(), None)
    wc = oracle.e4m3_to_f64(wq.codes.cpu().numpy()).astype(np.int32)
    qw = oracle.QuantWeight(wc, None, wq.scale.double().cpu().numpy(), wc.sum(1), None)
    return oracle.w4a8_linear(qa, qw)


@pytest.mark.parametrize("M,N,K", [(1, 16, 128), (130, 272, 384), (257, 512, 1024), (64, 4096, 4096)])
@pytest.mark.parametrize("sym", [True, False])
def test_w4a8_gemm_exact_accumulator(M, N, K, sym):
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(M * 7 + N + K)
    x = synth.activations(rng, M, K, outlier_frac=0.01, factor=30.0)
    w = synth.weights(rng, N, K)
    a = spinq.rotate_quant_act8(torch.from_numpy(x).cuda(), None, spinq.SPINQ_FMT_INT8_PLANES, sym)
    wq = spinq.quant_weight8(torch.from_numpy(w).cuda(), None, spinq.SPINQ_FMT_INT4_BYTES)
    y, acc = spinq.w4a8_gemm(a, wq, want_acc=True)
    torch.cuda.synchronize()
    ref = _w4a8_ref(a, wq, K, sym)
    assert np.array_equal(acc.cpu().numpy(), ref.acc)
    yn = y.double().cpu().numpy()
    assert rel_frob(yn, ref.y) <= 1e-2
    assert np.allclose(yn, ref.y, rtol=2e-3, atol=1e-3 * np.abs(ref.y).max())


def test_w4a8_extreme_codes_at_k_16384():
    """All codes at the extremes: |acc| = 1024 K = 2^24 must stay exact."""
    from paper_2405_16406_gb300 import spinq
    M, N, K = 128, 256, 16384
    planes = np.zeros((M, 2 * K), np.uint8)
    planes[:, :K] = oracle.f64_to_e4m3(np.array([-128.0]))[0]     # c = -128 = 16 * -8 + 0
    planes[:, K:] = 0
    wcodes = np.full((N, K), oracle.f64_to_e4m3(np.array([-8.0]))[0], np.uint8)
    a = spinq.ActCodes(torch.from_numpy(planes).cuda(), torch.ones(M, device="cuda"), None)
    wq = spinq.WeightCodes(torch.from_numpy(wcodes).cuda(), torch.full((N,), 1e-4, device="cuda"),
                           torch.full((N,), -8 * K, dtype=torch.int32, device="cuda"))
    _, acc = spinq.w4a8_gemm(a, wq, want_acc=True)
    torch.cuda.synchronize()
    assert bool((acc == 1024 * K).all())


@pytest.mark.parametrize("M,N,K", [(1, 16, 128), (130, 272, 384), (257, 512, 1024), (64, 4096, 4096)])
def test_fp8_gemm(M, N, K):
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(M + N * 3 + K)
    x = synth.activations(rng, M, K, outlier_frac=0.01, factor=30.0)
    w = synth.weights(rng, N, K)
    a = spinq.rotate_quant_act8(torch.from_numpy(x).cuda(), None, spinq.SPINQ_FMT_E4M3, True)
    wq = spinq.quant_weight8(torch.from_numpy(w).cuda(), None, spinq.SPINQ_FMT_E4M3)
    y = spinq.fp8_gemm(a, wq)
    torch.cuda.synchronize()
    ref = oracle.fp8_linear(a.codes.cpu().numpy(), a.scale.double().cpu().numpy(), wq.codes.cpu().numpy(),
                            wq.scale.double().cpu().numpy())
    yn = y.double().cpu().numpy()
    assert rel_frob(yn, ref) <= 1e-3
    assert np.allclose(yn, ref, rtol=2e-3, atol=1e-3 * np.abs(ref).max())


@pytest.mark.parametrize("variant", ["w4a8", "fp8"])
def test_rotated_down_proj_full_size_sampled(variant):
    """Config 3's down_proj (2048 x 14336 -> 4096, online H28 (x) H512) through
    the 8-bit path: codes against the oracle on sampled rows, GEMM outputs
    against the oracle's product of the same codes on sampled entries."""
    from paper_2405_16406_gb300 import spinq
    c = synth.llama3_8b_down_proj()
    xt, wt = torch.from_numpy(c.x).cuda(), torch.from_numpy(c.w).cuda()
    rows = np.array([0, 1, 511, 1024, 2047])
    if variant == "w4a8":
        a = spinq.rotate_quant_act8(xt, c.had, spinq.SPINQ_FMT_INT8_PLANES, True)
        wq = spinq.quant_weight8(wt, c.had, spinq.SPINQ_FMT_INT4_BYTES)
        y = spinq.w4a8_gemm(a, wq)
    else:
        a = spinq.rotate_quant_act8(xt, c.had, spinq.SPINQ_FMT_E4M3, True)
        wq = spinq.quant_weight8(wt, c.had, spinq.SPINQ_FMT_E4M3)
        y = spinq.fp8_gemm(a, wq)
    torch.cuda.synchronize()
    K = c.K
    sub = spinq.ActCodes(a.codes[torch.as_tensor(rows).cuda()], a.scale[torch.as_tensor(rows).cuda()], None)
    if variant == "w4a8":
        ref_rows = oracle.rotate_quant_act(c.x[rows], c.had, 8, True, 1.0)
        assert_codes_close(_planes_to_codes(sub.codes, K), ref_rows.codes, "w4a8 act codes")
        ref = _w4a8_ref(sub, wq, K, True)
        yr = ref.y
    else:
        ref_rows = oracle.rotate_quant_act_fp8(c.x[rows], c.had)
        _assert_e4m3_close(sub.codes.cpu().numpy(), ref_rows.codes, "fp8 act codes")
        yr = oracle.fp8_linear(sub.codes.cpu().numpy(), sub.scale.double().cpu().numpy(), wq.codes.cpu().numpy(),
                               wq.scale.double().cpu().numpy())
    yn = y[torch.as_tensor(rows).cuda()].double().cpu().numpy()
    assert rel_frob(yn, yr) <= 1e-2
    assert np.allclose(yn, yr, rtol=2e-3, atol=1e-3 * np.abs(yr).max())
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK
