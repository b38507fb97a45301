"""GPU parity: spinq_w4a4_gemm vs the oracle.

Bars: the int32 accumulator is bit-exact given identical codes (the oracle's
codes are fed to the GPU); the fp16 output is within 1e-2 relative Frobenius
error of the oracle's double-precision dequantized product.  Full-size
workloads are checked on sampled outputs the oracle computes one by one.
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


def to_gpu_act(S, a_codes, alpha, beta):
    packed = oracle.pack4(a_codes)
    return S.ActCodes(torch.from_numpy(packed).cuda(),
                      torch.from_numpy(alpha.astype(np.float32)).cuda(),
                      None if beta is None else torch.from_numpy(beta.astype(np.float32)).cuda())


def to_gpu_w(S, w_codes, scale):
    return S.WeightCodes(torch.from_numpy(oracle.pack4(w_codes)).cuda(),
                         torch.from_numpy(scale.astype(np.float32)).cuda(),
                         torch.from_numpy(w_codes.sum(1).astype(np.int32)).cuda())


def run(S, ac, al, be, wc, ws):
    a = to_gpu_act(S, ac, al, be)
    w = to_gpu_w(S, wc, ws)
    y, acc = S.w4a4_gemm(a, w, want_acc=True)
    torch.cuda.synchronize()
    return y.cpu().numpy(), acc.cpu().numpy()


def oracle_full(ac, al, be, wc, ws):
    # alpha / beta / scale as the fp32 values the GPU receives
    al32 = al.astype(np.float32).astype(np.float64)
    be32 = None if be is None else be.astype(np.float32).astype(np.float64)
    ws32 = ws.astype(np.float32).astype(np.float64)
    a = oracle.QuantAct(ac, None, al32, be32, None)
    w = oracle.QuantWeight(wc, None, ws32, wc.sum(1).astype(np.int32), None)
    return oracle.w4a4_linear(a, w)


def random_codes(rng, M, N, K, symmetric):
    ac = (rng.integers(-8, 8, (M, K)) if symmetric else rng.integers(0, 16, (M, K))).astype(np.int32)
    wc = rng.integers(-8, 8, (N, K)).astype(np.int32)
    al = rng.uniform(0.01, 1.0, M)
    be = None if symmetric else rng.uniform(-3.0, 0.0, M)
    ws = rng.uniform(1e-3, 1e-2, N)
    return ac, al, be, wc, ws


@pytest.mark.parametrize("M,N,K", [(1, 16, 128), (3, 48, 256), (128, 256, 128), (130, 272, 384),
                                   (257, 512, 1024), (16, 512, 256), (200, 4096, 512)])
@pytest.mark.parametrize("symmetric", [True, False])
def test_gemm_random_codes_exact(S, M, N, K, symmetric):
    rng = np.random.default_rng(M * 7 + N + K + symmetric)
    ac, al, be, wc, ws = random_codes(rng, M, N, K, symmetric)
    y, acc = run(S, ac, al, be, wc, ws)
    ref = oracle_full(ac, al, be, wc, ws)
    assert np.array_equal(acc, ref.acc)
    assert pu.rel_frob(y, ref.y) <= pu.Y_REL_FROB
    # elementwise: fp32 epilogue then one fp16 rounding
    assert np.allclose(y.astype(np.float64), ref.y, rtol=2e-3, atol=1e-3 * np.abs(ref.y).max())


@pytest.fixture
def gemm_kernel(S, request):
    """Forces one prefill GEMM kernel for the test and restores the default."""
    prev = S.spinq_gemm_select_kernel(request.param)
    assert prev >= 0
    yield request.param
    S.spinq_gemm_select_kernel(prev)


KERNELS = [1, 2, 3]   # 128 x 256 tiles, 256 x 256 tiles, 256 x 256 tiles on SM pairs


@pytest.mark.parametrize("gemm_kernel", KERNELS, indirect=True, ids=["tile128", "tile256", "pair"])
@pytest.mark.parametrize("M,N,K", [(129, 256, 128), (300, 528, 384), (1000, 1040, 1024), (2001, 784, 512),
                                   (513, 4096, 2048)])
@pytest.mark.parametrize("symmetric", [True, False])
def test_gemm_each_kernel_exact(S, gemm_kernel, M, N, K, symmetric):
    """Every prefill kernel, forced, on ragged M and N (partial tiles and SM
    pairs whose second CTA lies partly or wholly below M)."""
    rng = np.random.default_rng(M * 5 + N * 3 + K + symmetric)
    ac, al, be, wc, ws = random_codes(rng, M, N, K, symmetric)
    y, acc = run(S, ac, al, be, wc, ws)
    ref = oracle_full(ac, al, be, wc, ws)
    assert np.array_equal(acc, ref.acc)
    assert pu.rel_frob(y, ref.y) <= pu.Y_REL_FROB
    assert np.allclose(y.astype(np.float64), ref.y, rtol=2e-3, atol=1e-3 * np.abs(ref.y).max())
    st, _ = S.spinq_device_status()
    assert st == S.SPINQ_OK


@pytest.mark.parametrize("gemm_kernel", KERNELS, indirect=True, ids=["tile128", "tile256", "pair"])
def test_gemm_each_kernel_same_bits(S, gemm_kernel):
    """The kernels agree bit for bit (y and acc) with the automatic choice."""
    rng = np.random.default_rng(11)
    M, N, K = 777, 1296, 1536
    ac, al, be, wc, ws = random_codes(rng, M, N, K, False)
    y, acc = run(S, ac, al, be, wc, ws)
    prev = S.spinq_gemm_select_kernel(0)
    try:
        y0, acc0 = run(S, ac, al, be, wc, ws)
    finally:
        S.spinq_gemm_select_kernel(prev)
    assert np.array_equal(acc, acc0)
    assert np.array_equal(y.view(np.uint16), y0.view(np.uint16))


def test_gemm_select_kernel_rejects_unknown(S):
    assert S.spinq_gemm_select_kernel(S.SPINQ_GEMM_TCGEMV + 1) == -1
    assert S.spinq_gemm_select_kernel(-1) == -1
    assert S.spinq_gemm_select_kernel(0) == 0


def test_gemm_plan_follows_selection(S):
    assert S.spinq_w4a4_gemm_plan(2048, 4100, 4096) == -1   # N not a multiple of 16
    assert S.spinq_w4a4_gemm_plan(2048, 14336, 4000) == -1  # K not a multiple of 128
    for kind in (1, 2, 3):
        prev = S.spinq_gemm_select_kernel(kind)
        try:
            assert S.spinq_w4a4_gemm_plan(2048, 14336, 4096) == kind
            small = S.spinq_w4a4_gemm_plan(128, 14336, 4096)
            # SM pairs need more than 128 rows: the cost model decides there
            assert small == kind if kind != 3 else small in (1, 2)
        finally:
            S.spinq_gemm_select_kernel(prev)
    assert S.spinq_w4a4_gemm_plan(128, 14336, 4096) in (1, 2)
    assert S.spinq_w4a4_gemm_plan(2048, 14336, 4096) in (1, 2, 3)
    assert S.spinq_w4a4_gemm_plan(2, 14336, 4096) == 4      # one or two tokens: GEMV
    assert S.spinq_w4a4_gemm_plan(3, 14336, 4096) == 6      # 3 to 16: the tensor-core GEMV
    assert S.spinq_gemm_select_kernel(S.SPINQ_GEMM_TCGEMV + 1) == -1


@pytest.mark.parametrize("symmetric", [True, False])
def test_gemm_extreme_codes_long_k(S, symmetric):
    # largest accumulator magnitudes: every product at its extreme, K = 65536
    M, N, K = 130, 144, 65536
    for aval, wval in ((7, 7), (-8, -8), (7, -8)):
        ac = np.full((M, K), aval if symmetric else aval + 8, dtype=np.int32)
        wc = np.full((N, K), wval, dtype=np.int32)
        al, ws = np.full(M, 0.5), np.full(N, 0.25)
        be = None if symmetric else np.full(M, -1.0)
        y, acc = run(S, ac, al, be, wc, ws)
        ref = oracle_full(ac, al, be, wc, ws)
        assert np.array_equal(acc, ref.acc), (aval, wval)


def test_gemm_alternating_and_sparse_codes(S):
    M, N, K = 128, 256, 4096
    k = np.arange(K)
    ac = np.where(k % 2 == 0, 7, -8)[None, :].repeat(M, 0).astype(np.int32)
    ac[::3] = -ac[::3]
    ac = np.clip(ac, -8, 7)
    wc = np.where((k // 3) % 2 == 0, -8, 7)[None, :].repeat(N, 0).astype(np.int32)
    wc[:, ::5] = 0
    rng = np.random.default_rng(0)
    al, ws = rng.uniform(0.1, 1, M), rng.uniform(0.001, 0.01, N)
    y, acc = run(S, ac, al, None, wc, ws)
    assert np.array_equal(acc, oracle_full(ac, al, None, wc, ws).acc)


FULL = [
    ("gate_up", 2048, 4096, 14336, False),
    ("down_proj", 2048, 14336, 4096, True),
    ("l32_up_M8192", 8192, 3072, 8192, False),
    ("l32_down_M8192", 8192, 8192, 3072, False),
    ("l32_up_M1", 1, 3072, 8192, False),
    ("l32_down_M16", 16, 8192, 3072, False),
    ("l32_up_M128", 128, 3072, 8192, False),
    # ragged edges, each prefill kernel forced: M not a multiple of 32, N a
    # multiple of 16 but not of 32 (clipped TMA stores of y)
    ("ragged_M2000_pair", 2000, 3072, 14352, True, 3),
    ("ragged_M2000_tile256", 2000, 3072, 14352, True, 2),
    ("ragged_M2001_asym_pair", 2001, 3072, 12304, False, 3),
    ("ragged_M2001_asym_tile256", 2001, 3072, 12304, False, 2),
    ("ragged_M2001_asym_tile128", 2001, 512, 12288, False, 1),
]

@pytest.mark.parametrize("name,M,K,N,symmetric", [FULL[0], FULL[1]], ids=[FULL[0][0], FULL[1][0]])
def test_gemm_repeat_bit_identical(S, name, M, K, N, symmetric):
    # The accumulator is exact integer arithmetic, so repeated runs must agree
    # bit for bit over the whole matrix; a pipeline race (a shared-memory stage
    # refilled before every reader has read it) shows up as blocks that differ
    # from run to run.  One run is also checked against the oracle on samples.
    rng = np.random.default_rng(17 + len(name))
    ac, al, be, wc, ws = random_codes(rng, M, N, K, symmetric)
    a = to_gpu_act(S, ac, al, be)
    w = to_gpu_w(S, wc, ws)
    _, acc0 = S.w4a4_gemm(a, w, want_acc=True)
    for _ in range(3):
        _, acc = S.w4a4_gemm(a, w, want_acc=True)
        assert torch.equal(acc, acc0)
    ms, ns = rng.integers(0, M, 2000), rng.integers(0, N, 2000)
    racc, _ = oracle.w4a4_linear_sampled(ac, al, be, wc, ws, ms, ns)
    assert np.array_equal(acc0.cpu().numpy()[ms, ns], racc)


@pytest.mark.parametrize("M,N,K", [(2048, 16384, 128), (2048, 16384, 384), (1100, 16400, 640), (4096, 9728, 256)])
def test_gemm_tile256_many_tiles_per_cta(S, M, N, K):
    """256-row tiles, several per CTA, with an odd and an even number of K
    steps per tile (one step included): the unpack group that owns the next
    tile's first step alternates with the parity of the step count and
    unpacks it ahead, during the epilogue of the current tile.  Checked bit
    for bit against 128-row tiles and on sampled outputs against the oracle."""
    rng = np.random.default_rng(M + N + K)
    ac, al, be, wc, ws_ = random_codes(rng, M, N, K, False)
    a = to_gpu_act(S, ac, al, be)
    w = to_gpu_w(S, wc, ws_)
    prev = S.spinq_gemm_select_kernel(S.SPINQ_GEMM_TILE256)
    try:
        y, acc = S.w4a4_gemm(a, w, want_acc=True)
        S.spinq_gemm_select_kernel(S.SPINQ_GEMM_TILE128)
        y1, acc1 = S.w4a4_gemm(a, w, want_acc=True)
    finally:
        S.spinq_gemm_select_kernel(prev)
    torch.cuda.synchronize()
    assert torch.equal(acc, acc1)
    assert torch.equal(y.view(torch.int16), y1.view(torch.int16))
    ms = np.concatenate([rng.integers(0, M, 2000), [0, M - 1, 255, 256]])
    ns = np.concatenate([rng.integers(0, N, 2000), [N - 1, 0, 255, 256]])
    racc, _ = oracle.w4a4_linear_sampled(ac, al, be, wc, ws_, ms, ns)
    assert np.array_equal(acc.cpu().numpy()[ms, ns], racc)
    assert S.spinq_device_status()[0] == S.SPINQ_OK


@pytest.mark.parametrize("case", FULL, ids=[f[0] for f in FULL])
def test_gemm_full_size_sampled(S, case):
    name, M, K, N, symmetric = case[:5]
    kernel = case[5] if len(case) > 5 else 0
    rng = np.random.default_rng(len(name))
    ac, al, be, wc, ws = random_codes(rng, M, N, K, symmetric)
    prev = S.spinq_gemm_select_kernel(kernel)
    try:
        y, acc = run(S, ac, al, be, wc, ws)
    finally:
        S.spinq_gemm_select_kernel(prev)
    # sampled outputs (random + corners + tile edges)
    ms = np.concatenate([rng.integers(0, M, 3000), [0, M - 1, min(127, M - 1), min(128, M - 1)]])
    ns = np.concatenate([rng.integers(0, N, 3000), [N - 1, 0, min(255, N - 1), min(256, N - 1)]])
    al32 = al.astype(np.float32).astype(np.float64)
    be32 = None if be is None else be.astype(np.float32).astype(np.float64)
    ws32 = ws.astype(np.float32).astype(np.float64)
    racc, ry = oracle.w4a4_linear_sampled(ac, al32, be32, wc, ws32, ms, ns)
    assert np.array_equal(acc[ms, ns], racc)
    assert pu.rel_frob(y[ms, ns], ry) <= pu.Y_REL_FROB


LINEAR = [
    ("tiny", synth.tiny_linear, {}),
    ("down_proj_M256", synth.llama3_8b_down_proj, {"M": 256}),
    ("gate_up_M128", synth.llama3_8b_gate_up, {"M": 128}),
    ("l32_up_M16", synth.llama32_3b_up, {"M": 16}),
    ("l32_down_M128", synth.llama32_3b_down, {"M": 128}),
]


@pytest.mark.parametrize("name,builder,kw", LINEAR, ids=[c[0] for c in LINEAR])
def test_rotated_linear_end_to_end(S, name, builder, kw):
    """GPU rotate+quant -> GPU weight quant -> GPU GEMM vs the oracle chain."""
    c = builder(**kw)
    x = torch.from_numpy(c.x).cuda()
    w = torch.from_numpy(c.w).cuda()
    qa = S.rotate_quant_act(x, c.had, c.act_symmetric, c.clip)
    qw = S.quant_weight(w, c.had)
    y = S.w4a4_gemm(qa, qw)
    torch.cuda.synchronize()
    ra = oracle.rotate_quant_act(c.x, c.had, 4, c.act_symmetric, c.clip)
    rw = oracle.quant_weight(c.w, c.had)
    ref = oracle.w4a4_linear(ra, rw)
    assert pu.rel_frob(y.cpu().numpy(), ref.y) <= pu.Y_REL_FROB
    # and with the GPU's own codes, the accumulator is exact
    got_a = pu.gpu_codes(qa.codes.cpu().numpy(), c.act_symmetric)
    got_w = pu.gpu_codes(qw.codes.cpu().numpy(), True)
    y2, acc2 = S.w4a4_gemm(qa, qw, want_acc=True)
    ref2 = oracle.w4a4_linear(
        oracle.QuantAct(got_a, None, qa.scale.cpu().numpy().astype(np.float64),
                        None if qa.zero is None else qa.zero.cpu().numpy().astype(np.float64), None),
        oracle.QuantWeight(got_w, None, qw.scale.cpu().numpy().astype(np.float64), got_w.sum(1), None))
    assert np.array_equal(acc2.cpu().numpy(), ref2.acc)


FULL_CHAIN = [
    ("gate_up", synth.llama3_8b_gate_up, {}),
    ("down_proj", synth.llama3_8b_down_proj, {}),
]


@pytest.mark.parametrize("name,builder,kw", FULL_CHAIN, ids=[c[0] for c in FULL_CHAIN])
def test_rotated_linear_chain_full_size(S, name, builder, kw):
    """The whole chain at the configs' own size (2048 tokens; gate_up
    4096 -> 14336 with no online rotation, down_proj 14336 -> 4096 with R4 =
    H28 (x) H512): GPU rotate+quant of the activations, GPU weight quant, GPU
    GEMM.  On sampled rows and channels: the codes against the oracle's (the
    +-1 tie bar), the accumulator exactly and y (fp16) against the oracle's
    product of the GPU's own codes.  (y against the oracle chain is not a
    usable bar on a sample: with gate_up's coarse asymmetric codes one allowed
    tie flip moves a row of y by ~0.7 %.)"""
    c = builder(**kw)
    x = torch.from_numpy(c.x).cuda()
    w = torch.from_numpy(c.w).cuda()
    qa = S.rotate_quant_act(x, c.had, c.act_symmetric, c.clip)
    qw = S.quant_weight(w, c.had)
    y, acc = S.w4a4_gemm(qa, qw, want_acc=True)
    torch.cuda.synchronize()
    rng = np.random.default_rng(11)
    ms = np.unique(np.concatenate([rng.integers(0, c.M, 24), [0, c.M - 1]]))
    ns = np.unique(np.concatenate([rng.integers(0, c.N, 48), [0, c.N - 1]]))
    ms_t = torch.as_tensor(ms, device="cuda")
    ns_t = torch.as_tensor(ns, device="cuda")
    got_a = pu.gpu_codes(qa.codes[ms_t].cpu().numpy(), c.act_symmetric)
    got_w = pu.gpu_codes(qw.codes[ns_t].cpu().numpy(), True)
    ra = oracle.rotate_quant_act(c.x[ms], c.had, 4, c.act_symmetric, c.clip)
    rw = oracle.quant_weight(c.w[ns], c.had)
    pu.assert_codes_close(got_a, ra.codes, name + " activation codes")
    pu.assert_codes_close(got_w, rw.codes, name + " weight codes")
    ref = oracle.w4a4_linear(
        oracle.QuantAct(got_a, None, qa.scale[ms_t].cpu().numpy().astype(np.float64),
                        None if qa.zero is None else qa.zero[ms_t].cpu().numpy().astype(np.float64), None),
        oracle.QuantWeight(got_w, None, qw.scale[ns_t].cpu().numpy().astype(np.float64), got_w.sum(1), None))
    assert np.array_equal(acc.cpu().numpy()[np.ix_(ms, ns)], ref.acc)
    assert pu.rel_frob(y.cpu().numpy()[np.ix_(ms, ns)], ref.y) <= 2e-3


def test_rotation_reduces_quantization_error(S):
    """Sec. 2 / Fig. 2 and Sec. 3.1 on the device: with R4 the per-token int4
    activation error on outlier-channel inputs drops sharply (Fig. 2(b)), and
    the W4A4 layer output moves closer to the full-precision x W^T (the
    rotation itself leaves x W^T unchanged)."""
    c = synth.llama3_8b_down_proj(M=64)
    x = torch.from_numpy(c.x).cuda()
    w = torch.from_numpy(c.w).cuda()
    xd = c.x.astype(np.float64)
    ref = xd @ c.w.astype(np.float64).T

    def act_err(had):
        qa = S.rotate_quant_act(x, had, True)
        codes = pu.gpu_codes(qa.codes.cpu().numpy(), True)
        deq = codes * qa.scale.cpu().numpy().astype(np.float64)[:, None]
        target = oracle.rotate(xd, *had) if had else xd
        return pu.rel_frob(deq, target)

    # unrotated, the x100 outlier channels hold ~93% of a row's energy and the
    # int4 grid zeroes the rest (error ~ sqrt(0.07) ~ 0.26); after R4 the row is
    # near-Gaussian and int4 RTN leaves ~0.14
    assert act_err(c.had) < 0.7 * act_err(None)
    y = S.w4a4_gemm(S.rotate_quant_act(x, c.had, True), S.quant_weight(w, c.had))
    y0 = S.w4a4_gemm(S.rotate_quant_act(x, None, True), S.quant_weight(w, None))
    assert pu.rel_frob(y.cpu().numpy(), ref) < pu.rel_frob(y0.cpu().numpy(), ref)


# ------------------------------------------------------------------ split-K decode path
def run_splitk(S, ac, al, be, wc, ws_, workspace=None):
    a = to_gpu_act(S, ac, al, be)
    w = to_gpu_w(S, wc, ws_)
    y, acc = S.w4a4_gemm_splitk(a, w, workspace=workspace, want_acc=True)
    torch.cuda.synchronize()
    return y.cpu().numpy(), acc.cpu().numpy()


@pytest.fixture
def splitk_route(S, request):
    """Routes of the split-K entry point: the cost model's choice ("auto"),
    the split-K kernel with the slices the model picks ("sliced"), and the
    split-K kernel with the whole K range per tile ("whole_k")."""
    route = request.param
    prev_kind = S.spinq_gemm_select_kernel(0 if route == "auto" else S.SPINQ_GEMM_SPLITK)
    prev_cap = S.spinq_gemm_split_k(1 if route == "whole_k" else 0)
    assert prev_kind >= 0 and prev_cap >= 0
    yield route
    S.spinq_gemm_select_kernel(prev_kind)
    S.spinq_gemm_split_k(prev_cap)


SPLITK_SHAPES = [(1, 16, 128), (3, 48, 256), (16, 512, 1024), (17, 272, 384), (33, 1024, 512),
                 (64, 256, 128), (100, 384, 640), (128, 3072, 1024), (200, 256, 256),
                 (256, 512, 512), (300, 256, 256)]


@pytest.mark.parametrize("splitk_route", ["auto", "sliced", "whole_k"], indirect=True)
@pytest.mark.parametrize("M,N,K", SPLITK_SHAPES)
@pytest.mark.parametrize("symmetric", [True, False])
def test_splitk_random_codes_exact(S, splitk_route, M, N, K, symmetric):
    rng = np.random.default_rng(M * 13 + N + K + symmetric)
    ac, al, be, wc, ws_ = random_codes(rng, M, N, K, symmetric)
    kind, nsplit = S.spinq_w4a4_gemm_splitk_plan(M, N, K)
    if splitk_route != "auto" and M <= 256:
        assert kind == S.SPINQ_GEMM_SPLITK
        assert nsplit == 1 if splitk_route == "whole_k" else 1 <= nsplit <= min(64, K // 128)
    y, acc = run_splitk(S, ac, al, be, wc, ws_)
    ref = oracle_full(ac, al, be, wc, ws_)
    assert np.array_equal(acc, ref.acc)
    assert pu.rel_frob(y, ref.y) <= pu.Y_REL_FROB
    assert np.allclose(y.astype(np.float64), ref.y, rtol=2e-3, atol=1e-3 * np.abs(ref.y).max())


def test_splitk_plan_covers_every_route(S):
    """Under the default selection the split-K entry point's shapes above,
    with the decode configurations, reach the GEMV kernel, the split-K kernel
    with and without K slices, and the prefill kernels."""
    shapes = SPLITK_SHAPES + [(1, 8192, 3072), (16, 8192, 3072), (64, 8192, 3072), (128, 8192, 3072),
                              (128, 3072, 8192), (256, 8192, 3072)]
    routes = set()
    for M, N, K in shapes:
        kind, nsplit = S.spinq_w4a4_gemm_splitk_plan(M, N, K)
        assert kind in (1, 2, 3, 4, 5, 6)
        assert (nsplit >= 1) == (kind == S.SPINQ_GEMM_SPLITK)
        routes.add("sliced" if nsplit > 1 else "whole_k" if nsplit == 1 else kind)
        # the workspace exists exactly for K slices
        assert (S.spinq_w4a4_gemm_workspace_bytes(M, N, K) > 0) == (nsplit > 1)
    assert {"sliced", "whole_k", 4}.issubset(routes)
    assert routes & {1, 2, 3}
    assert S.spinq_w4a4_gemm_splitk_plan(16, 100, 1024)[0] == -1    # N not a multiple of 16
    assert S.spinq_w4a4_gemm_splitk_plan(16, 128, 1000)[0] == -1    # K not a multiple of 128


def test_splitk_workspace_follows_the_plan(S):
    for M, kind in ((1, S.SPINQ_GEMM_GEMV), (2, S.SPINQ_GEMM_GEMV), (3, S.SPINQ_GEMM_TCGEMV), (16, S.SPINQ_GEMM_TCGEMV)):
        assert S.spinq_w4a4_gemm_workspace_bytes(M, 8192, 3072) == 0
        assert S.gemm_workspace(M, 8192, 3072) is None
        assert S.spinq_w4a4_gemm_splitk_plan(M, 8192, 3072) == (kind, 0)
    # a few dozen tokens, narrow outputs, long K: every SM streams a slice of the weights
    kind, nsplit = S.spinq_w4a4_gemm_splitk_plan(32, 3072, 8192)
    assert kind == S.SPINQ_GEMM_SPLITK and nsplit > 1
    assert S.spinq_w4a4_gemm_workspace_bytes(32, 3072, 8192) == 32 * 3072 * 4 + 24 * 4
    # the tokens no longer fit in the GEMV kernel's shared memory
    assert S.spinq_w4a4_gemm_splitk_plan(4, 8192, 65536)[0] == S.SPINQ_GEMM_SPLITK
    # no slices, no workspace
    prev = S.spinq_gemm_split_k(1)
    try:
        assert S.spinq_w4a4_gemm_workspace_bytes(32, 3072, 8192) == 0
        assert S.spinq_w4a4_gemm_splitk_plan(32, 3072, 8192) == (S.SPINQ_GEMM_SPLITK, 1)
    finally:
        S.spinq_gemm_split_k(prev)
    assert S.spinq_gemm_split_k(65) == -1 and S.spinq_gemm_split_k(-1) == -1
    # a fixed count, at most one slice per 128-deep K step
    prev = S.spinq_gemm_split_k(7)
    prev_kind = S.spinq_gemm_select_kernel(S.SPINQ_GEMM_SPLITK)
    try:
        assert S.spinq_w4a4_gemm_splitk_plan(16, 3072, 8192) == (S.SPINQ_GEMM_SPLITK, 7)
        assert S.spinq_w4a4_gemm_splitk_plan(16, 3072, 512) == (S.SPINQ_GEMM_SPLITK, 4)
        assert S.spinq_w4a4_gemm_splitk_plan(2, 3072, 512) == (S.SPINQ_GEMM_SPLITK, 4)
    finally:
        S.spinq_gemm_split_k(prev)
        S.spinq_gemm_select_kernel(prev_kind)


@pytest.mark.parametrize("M,N,K", [(1, 16, 128), (2, 48, 256), (3, 272, 384), (4, 512, 1024), (1, 1040, 4096),
                                   (4, 8192, 8192), (3, 100 * 16, 14336), (1, 8192, 40960)])
@pytest.mark.parametrize("symmetric", [True, False])
def test_gemv_random_codes_exact(S, M, N, K, symmetric):
    """The GEMV kernel (M <= 4, selected: AUTO gives 3 and 4 tokens to the
    tensor-core GEMV where it covers K) through both entry points."""
    rng = np.random.default_rng(M * 31 + N + K + symmetric)
    ac, al, be, wc, ws_ = random_codes(rng, M, N, K, symmetric)
    ref = oracle_full(ac, al, be, wc, ws_)

    def go():
        assert S.spinq_w4a4_gemm_plan(M, N, K) == S.SPINQ_GEMM_GEMV
        return [run_splitk(S, ac, al, be, wc, ws_), run(S, ac, al, be, wc, ws_)]
    for entry, (y, acc) in zip(("splitk", "gemm"), _with_kernel(S, S.SPINQ_GEMM_GEMV, go)):
        assert np.array_equal(acc, ref.acc), entry
        assert pu.rel_frob(y, ref.y) <= pu.Y_REL_FROB
        assert np.allclose(y.astype(np.float64), ref.y, rtol=2e-3, atol=1e-3 * np.abs(ref.y).max())


def test_gemv_shared_memory_sizes_in_any_order(S):
    """One kernel launched with a large, a smaller and again the large shared
    memory size (the per-kernel limit must not shrink)."""
    rng = np.random.default_rng(5)
    for (M, N, K) in [(4, 256, 32768), (3, 256, 14336), (4, 256, 32768), (2, 256, 1024), (4, 256, 32768)]:
        ac, al, be, wc, ws_ = random_codes(rng, M, N, K, False)
        y, acc = _with_kernel(S, S.SPINQ_GEMM_GEMV, lambda: run_splitk(S, ac, al, be, wc, ws_))
        assert np.array_equal(acc, oracle_full(ac, al, be, wc, ws_).acc)


def test_gemv_extreme_codes_long_k(S):
    M, N, K = 3, 64, 65536 // 8   # M * K within the kernel's shared memory
    for aval, wval in ((7, 7), (-8, -8), (7, -8)):
        ac = np.full((M, K), aval, dtype=np.int32)
        wc = np.full((N, K), wval, dtype=np.int32)
        al, ws_ = np.full(M, 0.5), np.full(N, 0.25)
        y, acc = _with_kernel(S, S.SPINQ_GEMM_GEMV, lambda: run_splitk(S, ac, al, None, wc, ws_))
        assert np.array_equal(acc, oracle_full(ac, al, None, wc, ws_).acc)


def _with_kernel(S, kind, fn):
    prev = S.spinq_gemm_select_kernel(kind)
    try:
        return fn()
    finally:
        S.spinq_gemm_select_kernel(prev)


@pytest.mark.parametrize("M,N,K", [(1, 16, 128), (5, 48, 256), (8, 272, 1152), (9, 512, 1024), (16, 3072, 8192),
                                   (13, 1040, 4224), (16, 4096, 14336), (3, 8192, 3072), (12, 16, 40960)])
@pytest.mark.parametrize("symmetric", [True, False])
def test_tcgemv_random_codes_exact(S, M, N, K, symmetric):
    """The tensor-core GEMV (M <= 16) through both entry points: exact acc,
    y within the GEMM bars; K block counts that leave the 8 warps' last
    rounds partly empty."""
    rng = np.random.default_rng(M * 131 + N + K + symmetric)
    ac, al, be, wc, ws_ = random_codes(rng, M, N, K, symmetric)
    ref = oracle_full(ac, al, be, wc, ws_)

    def go():
        assert S.spinq_w4a4_gemm_plan(M, N, K) == S.SPINQ_GEMM_TCGEMV
        assert S.spinq_w4a4_gemm_splitk_plan(M, N, K) == (S.SPINQ_GEMM_TCGEMV, 0)
        assert S.spinq_w4a4_gemm_workspace_bytes(M, N, K) == 0
        return [run_splitk(S, ac, al, be, wc, ws_), run(S, ac, al, be, wc, ws_)]
    for y, acc in _with_kernel(S, S.SPINQ_GEMM_TCGEMV, go):
        assert np.array_equal(acc, ref.acc)
        assert pu.rel_frob(y, ref.y) <= pu.Y_REL_FROB
        assert np.allclose(y.astype(np.float64), ref.y, rtol=2e-3, atol=1e-3 * np.abs(ref.y).max())


@pytest.mark.parametrize("M", [3, 11, 16])
def test_tcgemv_same_bits_as_the_other_decode_kernels(S, M):
    """y and acc bit for bit against the kernel the cost model picks."""
    rng = np.random.default_rng(M)
    N, K = 1296, 3072
    ac, al, be, wc, ws_ = random_codes(rng, M, N, K, False)
    y0, acc0 = run_splitk(S, ac, al, be, wc, ws_)
    y1, acc1 = _with_kernel(S, S.SPINQ_GEMM_TCGEMV, lambda: run_splitk(S, ac, al, be, wc, ws_))
    assert np.array_equal(acc0, acc1)
    assert np.array_equal(y0.view(np.uint16), y1.view(np.uint16))


@pytest.mark.parametrize("symmetric", [True, False])
def test_tcgemv_extreme_codes_long_k(S, symmetric):
    """K = 65536 with every code at an extreme: the e4m3 accumulator reaches
    225 K 2^-18 (just below 2^6) and must stay exact."""
    M, N, K = 16, 32, 65536
    pairs = ((7, 7), (-8, -8), (7, -8)) if symmetric else ((15, 7), (0, -8), (15, -8))
    for aval, wval in pairs:
        ac = np.full((M, K), aval, dtype=np.int32)
        wc = np.full((N, K), wval, dtype=np.int32)
        al, ws_ = np.full(M, 0.5), np.full(N, 0.25)
        be = None if symmetric else np.full(M, -1.0)
        y, acc = _with_kernel(S, S.SPINQ_GEMM_TCGEMV, lambda: run_splitk(S, ac, al, be, wc, ws_))
        assert np.array_equal(acc, oracle_full(ac, al, be, wc, ws_).acc), (aval, wval)


@pytest.mark.parametrize("symmetric", [True, False])
def test_tcgemv_register_streamed_extreme_codes(S, symmetric):
    """The register-streamed form at its longest K (16 warps of 8 K blocks):
    every code at an extreme, 2^-44 units up to 225 K."""
    M, N, K = 16, 4096, 16384
    pairs = ((7, 7), (-8, -8), (7, -8)) if symmetric else ((15, 7), (0, -8), (15, -8))
    for aval, wval in pairs:
        ac = np.full((M, K), aval, dtype=np.int32)
        wc = np.full((N, K), wval, dtype=np.int32)
        al, ws_ = np.full(M, 0.5), np.full(N, 0.25)
        be = None if symmetric else np.full(M, -1.0)
        y, acc = _with_kernel(S, S.SPINQ_GEMM_TCGEMV, lambda: run_splitk(S, ac, al, be, wc, ws_))
        assert np.array_equal(acc, oracle_full(ac, al, be, wc, ws_).acc), (aval, wval)


@pytest.mark.parametrize("M,N,K", [(2, 8192, 3072), (16, 3072, 8192), (7, 14336, 4096), (16, 4096, 14336),
                                   (1, 1216, 2048), (4, 64, 1536), (16, 14592, 1024), (11, 20480, 384)])
def test_tcgemv_register_streamed_shapes(S, M, N, K):
    """The decode shapes of both configs, K block counts of 1, 2, 4 and 8 per
    warp, and 6 to 9 tiles per CTA (every reduction slot reused): exact acc
    against the oracle on random codes."""
    rng = np.random.default_rng(M * 7 + N + K)
    ac, al, be, wc, ws_ = random_codes(rng, M, N, K, M % 2 == 0)
    ref = oracle_full(ac, al, be, wc, ws_)
    y, acc = _with_kernel(S, S.SPINQ_GEMM_TCGEMV, lambda: run_splitk(S, ac, al, be, wc, ws_))
    assert np.array_equal(acc, ref.acc)
    assert pu.rel_frob(y, ref.y) <= pu.Y_REL_FROB


def test_auto_plan_takes_tcgemv_for_three_to_sixteen_tokens(S):
    """Automatic choice: the GEMV kernel up to 2 tokens, the tensor-core GEMV
    from 3 to 16 where its register-streamed form covers K (3072 = 24 K
    blocks), else from 5 to 8 (4224 = 33 K blocks); split-K beyond."""
    for M, want in ((1, S.SPINQ_GEMM_GEMV), (2, S.SPINQ_GEMM_GEMV), (3, S.SPINQ_GEMM_TCGEMV),
                    (8, S.SPINQ_GEMM_TCGEMV), (16, S.SPINQ_GEMM_TCGEMV)):
        assert S.spinq_w4a4_gemm_plan(M, 8192, 3072) == want
        assert S.spinq_w4a4_gemm_splitk_plan(M, 8192, 3072) == (want, 0)
    assert S.spinq_w4a4_gemm_splitk_plan(17, 8192, 3072)[0] == S.SPINQ_GEMM_SPLITK
    for M, want in ((4, S.SPINQ_GEMM_GEMV), (5, S.SPINQ_GEMM_TCGEMV), (8, S.SPINQ_GEMM_TCGEMV)):
        assert S.spinq_w4a4_gemm_plan(M, 8192, 4224) == want
    assert S.spinq_w4a4_gemm_splitk_plan(9, 8192, 4224)[0] == S.SPINQ_GEMM_SPLITK
    # a forced split-K selection keeps the split-K kernel
    prev = S.spinq_gemm_select_kernel(S.SPINQ_GEMM_SPLITK)
    try:
        assert S.spinq_w4a4_gemm_splitk_plan(6, 8192, 3072)[0] == S.SPINQ_GEMM_SPLITK
    finally:
        S.spinq_gemm_select_kernel(prev)


def test_tcgemv_plan_falls_back_beyond_its_range(S):
    def go():
        assert S.spinq_w4a4_gemm_plan(17, 4096, 4096) != S.SPINQ_GEMM_TCGEMV
        assert S.spinq_w4a4_gemm_splitk_plan(17, 4096, 4096)[0] != S.SPINQ_GEMM_TCGEMV
        assert S.spinq_w4a4_gemm_plan(16, 4096, 4096) == S.SPINQ_GEMM_TCGEMV
    _with_kernel(S, S.SPINQ_GEMM_TCGEMV, go)


def test_splitk_workspace_reused_and_left_zero(S):
    """The split-K kernel (selected: AUTO gives 16 tokens to the tensor-core
    GEMV) slices K here; its workspace is reused and left zero."""
    rng = np.random.default_rng(21)
    M, N, K = 16, 1024, 2048

    def go():
        ws = S.gemm_workspace(M, N, K)
        assert ws is not None   # the plan slices K here
        for rep in range(3):
            ac, al, be, wc, ws_ = random_codes(rng, M, N, K, rep % 2 == 0)
            y, acc = run_splitk(S, ac, al, be, wc, ws_, workspace=ws)
            assert np.array_equal(acc, oracle_full(ac, al, be, wc, ws_).acc)
            assert int(torch.count_nonzero(ws)) == 0
    _with_kernel(S, S.SPINQ_GEMM_SPLITK, go)


@pytest.mark.parametrize("splitk_route", ["sliced", "whole_k"], indirect=True)
@pytest.mark.parametrize("M", [16, 256])
def test_splitk_extreme_codes_long_k(S, splitk_route, M):
    """|acc| up to 64 K = 2^22 stays exact through the fp32 accumulator, the
    slices' partial sums and the unsliced epilogue."""
    N, K = 256, 65536
    for aval, wval in ((7, 7), (-8, -8), (7, -8)):
        ac = np.full((M, K), aval, dtype=np.int32)
        wc = np.full((N, K), wval, dtype=np.int32)
        al, ws_ = np.full(M, 0.5), np.full(N, 0.25)
        y, acc = run_splitk(S, ac, al, None, wc, ws_)
        # constant codes: every output's sum is K a w
        assert np.array_equal(acc, np.full((M, N), K * aval * wval, dtype=np.int32))
        if M <= 16:
            assert np.array_equal(acc, oracle_full(ac, al, None, wc, ws_).acc)


@pytest.mark.parametrize("name,M,K,N,symmetric", [("l32_up_M1", 1, 3072, 8192, False),
                                                  ("l32_up_M16", 16, 3072, 8192, False),
                                                  ("l32_up_M64", 64, 3072, 8192, False),
                                                  ("l32_down_M128", 128, 8192, 3072, False),
                                                  ("l32_down_M256", 256, 8192, 3072, False)])
def test_splitk_decode_configs_full(S, name, M, K, N, symmetric):
    rng = np.random.default_rng(len(name) + M)
    ac, al, be, wc, ws_ = random_codes(rng, M, N, K, symmetric)
    y, acc = run_splitk(S, ac, al, be, wc, ws_)
    ref = oracle_full(ac, al, be, wc, ws_)
    assert np.array_equal(acc, ref.acc)
    assert pu.rel_frob(y, ref.y) <= pu.Y_REL_FROB
