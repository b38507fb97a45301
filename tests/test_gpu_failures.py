"""Failure paths on the GPU, without a fault: bounded waits that give up and
a refused launch.

The next launch of the kernel under test issues no input copies
(spinq_debug_stall_launches), so its consumers wait on barriers that nothing
completes, and the wait limit is lowered to 1 ms: the waits run out of time,
the kernel records SPINQ_ETIMEOUT, every role leaves its loop, MMAs in flight
are drained (with the full limit) and tensor memory is released.  The test checks the status, restores the
controls and checks that the same call is correct again (the context stays
usable).  A launch refused on the host (a fake of a failing
launch) returns SPINQ_ECUDA and enqueues nothing."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_16406_gb300 import synth
from parity_util import assert_codes_close, gpu_codes, rel_frob

pytestmark = pytest.mark.gpu

DEFAULT_NS = 2_000_000_000


def _cases():
    """name -> (call, check of its output against the oracle)."""
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(0)
    x = synth.activations(rng, 256, 14336, outlier_frac=0.005, factor=100.0, swiglu=True)
    xt = torch.from_numpy(x).cuda()
    a_codes = torch.randint(0, 256, (256, 512), dtype=torch.uint8, device="cuda")
    w_codes = torch.randint(0, 256, (512, 512), dtype=torch.uint8, device="cuda")
    qa = spinq.ActCodes(a_codes, torch.ones(256, device="cuda"), None)
    ai = oracle.unpack4(a_codes.cpu().numpy(), True).astype(np.int64)
    wi = oracle.unpack4(w_codes.cpu().numpy(), True).astype(np.int64)
    qw = spinq.WeightCodes(w_codes, torch.full((512,), 0.01, device="cuda"),
                           torch.from_numpy(wi.sum(1).astype(np.int32)).cuda())
    f8a = torch.randint(0, 0x70, (256, 1024), dtype=torch.uint8, device="cuda")   # finite E4M3 codes
    f8w = torch.randint(0, 0x70, (512, 1024), dtype=torch.uint8, device="cuda")
    f8qa = spinq.ActCodes(f8a, torch.ones(256, device="cuda"), None)
    f8qw = spinq.WeightCodes(f8w, torch.full((512,), 0.01, device="cuda"), torch.zeros(512, dtype=torch.int32,
                                                                                          device="cuda"))

    def gemm(kernel):
        prev = spinq.spinq_gemm_select_kernel(kernel)
        try:
            return spinq.w4a4_gemm(qa, qw, want_acc=True)
        finally:
            spinq.spinq_gemm_select_kernel(prev)

    def check_paley(out):
        ref = oracle.rotate_quant_act(x, (28, 512), 4, True, 1.0)
        assert_codes_close(gpu_codes(out.codes.cpu().numpy(), True), ref.codes, "after the time-out")

    def check_gemm(out):   # |acc| <= 64 K < 2^53: exact in double
        assert np.array_equal(out[1].cpu().numpy(), (ai.astype(np.float64) @ wi.T.astype(np.float64)).astype(np.int64))

    def check_fp8(out):
        ref = oracle.fp8_linear(f8a.cpu().numpy(), np.ones(256), f8w.cpu().numpy(), np.full(512, 0.01))
        assert rel_frob(out.double().cpu().numpy(), ref) <= 1e-3

    return {
        "paley": (lambda: spinq.rotate_quant_act(xt, (28, 512)), check_paley),
        "gemm128": (lambda: gemm(spinq.SPINQ_GEMM_TILE128), check_gemm),
        "gemm256": (lambda: gemm(spinq.SPINQ_GEMM_TILE256), check_gemm),
        "fp8": (lambda: spinq.fp8_gemm(f8qa, f8qw), check_fp8),
    }


@pytest.mark.parametrize("which", ["paley", "gemm128", "gemm256", "fp8"])
def test_bounded_waits_give_up_and_report_timeout(which):
    from paper_2405_16406_gb300 import spinq
    call, check = _cases()[which]
    torch.cuda.synchronize()
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK
    try:
        assert spinq.spinq_debug_set_wait_limit_ns(1_000_000) == spinq.SPINQ_OK
        assert spinq.spinq_debug_stall_launches(1) == 0
        call()
        torch.cuda.synchronize()
        st, site = spinq.spinq_device_status()
        assert spinq.spinq_debug_stall_launches(0) == 0     # the stalled launch happened
    finally:
        spinq.spinq_debug_stall_launches(0)
        assert spinq.spinq_debug_set_wait_limit_ns(DEFAULT_NS) == spinq.SPINQ_OK
    assert st == spinq.SPINQ_ETIMEOUT and site > 0, (st, site)
    # the context is usable and the results are right again
    out = call()
    torch.cuda.synchronize()
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK
    check(out)


def test_refused_launch_returns_ecuda_and_enqueues_nothing():
    from paper_2405_16406_gb300 import spinq
    rng = np.random.default_rng(1)
    x = torch.from_numpy(synth.activations(rng, 64, 4096, outlier_frac=0.01, factor=30.0)).cuda()
    out = spinq.ActCodes(torch.full((64, 2048), 0xAB, dtype=torch.uint8, device="cuda"),
                         torch.full((64,), -1.0, device="cuda"), torch.full((64,), -1.0, device="cuda"))
    assert spinq.spinq_debug_fail_launches(1) == 0
    with pytest.raises(spinq.SpinqError) as e:
        spinq.rotate_quant_act(x, None, False, out=out)
    assert e.value.status == spinq.SPINQ_ECUDA
    torch.cuda.synchronize()
    assert bool((out.codes == 0xAB).all()) and bool((out.scale == -1.0).all())   # nothing ran
    assert spinq.spinq_debug_fail_launches(0) == 0                                 # the one refusal was used
    spinq.rotate_quant_act(x, None, False, out=out)
    torch.cuda.synchronize()
    ref = oracle.rotate_quant_act(x.cpu().numpy(), None, 4, False, 1.0)
    assert_codes_close(gpu_codes(out.codes.cpu().numpy(), False), ref.codes, "after the refusal")
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK
