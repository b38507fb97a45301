"""The no-allocation GEMM entry point (spinq_w4a4_gemm_noalloc).

It serves callers that cannot allocate device memory where they run the
layer: its split-K workspace is a fixed array inside the library instead of a
buffer the caller passes in.  This file checks, through the C ABI, that two
calls in a row give the same result as spinq_w4a4_gemm on the same inputs
(integer accumulator exact, fp16 output within the tests' tolerance), also
for a request whose K slices would not fit the fixed array.  It runs last and does
not depend on any other test.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _inputs(gen, M, N, K, symmetric):
    dev = "cuda"
    a_codes = torch.randint(0, 256, (M, K // 2), dtype=torch.uint8, device=dev, generator=gen)
    w_codes = torch.randint(0, 256, (N, K // 2), dtype=torch.uint8, device=dev, generator=gen)
    a_scale = torch.rand(M, device=dev, generator=gen) * 0.9 + 0.1
    a_zero = None if symmetric else -torch.rand(M, device=dev, generator=gen) * 3.0
    w_scale = torch.rand(N, device=dev, generator=gen) * 0.009 + 0.001
    # row sums of the signed weight codes (two's complement nibbles)
    nib = torch.stack([w_codes & 15, w_codes >> 4], dim=-1).reshape(N, K).to(torch.int32)
    w_rowsum = torch.where(nib >= 8, nib - 16, nib).sum(dim=1).to(torch.int32)
    return a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _call(fn, args, M, N, K):
    a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum = args
    y = torch.empty((M, N), dtype=torch.float16, device="cuda")
    acc = torch.empty((M, N), dtype=torch.int32, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = fn(_ptr(a_codes), _ptr(a_scale), _ptr(a_zero), _ptr(w_codes), _ptr(w_scale), _ptr(w_rowsum),
            M, N, K, _ptr(y), _ptr(acc), stream)
    return st, y, acc


def test_noalloc_matches_gemm_on_two_calls_in_a_row():
    from paper_2405_16406_gb300 import spinq as S
    gen = torch.Generator(device="cuda")
    gen.manual_seed(2024)
    for M, N, K, symmetric in ((16, 3072, 1024, False), (100, 2048, 512, True)):
        args = _inputs(gen, M, N, K, symmetric)
        st_ref, y_ref, acc_ref = _call(S.spinq_w4a4_gemm, args, M, N, K)
        st, y, acc = _call(S.spinq_w4a4_gemm_noalloc, args, M, N, K)
        torch.cuda.synchronize()
        assert st_ref == S.SPINQ_OK and st == S.SPINQ_OK
        assert torch.equal(acc, acc_ref)
        yr = y_ref.double().cpu().numpy()
        yn = y.double().cpu().numpy()
        assert np.linalg.norm(yn - yr) / np.linalg.norm(yr) <= 1e-2
        assert np.allclose(yn, yr, rtol=2e-3, atol=1e-3 * np.abs(yr).max())
    assert S.spinq_device_status()[0] == S.SPINQ_OK


def test_noalloc_serves_requests_beyond_its_scratch_unsliced():
    """A call whose K slices would need more partial sums than the 8 MiB
    scratch holds keeps the whole K range per tile and matches
    spinq_w4a4_gemm (the split-K kernel and two K slices are forced, so that
    the plan needs the workspace for this shape)."""
    from paper_2405_16406_gb300 import spinq as S
    gen = torch.Generator(device="cuda")
    gen.manual_seed(1)
    M, N, K = 256, 9728, 8192          # partial sums of 9.5 MiB
    args = _inputs(gen, M, N, K, True)
    st_ref, y_ref, acc_ref = _call(S.spinq_w4a4_gemm, args, M, N, K)
    prev = S.spinq_gemm_select_kernel(S.SPINQ_GEMM_SPLITK)
    prev_split = S.spinq_gemm_split_k(2)
    try:
        assert S.spinq_w4a4_gemm_workspace_bytes(M, N, K) > 8 << 20
        st, y, acc = _call(S.spinq_w4a4_gemm_noalloc, args, M, N, K)
    finally:
        S.spinq_gemm_select_kernel(prev)
        S.spinq_gemm_split_k(prev_split)
    torch.cuda.synchronize()
    assert st_ref == S.SPINQ_OK and st == S.SPINQ_OK
    assert torch.equal(acc, acc_ref)
    assert (y.float() - y_ref.float()).norm() <= 1e-2 * y_ref.float().norm()
    assert S.spinq_device_status()[0] == S.SPINQ_OK
