"""The no-allocation GEMM entry point (spinq_w4a4_gemm_noalloc).

It serves callers that cannot allocate device memory where they run the
layer (a serving runtime with a memory plan fixed at start-up, a thread that
may not call an allocator while streams are being captured, an embedder with
no allocator): its split-K workspace is a fixed array inside the library
instead of a buffer the caller passes in.

These tests force the split-K kernel with several K slices, so that the
partial sums and tile counters really live in that array, and check through
the C ABI that two calls in a row, then a call of another shape, give the
oracle's exact integer accumulator and its fp16 output within the parity
tolerance, and the same result as spinq_w4a4_gemm.  A request whose
partial sums would not fit the array is refused before anything is
enqueued.  The file runs last and depends on no other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from parity_util import Y_REL_FROB, rel_frob

pytestmark = pytest.mark.gpu


def _inputs(gen, M, N, K, symmetric):
    dev = "cuda"
    a_codes = torch.randint(0, 256, (M, K // 2), dtype=torch.uint8, device=dev, generator=gen)
    w_codes = torch.randint(0, 256, (N, K // 2), dtype=torch.uint8, device=dev, generator=gen)
    a_scale = torch.rand(M, device=dev, generator=gen) * 0.9 + 0.1
    a_zero = None if symmetric else -torch.rand(M, device=dev, generator=gen) * 3.0
    w_scale = torch.rand(N, device=dev, generator=gen) * 0.009 + 0.001
    w_int = oracle.unpack4(w_codes.cpu().numpy(), True)
    w_rowsum = torch.from_numpy(w_int.sum(axis=1).astype(np.int32)).cuda()
    return a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum


def _oracle(args, symmetric):
    a_codes, a_scale, a_zero, w_codes, w_scale, _ = args
    ac = oracle.unpack4(a_codes.cpu().numpy(), symmetric)
    wc = oracle.unpack4(w_codes.cpu().numpy(), True)
    qa = oracle.QuantAct(ac, None, a_scale.double().cpu().numpy(),
                         None if a_zero is None else a_zero.double().cpu().numpy(), None)
    qw = oracle.QuantWeight(wc, None, w_scale.double().cpu().numpy(), wc.sum(axis=1), None)
    return oracle.w4a4_linear(qa, qw)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _call(fn, args, M, N, K, y=None):
    a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum = args
    if y is None:
        y = torch.empty((M, N), dtype=torch.float16, device="cuda")
    acc = torch.empty((M, N), dtype=torch.int32, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = fn(_ptr(a_codes), _ptr(a_scale), _ptr(a_zero), _ptr(w_codes), _ptr(w_scale), _ptr(w_rowsum),
            M, N, K, _ptr(y), _ptr(acc), stream)
    return st, y, acc


def _check(S, st, y, acc, ref, y_gemm, acc_gemm):
    assert st == S.SPINQ_OK, S.spinq_status_string(st)
    assert np.array_equal(acc.cpu().numpy(), ref.acc)
    assert torch.equal(acc, acc_gemm)
    yn = y.double().cpu().numpy()
    assert rel_frob(yn, ref.y) <= Y_REL_FROB
    assert np.allclose(yn, ref.y, rtol=2e-3, atol=1e-3 * np.abs(ref.y).max())
    # the split-K and prefill epilogues round in a different order: y agrees
    # with spinq_w4a4_gemm within the same tolerance, not bit for bit
    yg = y_gemm.double().cpu().numpy()
    assert np.allclose(yn, yg, rtol=2e-3, atol=1e-3 * np.abs(yg).max())


def test_noalloc_splits_k_in_its_array_and_matches_oracle():
    """Split-K forced with 4 slices: the partial sums go through the fixed
    array.  Two calls in a row on one shape (the second starts from what the
    first left in the array), then a call of another shape."""
    from paper_2405_16406_gb300 import spinq as S
    gen = torch.Generator(device="cuda")
    gen.manual_seed(2024)
    prev = S.spinq_gemm_select_kernel(S.SPINQ_GEMM_SPLITK)
    prev_split = S.spinq_gemm_split_k(4)
    try:
        for M, N, K, symmetric, repeats in ((16, 4096, 4096, False, 2), (40, 3072, 8192, True, 1)):
            kind, nsplit = S.spinq_w4a4_gemm_splitk_plan(M, N, K)
            need = S.spinq_w4a4_gemm_workspace_bytes(M, N, K)
            assert kind == S.SPINQ_GEMM_SPLITK and nsplit == 4
            assert 0 < need <= S.SPINQ_NOALLOC_SCRATCH_BYTES
            args = _inputs(gen, M, N, K, symmetric)
            ref = _oracle(args, symmetric)
            st_g, y_g, acc_g = _call(S.spinq_w4a4_gemm, args, M, N, K)
            assert st_g == S.SPINQ_OK
            for _ in range(repeats):
                st, y, acc = _call(S.spinq_w4a4_gemm_noalloc, args, M, N, K)
                torch.cuda.synchronize()
                _check(S, st, y, acc, ref, y_g, acc_g)
    finally:
        S.spinq_gemm_select_kernel(prev)
        S.spinq_gemm_split_k(prev_split)
    assert S.spinq_device_status()[0] == S.SPINQ_OK


def test_noalloc_default_plan_matches_oracle():
    """The planner's own choice (no forced kernel) at a decode shape."""
    from paper_2405_16406_gb300 import spinq as S
    gen = torch.Generator(device="cuda")
    gen.manual_seed(7)
    M, N, K = 16, 3072, 8192
    args = _inputs(gen, M, N, K, False)
    ref = _oracle(args, False)
    st_g, y_g, acc_g = _call(S.spinq_w4a4_gemm, args, M, N, K)
    st, y, acc = _call(S.spinq_w4a4_gemm_noalloc, args, M, N, K)
    torch.cuda.synchronize()
    assert st_g == S.SPINQ_OK
    _check(S, st, y, acc, ref, y_g, acc_g)
    assert S.spinq_device_status()[0] == S.SPINQ_OK


def test_noalloc_refuses_requests_beyond_its_array():
    """A plan whose partial sums exceed the fixed array is refused with
    SPINQ_ESCRATCH and nothing is written."""
    from paper_2405_16406_gb300 import spinq as S
    gen = torch.Generator(device="cuda")
    gen.manual_seed(1)
    M, N, K = 256, 9728, 8192          # partial sums of 9.5 MiB
    args = _inputs(gen, M, N, K, True)
    prev = S.spinq_gemm_select_kernel(S.SPINQ_GEMM_SPLITK)
    prev_split = S.spinq_gemm_split_k(2)
    try:
        assert S.spinq_w4a4_gemm_workspace_bytes(M, N, K) > S.SPINQ_NOALLOC_SCRATCH_BYTES
        y = torch.full((M, N), 3.0, dtype=torch.float16, device="cuda")
        st, y, _ = _call(S.spinq_w4a4_gemm_noalloc, args, M, N, K, y=y)
    finally:
        S.spinq_gemm_select_kernel(prev)
        S.spinq_gemm_split_k(prev_split)
    torch.cuda.synchronize()
    assert st == S.SPINQ_ESCRATCH
    assert bool((y == 3.0).all())
    assert S.spinq_device_status()[0] == S.SPINQ_OK
