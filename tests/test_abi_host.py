"""Host-side checks of the C ABI that need no GPU: the library builds and
loads, exports every entry point include/spinq.h declares, and rejects
invalid arguments before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2405_16406_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def declared_entry_points():
    names = []
    for fn in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names += re.findall(r"\b(spinq_[a-z0-9_]+)\s*\(", src)
    return sorted(set(names))


def test_header_declares_the_four_hot_path_calls():
    names = declared_entry_points()
    for n in ("spinq_rotate_quant_act", "spinq_quant_weight", "spinq_w4a4_gemm", "spinq_rotate_quant_kv"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for n in declared_entry_points():
        assert hasattr(lib, n), f"libspinq.so does not export {n}"


def test_binding_names_match_header(lib):
    from paper_2405_16406_gb300 import spinq
    for n in declared_entry_points():
        assert n in spinq.EXPORTED and hasattr(spinq, n)


def test_status_strings(lib):
    from paper_2405_16406_gb300 import spinq
    for s in range(6):
        assert spinq.spinq_status_string(s).startswith("SPINQ_")
    assert "sm_103a" in spinq.spinq_version()


def test_invalid_arguments_rejected_before_launch(lib):
    from paper_2405_16406_gb300 import spinq as S
    q = S.quant_cfg(4, True, S.SPINQ_PER_TOKEN, 0, 1.0)
    fake = ctypes.c_void_p(1 << 20)   # never dereferenced: validation fails first
    # NULL input
    assert S.spinq_rotate_quant_act(None, 4, 256, 256, None, ctypes.byref(q), fake, fake, None, None) == S.SPINQ_EINVAL
    # K not a multiple of 32
    assert S.spinq_rotate_quant_act(fake, 4, 250, 256, None, ctypes.byref(q), fake, fake, None, None) == S.SPINQ_EINVAL
    # misaligned pointer
    assert S.spinq_rotate_quant_act(ctypes.c_void_p((1 << 20) + 2), 4, 256, 256, None, ctypes.byref(q), fake, fake,
                                    None, None) == S.SPINQ_EINVAL
    # Hadamard spec inconsistent with K
    had = S.HadCfg(1, 128)
    assert S.spinq_rotate_quant_act(fake, 4, 256, 256, ctypes.byref(had), ctypes.byref(q), fake, fake, None,
                                    None) == S.SPINQ_EINVAL
    # unsupported small Hadamard order (valid size, no kernel)
    had = S.HadCfg(36, 64)
    assert S.spinq_rotate_quant_act(fake, 4, 36 * 64, 36 * 64, ctypes.byref(had), ctypes.byref(q), fake, fake,
                                    None, None) == S.SPINQ_EUNSUPPORTED
    # clip outside (0, 1]
    bad = S.quant_cfg(4, True, S.SPINQ_PER_TOKEN, 0, 1.5)
    assert S.spinq_rotate_quant_act(fake, 4, 256, 256, None, ctypes.byref(bad), fake, fake, None, None) == S.SPINQ_EINVAL
    # bits != 4 -> unsupported
    b8 = S.quant_cfg(8, True, S.SPINQ_PER_TOKEN, 0, 1.0)
    assert S.spinq_rotate_quant_act(fake, 4, 256, 256, None, ctypes.byref(b8), fake, fake, None, None) == S.SPINQ_EUNSUPPORTED
    # asymmetric without a zero buffer
    qa = S.quant_cfg(4, False, S.SPINQ_PER_TOKEN, 0, 1.0)
    assert S.spinq_rotate_quant_act(fake, 4, 256, 256, None, ctypes.byref(qa), fake, fake, None, None) == S.SPINQ_EINVAL
    # GEMM: K not a multiple of 128, N not a multiple of 16
    assert S.spinq_w4a4_gemm(fake, fake, None, fake, fake, fake, 4, 32, 96, fake, None, None) == S.SPINQ_EINVAL
    assert S.spinq_w4a4_gemm(fake, fake, None, fake, fake, fake, 4, 40, 128, fake, None, None) == S.SPINQ_EINVAL
    # weight quantizer must be symmetric per-channel
    qw = S.quant_cfg(4, False, S.SPINQ_PER_CHANNEL, 0, 1.0)
    assert S.spinq_quant_weight(fake, 8, 256, None, ctypes.byref(qw), fake, fake, fake, None) == S.SPINQ_EUNSUPPORTED
    # KV: group must equal head_dim, spec must be {1, D}
    kvq = S.quant_cfg(4, False, S.SPINQ_PER_GROUP, 64, 1.0)
    had = S.HadCfg(1, 128)
    assert S.spinq_rotate_quant_kv(fake, fake, fake, fake, 1, 1, 4, 2, 128, ctypes.byref(had), ctypes.byref(kvq),
                                   fake, fake, fake, fake, fake, fake, None) == S.SPINQ_EUNSUPPORTED
    had = S.HadCfg(1, 64)
    kvq = S.quant_cfg(4, False, S.SPINQ_PER_GROUP, 128, 1.0)
    assert S.spinq_rotate_quant_kv(fake, fake, fake, fake, 1, 1, 4, 2, 128, ctypes.byref(had), ctypes.byref(kvq),
                                   fake, fake, fake, fake, fake, fake, None) == S.SPINQ_EINVAL


def test_empty_problems_are_ok_without_launch(lib):
    from paper_2405_16406_gb300 import spinq as S
    q = S.quant_cfg(4, True, S.SPINQ_PER_TOKEN, 0, 1.0)
    fake = ctypes.c_void_p(1 << 20)
    assert S.spinq_rotate_quant_act(fake, 0, 256, 256, None, ctypes.byref(q), fake, fake, None, None) == S.SPINQ_OK
    assert S.spinq_w4a4_gemm(fake, fake, None, fake, fake, fake, 0, 32, 128, fake, None, None) == S.SPINQ_OK


def test_gemm_controls_validate_on_the_host(lib):
    """The kernel selection, the K-slice control and the plan queries check
    their arguments on the host; rejected values change nothing."""
    from paper_2405_16406_gb300 import spinq as S
    for bad in (-1, S.SPINQ_GEMM_TCGEMV + 1, 99):
        assert S.spinq_gemm_select_kernel(bad) == -1
    prev = S.spinq_gemm_select_kernel(S.SPINQ_GEMM_TILE256)
    try:
        assert S.spinq_gemm_select_kernel(S.SPINQ_GEMM_TILE128) == S.SPINQ_GEMM_TILE256
    finally:
        S.spinq_gemm_select_kernel(prev)
    for bad in (-1, 65, 1000):
        assert S.spinq_gemm_split_k(bad) == -1
    prev = S.spinq_gemm_split_k(7)
    try:
        assert S.spinq_gemm_split_k(0) == 7
    finally:
        S.spinq_gemm_split_k(prev)
    # shapes every GEMM entry point rejects: no device query, -1
    for M, N, K in ((0, 256, 128), (16, 100, 128), (16, 256, 100), (16, 256, 0), (-1, 256, 128)):
        assert S.spinq_w4a4_gemm_plan(M, N, K) == -1
        assert S.spinq_w4a4_gemm_splitk_plan(M, N, K) == (-1, 0)
    assert S.spinq_w4a4_gemm_splitk_plan(16, 256, 65536 + 128) == (-1, 0)   # K above the exact-accumulator bound


def test_noalloc_rejects_invalid_arguments_on_the_host(lib):
    """spinq_w4a4_gemm_noalloc validates its arguments like spinq_w4a4_gemm
    before any device work: null pointers, K % 128, N % 16, misalignment and
    K above the exact-accumulator bound."""
    from paper_2405_16406_gb300 import spinq as S
    fake = ctypes.c_void_p(1 << 20)
    odd = ctypes.c_void_p((1 << 20) + 4)
    f = S.spinq_w4a4_gemm_noalloc
    assert f(None, fake, None, fake, fake, fake, 4, 32, 128, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, None, None, fake, fake, 4, 32, 128, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, None, fake, fake, fake, 4, 32, 128, None, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, None, fake, fake, fake, 4, 32, 96, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, None, fake, fake, fake, 4, 40, 128, fake, None, None) == S.SPINQ_EINVAL
    assert f(odd, fake, None, fake, fake, fake, 4, 32, 128, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, None, fake, fake, odd, 4, 32, 128, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, None, fake, fake, fake, 4, 32, 128, fake, odd, None) == S.SPINQ_EINVAL
    assert f(fake, fake, None, fake, fake, fake, -1, 32, 128, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, None, fake, fake, fake, 4, 32, 65536 + 128, fake, None, None) == S.SPINQ_EUNSUPPORTED
    # empty problems succeed without a launch
    assert f(fake, fake, None, fake, fake, fake, 0, 32, 128, fake, None, None) == S.SPINQ_OK
    assert "workspace" in S.spinq_status_string(S.SPINQ_ESCRATCH)


def test_cayley_step_rejects_invalid_arguments_on_the_host(lib):
    from paper_2405_16406_gb300 import spinq as S
    fake = ctypes.c_void_p(1 << 20)
    f = S.spinq_cayley_step
    assert f(None, fake, 2, 128, 0.1, 2, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, 2, 128, 0.1, -1, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, 2, 128, 0.1, 65, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, 2, 128, float("nan"), 2, fake, None, None) == S.SPINQ_EINVAL
    assert f(ctypes.c_void_p((1 << 20) + 4), fake, 2, 128, 0.1, 2, fake, None, None) == S.SPINQ_EINVAL
    assert f(fake, fake, 2, 96, 0.1, 2, fake, None, None) == S.SPINQ_EUNSUPPORTED
    assert f(fake, fake, 2, 256, 0.1, 2, fake, None, None) == S.SPINQ_EUNSUPPORTED
    assert f(fake, fake, 0, 128, 0.1, 2, fake, None, None) == S.SPINQ_OK


def test_8bit_entry_points_reject_invalid_arguments_on_the_host(lib):
    from paper_2405_16406_gb300 import spinq as S
    fake = ctypes.c_void_p(1 << 20)
    q8 = S.quant_cfg(8, True, S.SPINQ_PER_TOKEN, 0, 1.0)
    q4 = S.quant_cfg(4, True, S.SPINQ_PER_TOKEN, 0, 1.0)
    a8 = S.spinq_rotate_quant_act8
    assert a8(fake, 4, 200, 256, None, ctypes.byref(q8), S.SPINQ_FMT_E4M3, fake, fake, None, None) == S.SPINQ_EINVAL
    assert a8(fake, 4, 256, 256, None, ctypes.byref(q8), S.SPINQ_FMT_INT4_BYTES, fake, fake, None, None) == S.SPINQ_EINVAL
    assert a8(fake, 4, 256, 256, None, ctypes.byref(q4), S.SPINQ_FMT_E4M3, fake, fake, None, None) == S.SPINQ_EUNSUPPORTED
    qa = S.quant_cfg(8, False, S.SPINQ_PER_TOKEN, 0, 1.0)
    assert a8(fake, 4, 256, 256, None, ctypes.byref(qa), S.SPINQ_FMT_INT8_PLANES, fake, fake, None, None) == S.SPINQ_EINVAL
    assert a8(fake, 4, 256, 256, None, ctypes.byref(qa), S.SPINQ_FMT_E4M3, fake, fake, fake, None) == S.SPINQ_EUNSUPPORTED
    assert a8(fake, 0, 256, 256, None, ctypes.byref(q8), S.SPINQ_FMT_E4M3, fake, fake, None, None) == S.SPINQ_OK
    w8 = S.spinq_quant_weight8
    qw = S.quant_cfg(4, True, S.SPINQ_PER_CHANNEL, 0, 1.0)
    assert w8(fake, 8, 256, None, ctypes.byref(qw), S.SPINQ_FMT_INT4_BYTES, fake, fake, None, None) == S.SPINQ_EINVAL
    assert w8(fake, 8, 256, None, ctypes.byref(qw), S.SPINQ_FMT_INT8_PLANES, fake, fake, fake, None) == S.SPINQ_EINVAL
    g = S.spinq_w4a8_gemm
    assert g(fake, fake, None, fake, fake, fake, 4, 32, 16384 + 128, fake, None, None) == S.SPINQ_EUNSUPPORTED
    assert g(fake, fake, None, fake, fake, None, 4, 32, 256, fake, None, None) == S.SPINQ_EINVAL
    assert g(fake, fake, None, fake, fake, fake, 4, 40, 256, fake, None, None) == S.SPINQ_EINVAL
    f = S.spinq_fp8_gemm
    assert f(fake, fake, fake, fake, 4, 32, 96, fake, None) == S.SPINQ_EINVAL
    assert f(fake, fake, fake, fake, 0, 32, 128, fake, None) == S.SPINQ_OK


def test_attention_entry_points_reject_invalid_arguments_on_the_host(lib):
    from paper_2405_16406_gb300 import spinq as S
    fake = ctypes.c_void_p(1 << 20)
    f = S.spinq_decode_attention_kv4
    need = S.spinq_decode_attention_workspace_bytes(2, 64, 32, 8, 128)
    assert need > 0 and S.spinq_decode_attention_workspace_bytes(0, 64, 32, 8, 128) == 0
    args = [fake] * 7 + [None]
    assert f(*args, 2, 64, 30, 8, 128, 0.1, fake, fake, need, None) == S.SPINQ_EINVAL          # Hq % Hkv
    assert f(*args, 2, 64, 32, 8, 128, 0.1, fake, fake, need - 16, None) == S.SPINQ_EINVAL     # workspace
    assert f(*args, 2, 64, 32, 8, 96, 0.1, fake, fake, 1 << 30, None) == S.SPINQ_EUNSUPPORTED  # D
    assert f(*args, 2, 64, 48, 2, 128, 0.1, fake, fake, 1 << 30, None) == S.SPINQ_EUNSUPPORTED  # G = 24
    assert f(*args, 1, 1 << 23, 32, 8, 128, 0.1, fake, fake, 1 << 40, None) == S.SPINQ_EUNSUPPORTED  # 4 GiB batch
    assert f(*args, 0, 64, 32, 8, 128, 0.1, None, None, 0, None) == S.SPINQ_OK
    g = S.spinq_rope_rotate_quant_kv
    kvq = S.quant_cfg(4, False, S.SPINQ_PER_GROUP, 128, 1.0)
    had = S.HadCfg(1, 128)
    assert g(fake, fake, fake, fake, None, fake, 4096, 1, 4, 4, 2, 128, ctypes.byref(had), ctypes.byref(kvq),
             fake, fake, fake, fake, fake, fake, None) == S.SPINQ_EINVAL                       # no positions
    assert g(fake, fake, fake, fake, fake, ctypes.c_void_p((1 << 20) + 8), 4096, 1, 4, 4, 2, 128, ctypes.byref(had),
             ctypes.byref(kvq), fake, fake, fake, fake, fake, fake, None) == S.SPINQ_EINVAL    # table alignment


def test_signed_and_fused_entry_points_reject_invalid_arguments_on_the_host(lib):
    from paper_2405_16406_gb300 import spinq as S
    fake = ctypes.c_void_p(1 << 20)
    q = S.quant_cfg(4, True, S.SPINQ_PER_TOKEN, 0, 1.0)
    had = S.HadCfg(28, 512)
    # signs need a rotation and a mask
    assert S.spinq_rotate_quant_act_signed(fake, 4, 14336, 14336, None, fake, ctypes.byref(q), fake, fake, None,
                                           None) == S.SPINQ_EINVAL
    assert S.spinq_rotate_quant_act_signed(fake, 4, 14336, 14336, ctypes.byref(had), None, ctypes.byref(q), fake,
                                           fake, None, None) == S.SPINQ_EINVAL
    qw = S.quant_cfg(4, True, S.SPINQ_PER_CHANNEL, 0, 1.0)
    assert S.spinq_quant_weight_signed(fake, 4, 14336, None, fake, ctypes.byref(qw), fake, fake, fake,
                                       None) == S.SPINQ_EINVAL
    need = S.spinq_rotated_linear_workspace_bytes(2048, 14336)
    assert need >= 2048 * 7168 + 2 * 2048 * 4
    f = S.spinq_rotated_linear
    assert f(fake, 2048, 14336, 14336, ctypes.byref(had), None, ctypes.byref(q), fake, fake, fake, 4096, fake,
             fake, need - 256, None) == S.SPINQ_EINVAL          # workspace too small
    assert f(fake, 2048, 14336, 14336, ctypes.byref(had), None, ctypes.byref(q), fake, fake, fake, 4100, fake,
             fake, need, None) == S.SPINQ_EINVAL                 # N % 16
    assert f(fake, 0, 14336, 14336, ctypes.byref(had), None, ctypes.byref(q), fake, fake, fake, 4096, fake,
             None, 0, None) == S.SPINQ_OK


def test_debug_controls_validate_on_the_host(lib):
    from paper_2405_16406_gb300 import spinq as S
    assert S.spinq_debug_set_wait_limit_ns(0) == S.SPINQ_EINVAL
    assert S.spinq_debug_set_wait_limit_ns(-5) == S.SPINQ_EINVAL
    assert S.spinq_debug_fail_launches(-1) == -1
    assert S.spinq_debug_fail_launches(0) == 0
