"""RoPE + R3 + KV4 (spinq_rope_rotate_quant_kv) and decode attention over the
4-bit cache (spinq_decode_attention_kv4) on the GPU against the oracle.

Bars.  KV codes: +-1 on at most 1e-4 (ties), scales within 1e-5 (as the KV
path without RoPE).  Q': the GPU rounds its fp32 RoPE to fp16 and the oracle
its double RoPE; the two roundings can differ by one fp16 ulp (on ~1e-4 of
the elements), which moves every R3 output of that row by at most
ulp16(max|x|) / sqrt(D); with the R3 bound of the plain KV path this gives
|dq| <= ulp16(q) + 2^-20 |x| + 2 ulp16(max|x|) / sqrt(D).  Attention: the
oracle runs on the GPU's own codes and scales (dequantized in double), so the
kernel is compared on identical inputs; tensor-core products with fp32
accumulation (exact fp16 query times exact code), fp16 weights p v_scale / r
(relative rounding 2^-12 each) and the fp16 output rounding against double:
elementwise within 2e-3 |o| + 2e-3 max|o|."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2405_16406_gb300 import synth
from parity_util import assert_codes_close, assert_scale_close, assert_zero_close, rel_frob

pytestmark = pytest.mark.gpu

BASE = 500000.0


def _cos_sin(max_pos, D):
    th = BASE ** (-2.0 * np.arange(D // 2) / D)
    ang = np.arange(max_pos)[:, None] * th[None, :]
    return np.stack([np.cos(ang), np.sin(ang)], axis=-1).astype(np.float32)   # [max_pos, D/2, 2]


def _ulp16(v):
    a = np.abs(v)
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -14)))
    return 2.0 ** (e - 10)


@pytest.mark.parametrize("D", [64, 128])
def test_rope_rotate_quant_kv_matches_oracle(D):
    from paper_2405_16406_gb300 import spinq
    kv = synth.kv_case(seed=D, B=2, S=67, Hq=8, Hkv=2, D=D)
    rng = np.random.default_rng(D)
    pos = rng.integers(0, 8192, (kv.B, kv.S)).astype(np.int32)
    cs = _cos_sin(8192, D)
    out = spinq.rope_rotate_quant_kv(torch.from_numpy(kv.q).cuda(), torch.from_numpy(kv.k).cuda(),
                                     torch.from_numpy(kv.v).cuda(), torch.from_numpy(pos).cuda(),
                                     torch.from_numpy(cs).cuda())
    torch.cuda.synchronize()
    ref = oracle.rope_rotate_quant_kv(kv.q, kv.k, kv.v, pos, kv.had, BASE)
    gk = oracle.unpack4(out.k_codes.cpu().numpy().reshape(-1, D // 2), False)
    gv = oracle.unpack4(out.v_codes.cpu().numpy().reshape(-1, D // 2), False)
    assert_codes_close(gk, ref.k_codes.reshape(-1, D), "K")
    assert_codes_close(gv, ref.v_codes.reshape(-1, D), "V")
    # a one-ulp difference of the fp16 RoPE output moves the unnormalised
    # range of the rotated row by at most 2 ulp16(max|x|): alpha by that / 15
    # and beta by ulp16(max|x|), both times 1/sqrt(D)
    kp = oracle.f16_to_f64(oracle.f64_to_f16(
        oracle.rope(oracle.f16_to_f64(kv.k).reshape(-1, D), np.repeat(pos.reshape(-1), kv.Hkv), BASE)))
    u = _ulp16(np.abs(kp).max(axis=1)) / np.sqrt(D)
    ka, kb = ref.k_alpha.reshape(-1), ref.k_beta.reshape(-1)
    assert np.all(np.abs(out.k_scale.cpu().numpy().reshape(-1) - ka) <= 1e-5 * ka + 2 * u / 15)
    assert np.all(np.abs(out.k_zero.cpu().numpy().reshape(-1) - kb) <= 1e-5 * (np.abs(kb) + ka) + u)
    assert_scale_close(out.v_scale.cpu().numpy().reshape(-1), ref.v_alpha.reshape(-1), "v alpha")
    # Q'
    qp = oracle.rope(oracle.f16_to_f64(kv.q).reshape(-1, D), np.repeat(pos.reshape(-1), kv.Hq), BASE)
    qp16 = oracle.f16_to_f64(oracle.f64_to_f16(qp))
    got = out.q_out.cpu().numpy().astype(np.float64).reshape(-1, D)
    exact = ref.q_rot.reshape(-1, D)
    norm = np.linalg.norm(qp16, axis=1, keepdims=True)
    bound = _ulp16(exact) + 2.0 ** -20 * norm + 2 * _ulp16(np.abs(qp16).max(axis=1, keepdims=True)) / np.sqrt(D)
    assert np.all(np.abs(got - exact) <= bound)
    # position 0 everywhere is the plain R3 + KV4 path
    z = np.zeros_like(pos)
    out0 = spinq.rope_rotate_quant_kv(torch.from_numpy(kv.q).cuda(), torch.from_numpy(kv.k).cuda(),
                                      torch.from_numpy(kv.v).cuda(), torch.from_numpy(z).cuda(),
                                      torch.from_numpy(cs).cuda())
    plain = spinq.rotate_quant_kv(torch.from_numpy(kv.q).cuda(), torch.from_numpy(kv.k).cuda(),
                                  torch.from_numpy(kv.v).cuda())
    torch.cuda.synchronize()
    assert torch.equal(out0.k_codes, plain.k_codes) and torch.equal(out0.q_out, plain.q_out)


def _attention_case(seed, B, S, Hq, Hkv, D, lens=None):
    """A rotated, quantized cache from the GPU quantizer and decode queries."""
    from paper_2405_16406_gb300 import spinq
    kv = synth.kv_case(seed=seed, B=B, S=S, Hq=Hkv, Hkv=Hkv, D=D)
    cache = spinq.rotate_quant_kv(torch.from_numpy(kv.q).cuda(), torch.from_numpy(kv.k).cuda(),
                                  torch.from_numpy(kv.v).cuda())
    rng = np.random.default_rng(seed + 1)
    q = (rng.standard_normal((B, Hq, D)) * 2).astype(np.float16)
    L = None if lens is None else torch.tensor(lens, dtype=torch.int32, device="cuda")
    return cache, q, L


def _oracle_attention(cache, q, lens, D):
    ka = cache.k_scale.double().cpu().numpy()
    kb = cache.k_zero.double().cpu().numpy()
    va = cache.v_scale.double().cpu().numpy()
    vb = cache.v_zero.double().cpu().numpy()
    kc = oracle.unpack4(cache.k_codes.cpu().numpy(), False)
    vc = oracle.unpack4(cache.v_codes.cpu().numpy(), False)
    k = oracle.dequant_kv(kc, ka, kb)
    v = oracle.dequant_kv(vc, va, vb)
    return oracle.decode_attention(q.astype(np.float64), k, v, None if lens is None else lens.cpu().numpy())


@pytest.mark.parametrize("B,S,Hq,Hkv,D,lens", [
    (1, 1, 8, 8, 128, None),
    (2, 37, 32, 8, 128, [37, 5]),
    (3, 300, 16, 8, 64, [1, 300, 151]),
    (2, 1000, 64, 8, 128, None),
    (1, 513, 8, 4, 64, None),
])
def test_decode_attention_matches_oracle(B, S, Hq, Hkv, D, lens):
    from paper_2405_16406_gb300 import spinq
    cache, q, L = _attention_case(S + Hq, B, S, Hq, Hkv, D, lens)
    o = spinq.decode_attention_kv4(torch.from_numpy(q).cuda(), cache, L)
    torch.cuda.synchronize()
    ref = _oracle_attention(cache, q, L, D)
    got = o.cpu().numpy().astype(np.float64)
    assert rel_frob(got, ref) <= 2e-3
    assert np.all(np.abs(got - ref) <= 2e-3 * np.abs(ref) + 2e-3 * np.abs(ref).max())
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK


@pytest.mark.parametrize("v_mag", [1e-4, 30.0])
def test_decode_attention_value_scale_range(v_mag):
    """Values far below and above 1 (outputs up to ~2600, within fp16): the
    fp16 weights p v_scale / r are scaled by the running maximum r of the
    value scales, so they stay in [0, 1] and clear of the subnormal range."""
    from paper_2405_16406_gb300 import spinq
    B, S, Hq, Hkv, D = 2, 777, 16, 4, 128
    cache, q, _ = _attention_case(5, B, S, Hq, Hkv, D)
    cache = dataclasses.replace(cache, v_scale=cache.v_scale * v_mag, v_zero=cache.v_zero * v_mag)
    o = spinq.decode_attention_kv4(torch.from_numpy(q).cuda(), cache)
    torch.cuda.synchronize()
    ref = _oracle_attention(cache, q, None, D)
    got = o.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(got))
    assert np.all(np.abs(got - ref) <= 2e-3 * np.abs(ref) + 2e-3 * np.abs(ref).max())


def test_decode_attention_one_chunk_long_cache():
    """B * Hkv large enough that each (batch, kv head) runs as one chunk over
    a long cache (many steps per warp, the online rescaling over thousands of
    tokens)."""
    from paper_2405_16406_gb300 import spinq
    B, S, Hq, Hkv, D = 80, 1500, 64, 8, 64
    cache, q, _ = _attention_case(9, B, S, Hq, Hkv, D)
    assert spinq.spinq_decode_attention_workspace_bytes(B, S, Hq, Hkv, D) == B * Hq * (D + 2) * 4
    o = spinq.decode_attention_kv4(torch.from_numpy(q).cuda(), cache)
    torch.cuda.synchronize()
    got = o.cpu().numpy().astype(np.float64)
    for b in (0, 41, 79):
        sub = spinq.KVCodes(None, cache.k_codes[b:b + 1], cache.k_scale[b:b + 1], cache.k_zero[b:b + 1],
                            cache.v_codes[b:b + 1], cache.v_scale[b:b + 1], cache.v_zero[b:b + 1])
        ref = _oracle_attention(sub, q[b:b + 1], None, D)[0]
        assert np.all(np.abs(got[b] - ref) <= 2e-3 * np.abs(ref) + 2e-3 * np.abs(ref).max())
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK


def test_decode_attention_full_config4_cache_sampled():
    """Config 4's cache (B 8, S 4096, 32 q / 8 kv heads, D 128) from the
    RoPE + R3 + KV4 kernel, one decode query per head; three batches checked
    against the oracle on the same codes."""
    from paper_2405_16406_gb300 import spinq
    kv = synth.kv_case()
    rng = np.random.default_rng(11)
    pos = np.tile(np.arange(kv.S, dtype=np.int32), (kv.B, 1))
    cs = _cos_sin(kv.S + 1, kv.D)
    cache = spinq.rope_rotate_quant_kv(torch.from_numpy(kv.q).cuda(), torch.from_numpy(kv.k).cuda(),
                                       torch.from_numpy(kv.v).cuda(), torch.from_numpy(pos).cuda(),
                                       torch.from_numpy(cs).cuda())
    q = (rng.standard_normal((kv.B, kv.Hq, kv.D)) * 2).astype(np.float16)
    o = spinq.decode_attention_kv4(torch.from_numpy(q).cuda(), cache)
    torch.cuda.synchronize()
    got = o.cpu().numpy().astype(np.float64)
    for b in (0, 3, 7):
        sub = spinq.KVCodes(None, cache.k_codes[b:b + 1], cache.k_scale[b:b + 1], cache.k_zero[b:b + 1],
                            cache.v_codes[b:b + 1], cache.v_scale[b:b + 1], cache.v_zero[b:b + 1])
        ref = _oracle_attention(sub, q[b:b + 1], None, kv.D)[0]
        assert np.all(np.abs(got[b] - ref) <= 2e-3 * np.abs(ref) + 2e-3 * np.abs(ref).max())
    assert spinq.spinq_device_status()[0] == spinq.SPINQ_OK
