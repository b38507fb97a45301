"""Pins of the oracle's RoPE and decode attention (Sec. 3.1: R3 rotates Q and
K so that Q K^T is unchanged while the cache quantizes to 4 bits) against what
the mathematics fixes: RoPE keeps each rotated pair's norm, is the identity at
position 0, turns a D = 2 vector by p theta_0 = p radians, and makes
<RoPE(q, m), RoPE(k, n)> depend on m - n only; attention scores are unchanged
by a common orthonormal rotation of q and k (so R3 leaves the output alone);
equal keys give the mean of the values; a length of one returns the first
value; a dominant key selects its value."""
import numpy as np

import oracle


def test_rope_closed_forms():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((5, 16))
    np.testing.assert_allclose(oracle.rope(x, np.zeros(5, np.int64)), x, atol=0)
    y = oracle.rope(x, np.arange(5) * 37)
    np.testing.assert_allclose(np.hypot(y[:, :8], y[:, 8:]), np.hypot(x[:, :8], x[:, 8:]), rtol=1e-13)
    v = np.array([[1.0, 0.0]])
    for p in (1, 3, 100):
        np.testing.assert_allclose(oracle.rope(v, np.array([p]), base=10000.0), [[np.cos(p), np.sin(p)]], atol=1e-12)


def test_rope_relative_position_property():
    rng = np.random.default_rng(1)
    D = 128
    q, k = rng.standard_normal(D), rng.standard_normal(D)
    for m, n in ((7, 3), (4000, 10), (33, 33), (2, 90)):
        lhs = oracle.rope(q[None], np.array([m]))[0] @ oracle.rope(k[None], np.array([n]))[0]
        rhs = oracle.rope(q[None], np.array([m - n]))[0] @ k
        assert abs(lhs - rhs) <= 1e-9 * (np.abs(q) @ np.abs(k))


def _kv(rng, B, S, Hq, Hkv, D):
    return (rng.standard_normal((B, Hq, D)), rng.standard_normal((B, S, Hkv, D)),
            rng.standard_normal((B, S, Hkv, D)))


def test_attention_is_invariant_under_the_r3_rotation():
    rng = np.random.default_rng(2)
    B, S, Hq, Hkv, D = 2, 40, 8, 2, 64
    q, k, v = _kv(rng, B, S, Hq, Hkv, D)
    H = oracle.sylvester(D) / np.sqrt(D)
    o = oracle.decode_attention(q, k, v)
    o_rot = oracle.decode_attention(q @ H, k @ H, v)
    np.testing.assert_allclose(o_rot, o, atol=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(3)
    B, S, Hq, Hkv, D = 1, 12, 4, 2, 32
    q, k, v = _kv(rng, B, S, Hq, Hkv, D)
    keq = np.broadcast_to(k[:, :1], k.shape).copy()
    np.testing.assert_allclose(oracle.decode_attention(q, keq, v),
                               np.repeat(v.mean(axis=1), Hq // Hkv, axis=1), atol=1e-12)
    np.testing.assert_allclose(oracle.decode_attention(q, k, v, lens=np.array([1])),
                               np.repeat(v[:, 0], Hq // Hkv, axis=1), atol=1e-12)
    # key 5 of kv head 0 aligned with query head 0 and very large: selects v[5]
    k2 = k.copy()
    k2[0, 5, 0] = 1e3 * q[0, 0]
    o = oracle.decode_attention(q, k2, v)
    np.testing.assert_allclose(o[0, 0], v[0, 5, 0], atol=1e-9)
    # GQA: query heads 0, 1 read kv head 0; 2, 3 read kv head 1
    o = oracle.decode_attention(q, k, v)
    one = oracle.decode_attention(q[:, 2:3], k[:, :, 1:2], v[:, :, 1:2])
    np.testing.assert_allclose(o[:, 2:3], one, atol=1e-14)
