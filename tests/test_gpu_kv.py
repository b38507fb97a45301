"""GPU parity: spinq_rotate_quant_kv vs the oracle (R3 + asymmetric KV4)."""
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


def check(S, c, sample_rows=None, clip=1.0, in_place=False):
    q = torch.from_numpy(c.q).cuda()
    k = torch.from_numpy(c.k).cuda()
    v = torch.from_numpy(c.v).cuda()
    out = S.rotate_quant_kv(q, k, v, clip=clip, in_place_q=in_place)
    torch.cuda.synchronize()
    D = c.D
    qo = out.q_out.cpu().numpy().reshape(-1, D)
    kc = pu.gpu_codes(out.k_codes.cpu().numpy().reshape(-1, D // 2), False)
    vc = pu.gpu_codes(out.v_codes.cpu().numpy().reshape(-1, D // 2), False)
    ks, kz = out.k_scale.cpu().numpy().reshape(-1), out.k_zero.cpu().numpy().reshape(-1)
    vs, vz = out.v_scale.cpu().numpy().reshape(-1), out.v_zero.cpu().numpy().reshape(-1)
    qin, kin, vin = c.q.reshape(-1, D), c.k.reshape(-1, D), c.v.reshape(-1, D)
    if sample_rows is not None:
        rng = np.random.default_rng(0)
        rq = np.unique(np.concatenate([rng.integers(0, qin.shape[0], sample_rows), [0, qin.shape[0] - 1]]))
        rk = np.unique(np.concatenate([rng.integers(0, kin.shape[0], sample_rows), [0, kin.shape[0] - 1]]))
    else:
        rq, rk = np.arange(qin.shape[0]), np.arange(kin.shape[0])
    ref = oracle.rotate_quant_kv(qin[rq][None, None], kin[rk][None, None], vin[rk][None, None], c.had, 4, clip)
    # Q: the GPU rounds an fp32 rotation (error <= 2^-20 ||x_row||_2 for a
    # D <= 128 point transform with fp32 sums) once to fp16; the oracle rounds
    # the exact value once.  So |q_gpu - q_exact| <= ulp16(q_exact) + 2^-20 ||x_row||.
    got_q = qo[rq].astype(np.float64)
    exact = ref.q_rot.reshape(-1, D)
    xnorm = np.linalg.norm(qin[rq].astype(np.float64), axis=1, keepdims=True)
    ulp = np.spacing(np.abs(exact).astype(np.float16)).astype(np.float64)
    assert np.all(np.abs(got_q - exact) <= ulp + 2.0 ** -20 * xnorm)
    assert np.count_nonzero(got_q != ref.q_out.reshape(-1, D)) / got_q.size <= 1e-3
    pu.assert_codes_close(kc[rk], ref.k_codes.reshape(-1, D), "K codes")
    pu.assert_codes_close(vc[rk], ref.v_codes.reshape(-1, D), "V codes")
    pu.assert_scale_close(ks[rk], ref.k_alpha.reshape(-1), "K alpha")
    pu.assert_zero_close(kz[rk], ref.k_beta.reshape(-1), ref.k_alpha.reshape(-1), "K beta")
    pu.assert_scale_close(vs[rk], ref.v_alpha.reshape(-1), "V alpha")
    pu.assert_zero_close(vz[rk], ref.v_beta.reshape(-1), ref.v_alpha.reshape(-1), "V beta")


def test_kv_small_all_rows(S):
    check(S, synth.kv_case(B=2, S=37, Hq=4, Hkv=2, D=128))


def test_kv_d64_ragged(S):
    check(S, synth.kv_case(B=1, S=13, Hq=3, Hkv=1, D=64))


def test_kv_clip(S):
    check(S, synth.kv_case(B=1, S=64, Hq=8, Hkv=2, D=128), clip=0.95)


def test_kv_in_place_q(S):
    check(S, synth.kv_case(B=1, S=33, Hq=8, Hkv=8, D=128), in_place=True)


def test_kv_full_config_sampled(S):
    check(S, synth.kv_case(), sample_rows=20000)
