"""Variants of the path on the GPU against the oracle: the bidirectional
encoder (Eq. 1 with no mask: attention, column mass and whole pruned
forwards) and the literal soft-score criterion (column mass without the
||v|| factor, reading R1's alternative)."""

import dataclasses

import numpy as np
import pytest
import torch

from oracle import zsaa_oracle as O
from tests.helpers import bf16_ulp_close, need_gpu
from tests.test_gpu_forward import SMALL_BF16, SMALL_BF16_128, SMALL_CLS, check_case, run_case
from tests.test_gpu_ops import _np, _oracle_attention, _qkv
from paper_2509_01190_gb300 import inputs as I

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def z(zlib):
    need_gpu()
    return zlib


@pytest.mark.parametrize("B,N,Hq,Hkv,hd", [(2, 1, 4, 2, 64), (2, 65, 4, 2, 64), (1, 200, 4, 1, 128),
                                           (2, 130, 8, 2, 128), (1, 300, 4, 2, 64), (1, 600, 8, 2, 128)])
def test_bidirectional_attention_and_colmass_bf16(z, B, N, Hq, Hkv, hd):
    qkv = _qkv(B, N, Hq, Hkv, hd, 60 + N, torch.bfloat16)
    out = torch.empty(B * N, Hq * hd, device="cuda", dtype=torch.bfloat16)
    lse = torch.empty(B, Hq, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_attention_ex(qkv, B, N, Hq, Hkv, hd, z.ZSAA_BF16, False, out, lse)
    torch.cuda.synchronize()
    ref_o, ref_lse, Ps, _ = _oracle_attention(qkv, B, N, Hq, Hkv, hd, causal=False)
    got = _np(out).reshape(B, N, Hq * hd)
    ref_b = O.bf16_round(ref_o)
    tol = 1e-5 * np.abs(ref_o).max(axis=-1, keepdims=True)
    assert np.all(bf16_ulp_close(got, ref_b, 1, tol))
    assert np.mean(got == ref_b) > 0.95, np.mean(got == ref_b)
    np.testing.assert_allclose(_np(lse), ref_lse, rtol=1e-5, atol=1e-4)
    C = torch.empty(B, Hkv, N, device="cuda", dtype=torch.float32)
    lse_in = torch.from_numpy(ref_lse.astype(np.float32)).cuda()
    z.zsaa_op_colmass_ex(qkv, lse_in, B, N, Hq, Hkv, hd, z.ZSAA_BF16, False, C)
    torch.cuda.synchronize()
    refC = np.stack([O.column_mass(Ps[b], Hkv) for b in range(B)])
    np.testing.assert_allclose(_np(C), refC, rtol=2e-4, atol=1e-5)
    np.testing.assert_allclose(_np(C).sum(axis=2), (Hq // Hkv) * N, rtol=1e-4)
    # the causal entry points still mask: their column mass differs
    Cc = torch.empty_like(C)
    z.zsaa_op_attention(qkv, B, N, Hq, Hkv, hd, z.ZSAA_BF16, out, lse)
    z.zsaa_op_colmass(qkv, lse, B, N, Hq, Hkv, hd, z.ZSAA_BF16, Cc)
    torch.cuda.synchronize()
    if N > 1:
        assert np.abs(_np(Cc) - _np(C)).max() > 1e-3


@pytest.mark.parametrize("B,N,Hq,Hkv,hd", [(2, 64, 4, 4, 32), (1, 37, 4, 2, 32)])
def test_bidirectional_attention_and_colmass_f32(z, B, N, Hq, Hkv, hd):
    qkv = _qkv(B, N, Hq, Hkv, hd, 70 + N, torch.float32)
    out = torch.empty(B * N, Hq * hd, device="cuda", dtype=torch.float32)
    lse = torch.empty(B, Hq, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_attention_ex(qkv, B, N, Hq, Hkv, hd, z.ZSAA_F32, False, out, lse)
    torch.cuda.synchronize()
    ref_o, ref_lse, Ps, _ = _oracle_attention(qkv, B, N, Hq, Hkv, hd, causal=False)
    np.testing.assert_allclose(_np(out).reshape(B, N, Hq * hd), ref_o, rtol=1e-5, atol=1e-5)
    C = torch.empty(B, Hkv, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_colmass_ex(qkv, lse, B, N, Hq, Hkv, hd, z.ZSAA_F32, False, C)
    torch.cuda.synchronize()
    refC = np.stack([O.column_mass(Ps[b], Hkv) for b in range(B)])
    np.testing.assert_allclose(_np(C), refC, rtol=1e-5, atol=1e-6)


ENC = dataclasses.replace(SMALL_BF16, name="small-encoder", bidirectional=True)
ENC_128 = dataclasses.replace(SMALL_BF16_128, name="small-encoder-hd128", bidirectional=True)
ENC_CLS = dataclasses.replace(SMALL_CLS, name="small-encoder-cls", bidirectional=True)
SOFT = dataclasses.replace(SMALL_BF16, name="small-softscore", score_mode="softscore")


@pytest.mark.parametrize("accel", [1.0, 3.0])
def test_bidirectional_small_lm(z, accel):
    res = run_case(z, ENC, 3, 150, accel, seqs=[0, 2])
    check_case(res, "bf16")


def test_bidirectional_small_hd128_and_classifier(z):
    # the configuration of the causal hd-128 case
    check_case(run_case(z, ENC_128, 2, 333, 3.0, seqs=[0, 1]), "bf16")
    res = run_case(z, ENC_CLS, 4, 130, 3.0, seqs=[1, 3])
    check_case(res, "bf16")
    assert res["forced_logits"].shape == (4, 4)


def test_bidirectional_tiny_f32(z):
    wl = I.WORKLOADS["tiny"]
    shape = dataclasses.replace(wl["shape"], name="tiny-encoder", bidirectional=True)
    res = run_case(z, shape, wl["B"], wl["L"], wl["accels"][0], seqs=[0, 1])
    check_case(res, "f32")
    np.testing.assert_array_equal(res["nat_idx"][1], res["ores"]["idx"][1])


@pytest.mark.parametrize("accel", [2.0, 5.0])
def test_softscore_criterion_small_lm(z, accel):
    res = run_case(z, SOFT, 3, 180, accel, seqs=[0, 1, 2])
    check_case(res, "bf16")


def test_bidirectional_model_refuses_generation(z):
    w = I.make_weights(ENC, device="cuda")
    model = z.Model(z.config_from_shape(ENC), w, 1, 16)
    with pytest.raises(z.ZsaaError) as e:
        z.Cache(model, 1, 16, 2.0, 2)
    assert e.value.status == z.ZSAA_ERR_UNSUPPORTED
