"""Per-kernel parity on the GPU, through the C ABI: GEMM epilogues (tensor-core
bf16 and CUDA-core fp32), causal attention (Eq. 1) and the soft-score column
mass, each against the oracle's step (or a float64 matmul for a bare GEMM) on
seeded inputs spanning several tiles and a ragged tail."""

import math

import numpy as np
import pytest
import torch

from oracle import zsaa_oracle as O
from tests.helpers import accum_bound, bf16_ulp_close, need_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def z(zlib):
    need_gpu()
    return zlib


def _rand(shape, seed, scale=1.0, dtype=torch.bfloat16):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    return (torch.randn(*shape, generator=g, device="cuda") * scale).to(dtype)


def _np(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


# (3, 1024, 4096): the weight-streaming kernel's 16-warp form (K >= 4096, few bands)
@pytest.mark.parametrize("M,N,K", [(1, 64, 64), (300, 384, 256), (128, 256, 128), (517, 1024, 512),
                                   (40, 2048, 2048), (3, 1024, 4096)])
def test_linear_bf16_store_and_f32(z, M, N, K):
    A = _rand((M, K), 1)
    W = _rand((N, K), 2)
    ref = _np(A) @ _np(W).T
    out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
    z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE)
    out32 = torch.empty(M, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_linear(A, W, None, None, out32, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
    torch.cuda.synchronize()
    z.zsaa_device_status()
    tol = accum_bound(_np(A), _np(W))
    assert np.all(bf16_ulp_close(_np(out), O.bf16_round(ref), 1, tol))
    # the worst-case bound is loose; nearly every element must also be within 1 ulp
    assert np.mean(bf16_ulp_close(_np(out), O.bf16_round(ref), 1)) > 0.995
    assert np.all(np.abs(_np(out32) - ref) <= tol + 1e-6 * np.abs(ref))


def test_linear_bf16_large_n_lm_head(z):
    M, N, K = 37, 128256, 256
    A = _rand((M, K), 3)
    W = _rand((N, K), 4, 0.02)
    out = torch.empty(M, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
    torch.cuda.synchronize()
    ref = _np(A) @ _np(W).T
    assert np.all(np.abs(_np(out) - ref) <= accum_bound(_np(A), _np(W)) + 1e-6 * np.abs(ref))


# (8, 2048, 8192): a decode step's down projection (16-warp weight streaming)
@pytest.mark.parametrize("M,N,K", [(200, 256, 128), (5, 512, 1024), (1000, 2048, 256), (8, 2048, 8192)])
def test_linear_bf16_residual_in_place(z, M, N, K):
    A = _rand((M, K), 5, 0.1)
    W = _rand((N, K), 6, 0.1)
    H = _rand((M, N), 7)
    h0 = _np(H)
    z.zsaa_op_linear(A, W, None, H, H, M, N, K, z.ZSAA_BF16, z.EPI_RESID)
    torch.cuda.synchronize()
    ref = O.bf16_round(h0 + _np(A) @ _np(W).T)
    assert np.all(bf16_ulp_close(_np(H), ref, 1, accum_bound(_np(A), _np(W))))


@pytest.mark.parametrize("M,F,K", [(130, 384, 256), (7, 1024, 512), (600, 2048, 128)])
def test_linear_bf16_swiglu(z, M, F, K):
    A = _rand((M, K), 8)
    Wg = _rand((F, K), 9, 0.1)
    Wu = _rand((F, K), 10, 0.1)
    out = torch.empty(M, F, device="cuda", dtype=torch.bfloat16)
    z.zsaa_op_linear(A, Wg, Wu, None, out, M, F, K, z.ZSAA_BF16, z.EPI_SWIGLU)
    torch.cuda.synchronize()
    g = _np(A) @ _np(Wg).T
    u = _np(A) @ _np(Wu).T
    ref = O.bf16_round(O.silu(g) * u)
    # d(silu(g) u) = silu'(g) u dg + silu(g) du, |silu'| <= 1.1
    tol = 1.1 * np.abs(u) * accum_bound(_np(A), _np(Wg)) + np.abs(O.silu(g)) * accum_bound(_np(A), _np(Wu))
    assert np.all(bf16_ulp_close(_np(out), ref, 2, tol))


@pytest.mark.parametrize("hd,Hq,Hkv", [(64, 4, 2), (128, 2, 1)])
def test_linear_bf16_rope(z, hd, Hq, Hkv):
    M, K = 333, 256
    N = (Hq + 2 * Hkv) * hd
    rope_cols = (Hq + Hkv) * hd
    A = _rand((M, K), 11)
    W = _rand((N, K), 12, 0.1)
    pos = torch.randint(0, 4096, (M,), generator=torch.Generator().manual_seed(3)).to(torch.int32).cuda()
    out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
    z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_ROPE, pos=pos,
                     rope_cols=rope_cols, rope_hd=hd, rope_theta=500000.0)
    torch.cuda.synchronize()
    acc = _np(A) @ _np(W).T
    cos, sin = O.rope_angles(pos.cpu().numpy(), hd, 500000.0)
    qk = O.apply_rope(acc[:, :rope_cols].reshape(M, Hq + Hkv, hd), cos, sin).reshape(M, rope_cols)
    ref = O.bf16_round(np.concatenate([qk, acc[:, rope_cols:]], axis=1))
    # each rotated value mixes two accumulators; the float32 table adds ~1e-7 relative
    b = accum_bound(_np(A), _np(W))
    bq = b[:, :rope_cols].reshape(M, Hq + Hkv, hd)
    half = hd // 2
    pair = np.concatenate([bq[..., :half] + bq[..., half:], bq[..., :half] + bq[..., half:]], axis=-1)
    tol = np.concatenate([pair.reshape(M, rope_cols), b[:, rope_cols:]], axis=1) + 1e-6 * np.abs(acc)
    assert np.all(bf16_ulp_close(_np(out), ref, 2, tol))


# The projections of the Llama-3.2-1B shape at the full bench batch (8 x 512
# rows): these take the 256-wide tiles that the bench runs.
FULL_1B = [("qkv_rope", 4096, 3072, 2048), ("o_resid", 4096, 2048, 2048),
           ("gate_up_swiglu", 4096, 8192, 2048), ("down_resid", 4096, 2048, 8192)]


@pytest.mark.parametrize("name,M,N,K", FULL_1B)
def test_linear_bf16_full_1b_shapes(z, name, M, N, K):
    A = _rand((M, K), 31)
    W = _rand((N, K), 32, 0.02)
    An, Wn = _np(A), _np(W)
    if name == "qkv_rope":
        hd, rope_cols = 64, 2560
        pos = torch.arange(M, dtype=torch.int32, device="cuda") % 512
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_ROPE, pos=pos,
                         rope_cols=rope_cols, rope_hd=hd, rope_theta=500000.0)
        acc = An @ Wn.T
        cos, sin = O.rope_angles(pos.cpu().numpy(), hd, 500000.0)
        qk = O.apply_rope(acc[:, :rope_cols].reshape(M, -1, hd), cos, sin).reshape(M, rope_cols)
        ref = O.bf16_round(np.concatenate([qk, acc[:, rope_cols:]], axis=1))
        b = accum_bound(An, Wn)
        tol = 2 * b.max(axis=1, keepdims=True) + 1e-6 * np.abs(acc)
    elif name == "gate_up_swiglu":
        W2 = _rand((N, K), 33, 0.02)
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        z.zsaa_op_linear(A, W, W2, None, out, M, N, K, z.ZSAA_BF16, z.EPI_SWIGLU)
        g = An @ Wn.T
        u = An @ _np(W2).T
        ref = O.bf16_round(O.silu(g) * u)
        tol = 1.1 * np.abs(u) * accum_bound(An, Wn) + np.abs(O.silu(g)) * accum_bound(An, _np(W2))
    else:
        H = _rand((M, N), 34)
        h0 = _np(H)
        z.zsaa_op_linear(A, W, None, H, H, M, N, K, z.ZSAA_BF16, z.EPI_RESID)
        out = H
        ref = O.bf16_round(h0 + An @ Wn.T)
        tol = accum_bound(An, Wn)
    torch.cuda.synchronize()
    z.zsaa_device_status()
    got = _np(out)
    assert np.all(bf16_ulp_close(got, ref, 2, tol)), name
    assert np.mean(bf16_ulp_close(got, ref, 1)) > 0.995, name


# Small M with deep K: fewer tiles than SMs, so the GEMM splits K and a
# finishing kernel sums the fp32 partials in a fixed order (every epilogue).
@pytest.mark.parametrize("epi", ["store", "store_f32", "resid", "swiglu", "rope"])
def test_linear_bf16_split_k(z, epi):
    M, K = 40, 4096
    A = _rand((M, K), 51)
    An = _np(A)
    if epi == "rope":
        hd, Hq, Hkv = 64, 4, 2
        N, rope_cols = (Hq + 2 * Hkv) * hd, (Hq + Hkv) * hd
        W = _rand((N, K), 52, 0.02)
        pos = torch.arange(100, 100 + M, dtype=torch.int32, device="cuda")
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_ROPE, pos=pos,
                         rope_cols=rope_cols, rope_hd=hd, rope_theta=10000.0)
        acc = An @ _np(W).T
        cos, sin = O.rope_angles(pos.cpu().numpy(), hd, 10000.0)
        qk = O.apply_rope(acc[:, :rope_cols].reshape(M, -1, hd), cos, sin).reshape(M, rope_cols)
        ref = O.bf16_round(np.concatenate([qk, acc[:, rope_cols:]], axis=1))
        tol = 2 * accum_bound(An, _np(W)).max(axis=1, keepdims=True)
    elif epi == "swiglu":
        F = 1024
        Wg, Wu = _rand((F, K), 53, 0.02), _rand((F, K), 54, 0.02)
        out = torch.empty(M, F, device="cuda", dtype=torch.bfloat16)
        z.zsaa_op_linear(A, Wg, Wu, None, out, M, F, K, z.ZSAA_BF16, z.EPI_SWIGLU)
        g, u = An @ _np(Wg).T, An @ _np(Wu).T
        ref = O.bf16_round(O.silu(g) * u)
        tol = 1.1 * np.abs(u) * accum_bound(An, _np(Wg)) + np.abs(O.silu(g)) * accum_bound(An, _np(Wu))
    else:
        N = 2048
        W = _rand((N, K), 55, 0.02)
        acc = An @ _np(W).T
        tol = accum_bound(An, _np(W))
        if epi == "resid":
            H = _rand((M, N), 56)
            h0 = _np(H)
            z.zsaa_op_linear(A, W, None, H, H, M, N, K, z.ZSAA_BF16, z.EPI_RESID)
            out, ref = H, O.bf16_round(h0 + acc)
        elif epi == "store":
            out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
            z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE)
            ref = O.bf16_round(acc)
        else:
            out = torch.empty(M, N, device="cuda", dtype=torch.float32)
            z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
            ref = acc
    torch.cuda.synchronize()
    z.zsaa_device_status()
    got = _np(out)
    if epi == "store_f32":
        assert np.all(np.abs(got - ref) <= tol + 1e-6 * np.abs(ref))
    else:
        assert np.all(bf16_ulp_close(got, ref, 2, tol)), epi
        assert np.mean(bf16_ulp_close(got, ref, 1)) > 0.995, epi


@pytest.mark.parametrize("epi", ["store", "resid", "swiglu"])
def test_linear_f32(z, epi):
    M, N, K = 77, 130, 96
    A = _rand((M, K), 13, dtype=torch.float32)
    W = _rand((N, K), 14, dtype=torch.float32)
    W2 = _rand((N, K), 15, dtype=torch.float32)
    H = _rand((M, N), 16, dtype=torch.float32)
    h0 = _np(H)
    e = {"store": z.EPI_STORE, "resid": z.EPI_RESID, "swiglu": z.EPI_SWIGLU}[epi]
    out = H if epi == "resid" else torch.empty(M, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_linear(A, W, W2 if epi == "swiglu" else None, H if epi == "resid" else None, out,
                     M, N, K, z.ZSAA_F32, e)
    torch.cuda.synchronize()
    acc = _np(A) @ _np(W).T
    u = _np(A) @ _np(W2).T
    ref = {"store": acc, "resid": h0 + acc, "swiglu": O.silu(acc) * u}[epi]
    b = accum_bound(_np(A), _np(W))
    tol = {"store": b, "resid": b, "swiglu": 1.1 * np.abs(u) * b
           + np.abs(O.silu(acc)) * accum_bound(_np(A), _np(W2))}[epi]
    assert np.all(np.abs(_np(out) - ref) <= tol + 2e-7 * np.abs(ref))


def _qkv(B, N, Hq, Hkv, hd, seed, dtype):
    return _rand((B * N, (Hq + 2 * Hkv) * hd), seed, 1.0, dtype)


def _oracle_attention(qkv, B, N, Hq, Hkv, hd, causal=True):
    x = _np(qkv).reshape(B, N, Hq + 2 * Hkv, hd)
    per = Hq // Hkv
    outs, lses, Ps = [], [], []
    for b in range(B):
        q, k, v = x[b, :, :Hq], x[b, :, Hq:Hq + Hkv], x[b, :, Hq + Hkv:]
        o = np.empty((N, Hq, hd))
        P = np.empty((Hq, N, N))
        lse = np.empty((Hq, N))
        for h in range(Hq):
            g = h // per
            P[h] = O.attention_probs(q[:, h], k[:, g], causal=causal)
            o[:, h] = P[h] @ v[:, g]
            s = (q[:, h] @ k[:, g].T) / math.sqrt(hd)
            if causal:
                s = np.where(np.tril(np.ones((N, N), bool)), s, -np.inf)
            mx = s.max(axis=1)
            lse[h] = (mx + np.log(np.exp(s - mx[:, None]).sum(axis=1))) / math.log(2.0)
        outs.append(o.reshape(N, Hq * hd))
        lses.append(lse)
        Ps.append(P)
    return np.stack(outs), np.stack(lses), Ps, x


# Shapes with an even number of query heads per KV head run the two-tile
# kernel (k_attn_pp.cu) at every length, the short kept lengths of the deep
# pruned layers included (18..255 keys); odd ratios run the one-tile kernel.
@pytest.mark.parametrize("B,N,Hq,Hkv,hd", [(2, 1, 4, 2, 64), (2, 65, 4, 2, 64), (1, 200, 4, 1, 128),
                                           (2, 130, 8, 2, 128), (1, 64, 2, 2, 64), (2, 300, 4, 2, 64),
                                           (1, 517, 8, 2, 64), (1, 1024, 4, 4, 64), (2, 300, 4, 2, 128),
                                           (1, 517, 8, 2, 128), (1, 1024, 4, 4, 128), (3, 63, 2, 1, 128),
                                           (3, 18, 8, 2, 64), (2, 47, 8, 2, 128), (4, 128, 8, 2, 64),
                                           (2, 129, 8, 2, 128), (2, 255, 8, 2, 64), (1, 2048, 8, 2, 128),
                                           (1, 700, 16, 2, 64)])
def test_attention_and_colmass_bf16(z, B, N, Hq, Hkv, hd):
    _check_attention_bf16(z, _qkv(B, N, Hq, Hkv, hd, 20 + N, torch.bfloat16), B, N, Hq, Hkv, hd)


def _growing_scores_qkv(N, Hq, Hkv, hd, seed, rise_log2, wave):
    """qkv rows whose scores q.k/sqrt(hd) climb along the keys by about
    rise_log2 (log2 units) over the sequence, plus a wave of that amplitude
    (wave > 0), so a query's running maximum keeps moving: inside a key block
    by more than 2^8 (rescaling the block's P already written) and from block
    to block (rescaling O)."""
    g = torch.Generator().manual_seed(seed)
    u = torch.randn(hd, generator=g)
    u /= u.norm()
    a = 8.0
    j = torch.arange(N, dtype=torch.float64)
    beta = (rise_log2 / 1.4426950408889634) * math.sqrt(hd) / a
    amp = beta * (j / N + wave * torch.sin(j / 23.0))
    x = 0.05 * torch.randn(N, Hq + 2 * Hkv, hd, generator=g, dtype=torch.float64)
    x[:, :Hq] += a * u.double()
    x[:, Hq:Hq + Hkv] += amp[:, None, None] * u.double()
    return x.reshape(N, -1).to(torch.bfloat16).cuda()


@pytest.mark.parametrize("hd,rise,wave", [(64, 150.0, 0.0), (128, 150.0, 0.0), (64, 60.0, 0.4),
                                          (128, 400.0, 0.3)])
def test_attention_running_max_rescales(z, hd, rise, wave):
    N, Hq, Hkv = 300, 4, 2
    _check_attention_bf16(z, _growing_scores_qkv(N, Hq, Hkv, hd, 7 + hd, rise, wave), 1, N, Hq, Hkv, hd)


def _check_attention_bf16(z, qkv, B, N, Hq, Hkv, hd):
    out = torch.empty(B * N, Hq * hd, device="cuda", dtype=torch.bfloat16)
    lse = torch.empty(B, Hq, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_attention(qkv, B, N, Hq, Hkv, hd, z.ZSAA_BF16, out, lse)
    torch.cuda.synchronize()
    ref_o, ref_lse, Ps, _ = _oracle_attention(qkv, B, N, Hq, Hkv, hd)
    got = _np(out).reshape(B, N, Hq * hd)
    # fp32 softmax with P entering P V as a bf16 hi/lo pair: within one bf16 ulp
    # of the rounded exact output (plus 1e-5 of the row scale), mostly identical
    ref_b = O.bf16_round(ref_o)
    tol = 1e-5 * np.abs(ref_o).max(axis=-1, keepdims=True)
    assert np.all(bf16_ulp_close(got, ref_b, 1, tol))
    assert np.mean(got == ref_b) > 0.95, np.mean(got == ref_b)
    np.testing.assert_allclose(_np(lse), ref_lse, rtol=1e-5, atol=1e-4)
    # column mass from the oracle's lse, so it is checked on its own
    C = torch.empty(B, Hkv, N, device="cuda", dtype=torch.float32)
    lse_in = torch.from_numpy(ref_lse.astype(np.float32)).cuda()
    z.zsaa_op_colmass(qkv, lse_in, B, N, Hq, Hkv, hd, z.ZSAA_BF16, C)
    torch.cuda.synchronize()
    refC = np.stack([O.column_mass(Ps[b], Hkv) for b in range(B)])
    np.testing.assert_allclose(_np(C), refC, rtol=2e-4, atol=1e-5)
    # every query row sums to one: each group's columns total (Hq/Hkv) * N
    np.testing.assert_allclose(_np(C).sum(axis=2), (Hq // Hkv) * N, rtol=1e-4)


@pytest.mark.parametrize("B,N,Hq,Hkv,hd", [(2, 64, 4, 4, 32), (1, 37, 4, 2, 32)])
def test_attention_and_colmass_f32(z, B, N, Hq, Hkv, hd):
    qkv = _qkv(B, N, Hq, Hkv, hd, 40 + N, torch.float32)
    out = torch.empty(B * N, Hq * hd, device="cuda", dtype=torch.float32)
    lse = torch.empty(B, Hq, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_attention(qkv, B, N, Hq, Hkv, hd, z.ZSAA_F32, out, lse)
    torch.cuda.synchronize()
    ref_o, ref_lse, Ps, _ = _oracle_attention(qkv, B, N, Hq, Hkv, hd)
    np.testing.assert_allclose(_np(out).reshape(B, N, Hq * hd), ref_o, rtol=1e-5, atol=1e-5)
    C = torch.empty(B, Hkv, N, device="cuda", dtype=torch.float32)
    z.zsaa_op_colmass(qkv, lse, B, N, Hq, Hkv, hd, z.ZSAA_F32, C)
    torch.cuda.synchronize()
    refC = np.stack([O.column_mass(Ps[b], Hkv) for b in range(B)])
    np.testing.assert_allclose(_np(C), refC, rtol=1e-5, atol=1e-6)
