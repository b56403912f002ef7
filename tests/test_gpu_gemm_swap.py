"""Parity of the swapped-operand tensor-core GEMM (a few hundred rows: weight
band as the 128-row MMA operand, K split over a thread-block cluster, partial
sums added in cluster-rank order) against a float64 matmul of the same bf16
operands, for every epilogue, across the row counts where the path starts and
ends (next to the weight-streaming and the tiled kernels), row blocks, ragged
column bands, and the deep-layer shapes of the pruned Llama-3.2-1B forward."""

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


def _rand(shape, seed, scale=1.0):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    return (torch.randn(*shape, generator=g, device="cuda") * scale).to(torch.bfloat16)


def _np(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _run(z, epi, M, N, K, seed, hd=64, rope_cols=0):
    """One GEMM through the C ABI; returns (output, float64 reference, tolerance)."""
    A = _rand((M, K), seed)
    W = _rand((N, K), seed + 1, 0.05)
    An, Wn = _np(A), _np(W)
    tol = accum_bound(An, Wn)
    if epi == "swiglu":
        W2 = _rand((N, K), seed + 2, 0.05)
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        z.zsaa_op_linear(A, W, W2, None, out, M, N, K, z.ZSAA_BF16, z.EPI_SWIGLU)
        g, u = An @ Wn.T, An @ _np(W2).T
        ref = O.bf16_round(O.silu(g) * u)
        tol = 1.1 * np.abs(u) * tol + np.abs(O.silu(g)) * accum_bound(An, _np(W2))
    elif epi == "rope":
        pos = torch.randint(0, 4096, (M,), generator=torch.Generator().manual_seed(seed)).to(torch.int32).cuda()
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_ROPE, pos=pos,
                         rope_cols=rope_cols, rope_hd=hd, rope_theta=500000.0)
        acc = An @ Wn.T
        cos, sin = O.rope_angles(pos.cpu().numpy(), hd, 500000.0)
        qk = O.apply_rope(acc[:, :rope_cols].reshape(M, -1, hd), cos, sin).reshape(M, rope_cols)
        ref = O.bf16_round(np.concatenate([qk, acc[:, rope_cols:]], axis=1))
        tol = 2 * tol.max(axis=1, keepdims=True) + 1e-6 * np.abs(acc)
    elif epi == "resid":
        H = _rand((M, N), seed + 3)
        h0 = _np(H)
        z.zsaa_op_linear(A, W, None, H, H, M, N, K, z.ZSAA_BF16, z.EPI_RESID)
        out, ref = H, O.bf16_round(h0 + An @ Wn.T)
    elif epi == "store_f32":
        out = torch.empty(M, N, device="cuda", dtype=torch.float32)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
        ref = An @ Wn.T
    else:
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE)
        ref = O.bf16_round(An @ Wn.T)
    torch.cuda.synchronize()
    z.zsaa_device_status()
    return out, ref, tol


def _check(out, ref, tol, epi, what):
    got = _np(out)
    if epi == "store_f32":
        assert np.all(np.abs(got - ref) <= tol + 1e-6 * np.abs(ref)), what
    else:
        assert np.all(bf16_ulp_close(got, ref, 2, tol)), what
        assert np.mean(bf16_ulp_close(got, ref, 1)) > 0.995, what


# 16 rows: weight streaming; 17..: swapped operands (one row block up to 256,
# two from 257); ragged last band (N = 1040 is 8 bands of 128 plus 16 columns).
@pytest.mark.parametrize("M", [16, 17, 40, 144, 256, 257, 600, 1024, 1100])
@pytest.mark.parametrize("epi", ["store", "store_f32", "resid"])
def test_swap_plain_epilogues(z, epi, M):
    out, ref, tol = _run(z, epi, M, 1040, 1024, 100 + M)
    _check(out, ref, tol, epi, f"{epi} M={M}")


@pytest.mark.parametrize("M", [17, 144, 256, 300, 1024])
def test_swap_swiglu(z, M):
    # 1088 output columns: 17 bands of 64 gate + 64 up rows
    out, ref, tol = _run(z, "swiglu", M, 1088, 512, 200 + M)
    _check(out, ref, tol, "swiglu", f"M={M}")


@pytest.mark.parametrize("hd,Hq,Hkv", [(64, 4, 2), (128, 2, 1), (64, 3, 2)])
@pytest.mark.parametrize("M", [24, 144, 333])
def test_swap_rope(z, M, hd, Hq, Hkv):
    # (64, 3, 2): 320 rotated columns -- a 128-row band holds rotated and value heads
    N = (Hq + 2 * Hkv) * hd
    out, ref, tol = _run(z, "rope", M, N, 768, 300 + M, hd=hd, rope_cols=(Hq + Hkv) * hd)
    _check(out, ref, tol, "rope", f"M={M} hd={hd}")


# The deep layers of the pruned 1B forward (accel 4 keeps 144..456 rows of 8
# sequences there): QKV with RoPE, O and down with the residual, gate/up SwiGLU.
DEEP_1B = [("qkv", 144, 3072, 2048), ("o", 232, 2048, 2048), ("gate_up", 144, 8192, 2048),
           ("down", 184, 2048, 8192), ("o", 456, 2048, 2048)]


@pytest.mark.parametrize("name,M,N,K", DEEP_1B)
def test_swap_deep_1b_shapes(z, name, M, N, K):
    epi = {"qkv": "rope", "o": "resid", "gate_up": "swiglu", "down": "resid"}[name]
    out, ref, tol = _run(z, epi, M, N, K, 400 + M, hd=64, rope_cols=2560)
    _check(out, ref, tol, epi, f"{name} M={M}")


def test_swap_deterministic(z):
    # the cluster adds its partial sums in rank order: repeated calls agree bit for bit
    M, N, K = 200, 2048, 4096
    A = _rand((M, K), 7)
    W = _rand((N, K), 8, 0.05)
    outs = []
    for _ in range(3):
        out = torch.empty(M, N, device="cuda", dtype=torch.float32)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
        outs.append(out)
    torch.cuda.synchronize()
    z.zsaa_device_status()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


# Very wide float32 outputs (LM heads): several 128-row weight bands per CTA,
# one TMEM accumulator each.  40000 columns end in half a band; 300 and 600
# rows take two and three row blocks (two or three bands per CTA).
@pytest.mark.parametrize("M", [17, 144, 300, 600])
def test_swap_wide_head_f32(z, M):
    out, ref, tol = _run(z, "store_f32", M, 40000, 256, 500 + M)
    _check(out, ref, tol, "store_f32", f"head M={M}")
