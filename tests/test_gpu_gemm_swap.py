"""Parity of the swapped-operand tensor-core GEMM (a few hundred rows: weight
band as the 128-row MMA operand, K split over a thread-block cluster, partial
sums added in cluster-rank order) against a float64 matmul of the same bf16
operands, for every epilogue, across the row counts where the path starts and
ends (next to the weight-streaming and the tiled kernels), row blocks, ragged
column bands, and the deep-layer shapes of the pruned Llama-3.2-1B forward."""

import pytest
import torch

from tests.helpers import check_linear, linear_case, need_gpu, rand_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def z(zlib):
    need_gpu()
    return zlib


# 16 rows: weight streaming; 17..: swapped operands (one row block up to 256,
# two from 257); ragged last band (N = 1040 is 8 bands of 128 plus 16 columns).
@pytest.mark.parametrize("M", [16, 17, 40, 144, 256, 257, 600, 1024, 1100])
@pytest.mark.parametrize("epi", ["store", "store_f32", "resid"])
def test_swap_plain_epilogues(z, epi, M):
    out, ref, tol = linear_case(z, epi, M, 1040, 1024, 100 + M)
    check_linear(out, ref, tol, epi, f"{epi} M={M}")


@pytest.mark.parametrize("M", [17, 144, 256, 300, 1024])
def test_swap_swiglu(z, M):
    # 1088 output columns: 17 bands of 64 gate + 64 up rows
    out, ref, tol = linear_case(z, "swiglu", M, 1088, 512, 200 + M)
    check_linear(out, ref, tol, "swiglu", f"M={M}")


@pytest.mark.parametrize("hd,Hq,Hkv", [(64, 4, 2), (128, 2, 1), (64, 3, 2)])
@pytest.mark.parametrize("M", [24, 144, 333])
def test_swap_rope(z, M, hd, Hq, Hkv):
    # (64, 3, 2): 320 rotated columns -- a 128-row band holds rotated and value heads
    N = (Hq + 2 * Hkv) * hd
    out, ref, tol = linear_case(z, "rope", M, N, 768, 300 + M, hd=hd, rope_cols=(Hq + Hkv) * hd)
    check_linear(out, ref, tol, "rope", f"M={M} hd={hd}")


# The deep layers of the pruned 1B forward (accel 4 keeps 144..456 rows of 8
# sequences there): QKV with RoPE, O and down with the residual, gate/up SwiGLU.
DEEP_1B = [("qkv", 144, 3072, 2048), ("o", 232, 2048, 2048), ("gate_up", 144, 8192, 2048),
           ("down", 184, 2048, 8192), ("o", 456, 2048, 2048)]


@pytest.mark.parametrize("name,M,N,K", DEEP_1B)
def test_swap_deep_1b_shapes(z, name, M, N, K):
    epi = {"qkv": "rope", "o": "resid", "gate_up": "swiglu", "down": "resid"}[name]
    out, ref, tol = linear_case(z, epi, M, N, K, 400 + M, hd=64, rope_cols=2560)
    check_linear(out, ref, tol, epi, f"{name} M={M}")


# The 8B projections below their crossovers to the tiled kernel (N, K >= 4096:
# RoPE up to 256 rows, residual up to 512): QKV, O, and down with 14336-deep K.
DEEP_8B = [("rope", 192, 6144, 4096), ("resid", 456, 4096, 4096), ("resid", 300, 4096, 14336)]


@pytest.mark.parametrize("epi,M,N,K", DEEP_8B)
def test_swap_deep_8b_shapes(z, epi, M, N, K):
    kw = dict(hd=128, rope_cols=5120) if epi == "rope" else {}
    out, ref, tol = linear_case(z, epi, M, N, K, 450 + M, **kw)
    check_linear(out, ref, tol, epi, f"{epi} M={M} N={N} K={K}")


def test_swap_deterministic(z):
    # the cluster adds its partial sums in rank order: repeated calls agree bit for bit
    M, N, K = 200, 2048, 4096
    A = rand_bf16((M, K), 7)
    W = rand_bf16((N, K), 8, 0.05)
    outs = []
    for _ in range(3):
        out = torch.empty(M, N, device="cuda", dtype=torch.float32)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
        outs.append(out)
    torch.cuda.synchronize()
    z.zsaa_device_status()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])

