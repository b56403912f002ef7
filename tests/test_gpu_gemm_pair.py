"""Parity of the CTA-pair tensor-core GEMM (many rows: 256 x 256 tiles on the
2-SM tcgen05 MMA, each CTA of a cluster pair staging half of the A rows and
half of the weight rows) against a float64 matmul of the same bf16 operands,
for every epilogue.  The shapes are ones the routing sends to the pair kernel
on a 152-SM GB300 (two or more waves of whole tiles, pairs saving a wave or
more; the launch list of the forward shows the kernel): odd numbers of 128-row
tiles, so the last pair's second CTA has no rows; ragged columns, so the last
tile's second weight half lies wholly past N; and the large-row projections
of the Llama-3.2-1B forward."""

import pytest
import torch

from tests.helpers import check_linear, linear_case, need_gpu, rand_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def z(zlib):
    need_gpu()
    return zlib


# N = 2064: eight 256-column tiles and 16 columns; 2056 rows: 17 tiles of 128
# (the last pair half empty, its first half 8 rows), 2300: 18 (ragged).
@pytest.mark.parametrize("M", [2056, 2300])
@pytest.mark.parametrize("epi", ["store", "store_f32", "resid"])
def test_pair_plain_epilogues(z, epi, M):
    out, ref, tol = linear_case(z, epi, M, 2064, 512, 600 + M)
    check_linear(out, ref, tol, epi, f"{epi} M={M}")


@pytest.mark.parametrize("M", [2056, 2300])
def test_pair_swiglu(z, M):
    # 1088 outputs: eight tiles of 128 gate + 128 up rows, the ninth 64 + 64
    out, ref, tol = linear_case(z, "swiglu", M, 1088, 512, 700 + M)
    check_linear(out, ref, tol, "swiglu", f"M={M}")


@pytest.mark.parametrize("hd,Hq,Hkv", [(64, 32, 8), (128, 16, 4), (64, 30, 9)])
def test_pair_rope(z, hd, Hq, Hkv):
    # 3072 columns (12 tiles); each CTA's 128 tile columns are whole heads;
    # (64, 30, 9): 2496 rotated columns, so one CTA half holds a rotated key
    # head and a value head
    M = 2300
    N = (Hq + 2 * Hkv) * hd
    out, ref, tol = linear_case(z, "rope", M, N, 512, 800 + hd + Hq, hd=hd, rope_cols=(Hq + Hkv) * hd)
    check_linear(out, ref, tol, "rope", f"hd={hd} Hq={Hq}")


# Layers of the pruned 1B forward on the pair kernel: QKV with RoPE, O and
# down with the residual, gate/up SwiGLU, at kept-row counts of accel 1 and 4
# (288 rows: three 128-row tiles, two pairs).
LARGE_1B = [("qkv", 3296, 3072, 2048), ("o", 4096, 2048, 2048), ("gate_up", 288, 8192, 2048),
            ("gate_up", 3296, 8192, 2048), ("down", 4096, 2048, 8192)]


@pytest.mark.parametrize("name,M,N,K", LARGE_1B)
def test_pair_large_1b_shapes(z, name, M, N, K):
    epi = {"qkv": "rope", "o": "resid", "gate_up": "swiglu", "down": "resid"}[name]
    out, ref, tol = linear_case(z, epi, M, N, K, 900 + M, hd=64, rope_cols=2560)
    check_linear(out, ref, tol, epi, f"{name} M={M}")


def test_pair_deterministic(z):
    M, N, K = 2048, 2048, 2048
    A = rand_bf16((M, K), 17)
    W = rand_bf16((N, K), 18, 0.05)
    outs = []
    for _ in range(3):
        out = torch.empty(M, N, device="cuda", dtype=torch.float32)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
        outs.append(out)
    torch.cuda.synchronize()
    z.zsaa_device_status()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])



# Deep K with two or more waves of pair tiles and a ragged last one: the last
# tiles' k-blocks are split over the pairs (from 40% of the last wave idle at
# 64 k-blocks, 25% at 128 and more).  1204 rows x 4096 columns at K = 4096: 80
# pair tiles (5 x 16), fewer than two waves, so every tile is split, over one
# or two pairs; 2440 x 2048 at K = 8192: 80 pair tiles of 128 k-blocks.
@pytest.mark.parametrize("M,N,K", [(1204, 4096, 4096), (2440, 2048, 8192)])
@pytest.mark.parametrize("epi", ["store_f32", "resid"])
def test_pair_streamk_plain(z, epi, M, N, K):
    out, ref, tol = linear_case(z, epi, M, N, K, 1000 + M + N)
    check_linear(out, ref, tol, epi, f"{epi} M={M} N={N} K={K}")


def test_pair_streamk_swiglu(z):
    out, ref, tol = linear_case(z, "swiglu", 1204, 2048, 4096, 1100)
    check_linear(out, ref, tol, "swiglu", "M=1204 K=4096")


def test_pair_streamk_rope(z):
    # 16 query + 4 key heads rotated, 4 value heads, hd 128: 84 pair tiles (7 x 12)
    out, ref, tol = linear_case(z, "rope", 1700, 3072, 4096, 1200, hd=128, rope_cols=2560)
    check_linear(out, ref, tol, "rope", "hd=128 K=4096")


def test_pair_streamk_down_1b(z):
    # the 1B down projection at 3296 kept rows: 104 pair tiles of 128 k-blocks
    out, ref, tol = linear_case(z, "resid", 3296, 2048, 8192, 1300)
    check_linear(out, ref, tol, "resid", "down M=3296")


# Very deep K (>= 192 k-blocks, like the 8B down projection) with a ragged last
# wave: the remainder tiles are cut into aligned k-parts (3072 rows x 2048
# columns at K = 12288: 96 pair tiles, one whole wave, the last 20 tiles in
# three parts of 64 k-blocks, the third adding the other two's partials).
@pytest.mark.parametrize("epi,N", [("resid", 2048), ("store_f32", 2048), ("swiglu", 1024)])
def test_pair_aligned_tail_split(z, epi, N):
    out, ref, tol = linear_case(z, epi, 3072, N, 12288, 1600 + N)
    check_linear(out, ref, tol, epi, f"{epi} M=3072 N={N} K=12288")


def test_pair_aligned_tail_split_deterministic(z):
    # the partials are added in part order: repeated calls agree bit for bit
    M, N, K = 3072, 2048, 12288
    A = rand_bf16((M, K), 31)
    W = rand_bf16((N, K), 32, 0.05)
    outs = []
    for _ in range(3):
        out = torch.empty(M, N, device="cuda", dtype=torch.float32)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
        outs.append(out)
    torch.cuda.synchronize()
    z.zsaa_device_status()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


# Deep-K plans of the pruned Llama-3.1-8B forward at a few hundred rows, one
# wave each: whole pair tiles (down-like, 48 pair tiles of 128 k-blocks),
# 128-wide one-CTA tiles (QKV + RoPE, hd 128, 144 tiles) and 256-wide one-CTA
# tiles for a single 128-row tile (gate/up + SwiGLU, 112 tiles).
EIGHT_B_TILED = [("resid", 744, 4096, 8192, 64, 0), ("rope", 316, 6144, 4096, 128, 5120),
                 ("swiglu", 92, 14336, 4096, 64, 0)]


@pytest.mark.parametrize("epi,M,N,K,hd,rope_cols", EIGHT_B_TILED)
def test_deep_k_one_wave_plans(z, epi, M, N, K, hd, rope_cols):
    kw = dict(hd=hd, rope_cols=rope_cols) if epi == "rope" else {}
    out, ref, tol = linear_case(z, epi, M, N, K, 1500 + M, **kw)
    check_linear(out, ref, tol, epi, f"{epi} M={M} N={N} K={K}")


def test_pair_streamk_deterministic(z):
    # split tiles add their partials in pair order: repeated calls agree bit for bit
    M, N, K = 1204, 4096, 4096
    A = rand_bf16((M, K), 21)
    W = rand_bf16((N, K), 22, 0.05)
    outs = []
    for _ in range(3):
        out = torch.empty(M, N, device="cuda", dtype=torch.float32)
        z.zsaa_op_linear(A, W, None, None, out, M, N, K, z.ZSAA_BF16, z.EPI_STORE_F32)
        outs.append(out)
    torch.cuda.synchronize()
    z.zsaa_device_status()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


# Very wide float32 outputs (LM heads, N >= 32768) run on the tiled kernel at
# every row count: one CTA or CTA pairs by waves.  40000 columns end in a
# partial tile; 17 and 144 rows leave most of a 256-row pair tile empty.
@pytest.mark.parametrize("M", [17, 144, 300, 600])
def test_tiled_wide_head_f32(z, M):
    out, ref, tol = linear_case(z, "store_f32", M, 40000, 256, 500 + M)
    check_linear(out, ref, tol, "store_f32", f"head M={M}")
