"""Parity of the one-CTA tiled GEMM on the shapes that otherwise run on CTA
pairs: its whole-tile path and its stream-K path (deep K, ragged last wave),
the fallback where pairs cannot be scheduled, against the same float64
references as the pair tests.  ZSAA_GEMM_PAIRS=0 is read once per process,
so the cases run in a child process with it set."""

import os
import subprocess
import sys

import pytest

from tests.helpers import check_linear, linear_case, need_gpu

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (epilogue, M, N, K): whole tiles (two waves; 5000 x 2048 at K = 4096: 320
# tiles, a full last wave), then deep K split over the CTAs where the last of
# two or more waves is ragged (1204 rows: 160 tiles of 64 k-blocks; 1700 rows of
# RoPE: 168; the 1B down projection at 3296 rows: 208 tiles of 128 k-blocks),
# and with 192 k-blocks the last wave's tiles cut into aligned k-parts (5760 x
# 1024: 180 tiles, the last 28 in four parts; SwiGLU 3072 x 1024: 40 in three)
CASES = [("store", 2056, 2064, 512), ("swiglu", 2300, 1088, 512), ("rope", 2300, 3072, 512),
         ("store_f32", 1204, 4096, 4096), ("resid", 5000, 2048, 4096), ("swiglu", 1204, 2048, 4096),
         ("rope", 1700, 3072, 4096), ("resid", 3296, 2048, 8192),
         ("resid", 5760, 1024, 12288), ("swiglu", 3072, 1024, 12288)]


def _run_cases():
    from paper_2509_01190_gb300 import zsaa as z
    for i, (epi, M, N, K) in enumerate(CASES):
        out, ref, tol = linear_case(z, epi, M, N, K, 1400 + i, hd=64, rope_cols=2560)
        check_linear(out, ref, tol, epi, f"one CTA {epi} M={M} N={N} K={K}")
        print(f"ok {epi} M={M} N={N} K={K}", flush=True)


def test_one_cta_tiled_paths(zlib):
    need_gpu()
    env = dict(os.environ, ZSAA_GEMM_PAIRS="0")
    r = subprocess.run([sys.executable, "-m", "tests.test_gpu_gemm_one_cta"], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert r.stdout.count("ok ") == len(CASES), r.stdout


if __name__ == "__main__":
    sys.path.insert(0, ROOT)
    _run_cases()
