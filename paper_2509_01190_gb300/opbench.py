"""Time one operator of the pruned prefill path in isolation.

Used for single-kernel profiler captures: each run does ``--warmup`` launches,
synchronises, then ``--iters`` launches timed with CUDA events on the current
stream, and prints the mean time with the algorithmic rate.

    python -m paper_2509_01190_gb300.opbench gemm gate_up --model 1b --rows 4096
    python -m paper_2509_01190_gb300.opbench gemm o --model 1b --rows 144 --graph --cold-weights
    python -m paper_2509_01190_gb300.opbench attention --model 1b --batch 8 --seq 512
    python -m paper_2509_01190_gb300.opbench colmass --model 1b --batch 8 --seq 512
    python -m paper_2509_01190_gb300.opbench score_select --batch 32 --seq 4096 --dim 4096 --accel 4

GEMM names follow the layer: qkv (RoPE epilogue), o (residual), gate_up
(SwiGLU), down (residual), lm_head (float32 logits).
"""
from __future__ import annotations

import argparse

import torch

from . import zsaa as z
from .inputs import LLAMA_1B, LLAMA_8B

SHAPES = {"1b": LLAMA_1B, "8b": LLAMA_8B}


def _time(fn, warmup: int, iters: int, graph: bool = False) -> float:
    """Mean microseconds per call.  With graph=True the iters calls are captured
    in one CUDA graph and the replay is timed, so host-side launch cost (ctypes
    marshalling, tensor-map encoding) is left out as it is in the forward."""
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    z.zsaa_device_status()
    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(iters):
                fn()
        g.replay()
        torch.cuda.synchronize()
        run = g.replay
    else:
        def run():
            for _ in range(iters):
                fn()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    run()
    e1.record()
    torch.cuda.synchronize()
    z.zsaa_device_status()
    return 1e3 * e0.elapsed_time(e1) / iters


def main(argv=None) -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("op", choices=["gemm", "attention", "colmass", "score_select"])
    ap.add_argument("which", nargs="?", default="gate_up",
                    choices=["qkv", "o", "gate_up", "down", "lm_head"])
    ap.add_argument("--model", default="1b", choices=sorted(SHAPES))
    ap.add_argument("--rows", type=int, default=4096, help="GEMM rows M (kept positions x batch)")
    ap.add_argument("--batch", type=int, default=8)
    ap.add_argument("--seq", type=int, default=512)
    ap.add_argument("--dim", type=int, default=4096)
    ap.add_argument("--accel", type=float, default=4.0)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--iters", type=int, default=10)
    ap.add_argument("--graph", action="store_true", help="time a CUDA-graph replay of the iters calls")
    ap.add_argument("--cold-weights", action="store_true",
                    help="gemm: cycle through enough weight copies (> 320 MB) that weights come from HBM")
    a = ap.parse_args(argv)
    dev = "cuda"
    g = torch.Generator(device=dev).manual_seed(0)
    bf = torch.bfloat16
    sh = SHAPES[a.model]
    d, hd, Hq, Hkv = sh.d_model, sh.head_dim, sh.n_heads, sh.n_kv_heads

    if a.op == "gemm":
        M = a.rows
        qkv_n = (Hq + 2 * Hkv) * hd
        N, K, epi = {"qkv": (qkv_n, d, z.EPI_ROPE), "o": (d, Hq * hd, z.EPI_RESID),
                     "gate_up": (sh.ffn_dim, d, z.EPI_SWIGLU), "down": (d, sh.ffn_dim, z.EPI_RESID),
                     "lm_head": (sh.vocab, d, z.EPI_STORE_F32)}[a.which]
        A = torch.randn(M, K, device=dev, generator=g).to(bf)
        n_w = 2 if epi == z.EPI_SWIGLU else 1
        copies = max(1, -(-320 * 2 ** 20 // (n_w * N * K * 2))) if a.cold_weights else 1
        Ws = [(torch.randn(N, K, device=dev, generator=g) * 0.02).to(bf) for _ in range(copies)]
        W2s = [(torch.randn(N, K, device=dev, generator=g) * 0.02).to(bf) if epi == z.EPI_SWIGLU else None
               for _ in range(copies)]
        turn = [0]

        def weights():
            i = turn[0] % copies
            turn[0] += 1
            return Ws[i], W2s[i]
        out = torch.zeros(M, N, device=dev, dtype=torch.float32 if epi == z.EPI_STORE_F32 else bf)
        pos = torch.arange(M, device=dev, dtype=torch.int32) % a.seq if epi == z.EPI_ROPE else None
        resid = out if epi == z.EPI_RESID else None
        rope = dict(pos=pos, rope_cols=(Hq + Hkv) * hd, rope_hd=hd, rope_theta=sh.rope_theta) \
            if epi == z.EPI_ROPE else {}
        us = _time(lambda: z.zsaa_op_linear(A, *weights(), resid, out, M, N, K, z.ZSAA_BF16, epi, **rope),
                   a.warmup, a.iters, a.graph)
        n_eff = 2 * N if epi == z.EPI_SWIGLU else N
        print(f"gemm {a.which} M={M} N={N} K={K}: {us:.1f} us, {2.0 * M * n_eff * K / us / 1e6:.0f} TFLOP/s")
    elif a.op in ("attention", "colmass"):
        B, N = a.batch, a.seq
        qkv = torch.randn(B * N, (Hq + 2 * Hkv) * hd, device=dev, generator=g).to(bf)
        out = torch.empty(B * N, Hq * hd, device=dev, dtype=bf)
        lse = torch.empty(B, Hq, N, device=dev)
        C = torch.empty(B, Hkv, N, device=dev)
        z.zsaa_op_attention(qkv, B, N, Hq, Hkv, hd, z.ZSAA_BF16, out, lse)
        if a.op == "attention":
            us = _time(lambda: z.zsaa_op_attention(qkv, B, N, Hq, Hkv, hd, z.ZSAA_BF16, out, lse),
                       a.warmup, a.iters, a.graph)
        else:
            us = _time(lambda: z.zsaa_op_colmass(qkv, lse, B, N, Hq, Hkv, hd, z.ZSAA_BF16, C),
                       a.warmup, a.iters, a.graph)
        # causal: N(N+1)/2 query-key pairs per head; QK^T and PV are 2*hd flops each
        mult = 4 if a.op == "attention" else 2
        flops = mult * B * Hq * hd * N * (N + 1) / 2
        print(f"{a.op} B={B} N={N} Hq={Hq} Hkv={Hkv} hd={hd}: {us:.1f} us, {flops / us / 1e6:.1f} TFLOP/s")
    else:
        B, L, dd = a.batch, a.seq, a.dim
        k = int(L // a.accel)
        hidden = torch.randn(B, L, dd, device=dev, generator=g).to(bf)
        idx = torch.empty(B, k, device=dev, dtype=torch.int32)
        rows = torch.empty(B, k, dd, device=dev, dtype=bf)
        us = _time(lambda: z.zsaa_score_select(hidden, B, L, dd, k, idx, rows), a.warmup, a.iters, a.graph)
        nbytes = 2.0 * B * L * dd + 2.0 * B * k * dd
        print(f"score_select B={B} L={L} d={dd} k={k}: {us:.1f} us, {nbytes / us / 1e3:.0f} GB/s")


if __name__ == "__main__":
    main()
