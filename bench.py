#!/usr/bin/env python
"""Benchmark of the pruned prefill (Zero-Shot Adjustable Acceleration) on GB300.

Headline workload: the Llama-3-8B-shaped decoder (32 layers, d=4096, 32/8
heads of 128, SwiGLU 14336, vocab 128256), bf16, random-init N(0, 0.02)
weights, batch 4 x 2048 uniform random tokens -- the largest of the model
workloads, and one GPU holds it.  One step = one pruned prefill of the whole
batch at the headline acceleration factor (--accel, default 4): every row of
the path (plan, embed, per layer RMSNorm / QKV+RoPE / attention / O+residual
/ column mass / score / top-k / gather + RMSNorm / SwiGLU MLP + residual,
then the LM head on the kept rows).

Prints ONE JSON line (rank 0).  value = prefill tokens/s (B*L input tokens per
forward, all ranks) timed with CUDA events on the launch stream, L2 flushed
(256 MiB write) between timed steps.  The other keys: the roofline of the
dominant kernel class and every GEMM class against its own bound (from the
library's per-kernel trace), the end-to-end rate through zsaa_forward_host
with pinned host buffers, the CPU oracle on the host cores, SM clocks during
the timed region, and (last on the line, short) the accel sweep with the
speedup over the same library's unpruned forward, the isolated
score/select/gather microbench and the sweeps of the 1B workloads.

--impl reference times the CPU oracle (the reference arm for this build) on a
bounded sample of the same workload: the oracle's forward of the first
sequence, one decoder layer per step (the head with the last layer), rated by
the modelled FLOPs of the layers it ran.
Multi-GPU (torchrun): every rank runs its own batch (sequences are
independent; no collective on the data path), value = all ranks' tokens /
max over ranks of the timed span.
"""

from __future__ import annotations

import argparse

import numpy as np
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# DRAM bytes per launch from single-launch ncu captures (dram__bytes_read.sum +
# dram__bytes_write.sum, profiles/), keyed by (kernel class, workload): the
# launch captured, its bytes, and the sha256 of the sources it was measured
# on.  Reported only while those sources are unchanged, else null.
TRAFFIC = {
    # profiles/gemm_gate_up_swiglu_8b_traffic.md: the first layer's MLP at accel 4
    ("gemm_gate_up_swiglu", "8b"): {
        "launch": "gate/up + SwiGLU, M=7272 rows (layer 1 of the accel-4 forward), N=2x14336, K=4096",
        "bytes": 1343622912.0,
        "algorithmic_bytes": 502956032.0,
        "sources": {
            "paper_2509_01190_gb300/csrc/k_gemm_tc.cu": "476652139b6316266382a408d78f0d679ecabad54bb26d64f2f15e01a1c5d7f0",
            "paper_2509_01190_gb300/csrc/common.cuh": "9e474368fc0200765d2891a8fa691189a035962da12ffe00a8ef80d040644cbf",
            "paper_2509_01190_gb300/csrc/kernels.h": "c895255d48b1cd8b7810c67d6c8082cc110807e30ffdb7a90ddc0a9faca5635b",
        },
    },
}


def measured_traffic(kernel_name, workload):
    """The ncu-measured DRAM bytes of one launch of `kernel_name`, or None."""
    import hashlib
    rec = TRAFFIC.get((kernel_name, workload))
    if rec is None:
        return None
    for rel, digest in rec["sources"].items():
        try:
            with open(os.path.join(ROOT, rel), "rb") as f:
                if hashlib.sha256(f.read()).hexdigest() != digest:
                    return None
        except OSError:
            return None
    return {"bytes": rec["bytes"], "launch": rec["launch"], "algorithmic_bytes": rec["algorithmic_bytes"]}


def _tensors(obj):
    """Every tensor in a nest of dicts, lists and tuples."""
    import torch
    if isinstance(obj, torch.Tensor):
        yield obj
    elif isinstance(obj, dict):
        for v in obj.values():
            yield from _tensors(v)
    elif isinstance(obj, (list, tuple)):
        for v in obj:
            yield from _tensors(v)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    except OSError:
        return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle samples every 200 ms while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-f", self.path], stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            with open(self.path) as f:
                for line in f:
                    parts = [x.strip() for x in line.split(",")]
                    if len(parts) >= 9:
                        rows.append(parts)
        except OSError:
            pass
        finally:
            try:
                os.unlink(self.path)
            except OSError:
                pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        smax = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = [n for i, n in enumerate(names) if any(r[5 + i].lower() == "active" for r in rows)]
        power = [num(r[3]) for r in rows if num(r[3]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(power) if power else None}


def oracle_config(shape):
    from oracle import zsaa_oracle as O
    return O.OracleConfig(
        n_layers=shape.n_layers, d_model=shape.d_model, n_heads=shape.n_heads,
        n_kv_heads=shape.n_kv_heads, head_dim=shape.head_dim, ffn_dim=shape.ffn_dim,
        vocab=shape.vocab, n_classes=shape.n_classes, rope_theta=shape.rope_theta,
        rms_eps=shape.rms_eps, dtype=shape.dtype, prune_layers=shape.prune_layers(),
        plan_mode=shape.plan_mode)


def cpu_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return os.cpu_count()


class OracleStepper:
    """The oracle's pruned prefill of one sequence after another, one decoder
    layer per step (the head runs with the last layer), for the CPU baseline
    and the reference arm.  A step's work is the modelled FLOPs of what it ran
    (the planner's cost model, R5), so the rate in tokens/s is
    L * (modelled work done / modelled work of one sequence) / seconds."""

    def __init__(self, shape, weights_np, tokens, accel):
        from oracle import zsaa_oracle as O
        self.O = O
        self.cfg = oracle_config(shape)
        self.w = weights_np
        self.tokens = tokens
        self.L = tokens.shape[1]
        self.alpha, self.sched = O.plan(self.cfg, self.L, accel)
        self.total = O.model_cost(self.cfg, self.sched)
        f = O.layer_flops_per_row(self.cfg)
        dq = self.cfg.n_heads * self.cfg.head_dim
        self.layer_cost = [n * f + 2 * n * n * dq for n in self.sched[:-1]]
        self.head_cost = self.total - sum(self.layer_cost)
        self.store = O._Store(self.cfg.dtype)
        self.seq = 0
        self.layer = 0
        self.h = self.pos = None

    def step(self):
        """Runs one layer; returns its modelled FLOPs."""
        O = self.O
        if self.layer == 0:
            t = self.tokens[self.seq % len(self.tokens)]
            self.h = self.store(O._as64(self.w["embed"])[t])
            self.pos = np.arange(self.L)
        l = self.layer + 1
        self.h, self.pos, _, _ = O.decoder_layer(self.cfg, self.w["layers"][l - 1], l, self.h, self.pos,
                                                 self.sched[l], self.store)
        cost = self.layer_cost[self.layer]
        self.layer += 1
        if self.layer == self.cfg.n_layers:
            O.head(self.cfg, self.w, self.h, self.store)
            cost += self.head_cost
            self.layer = 0
            self.seq += 1
        return cost

    def tokens_per_s(self, work, seconds):
        return self.L * (work / self.total) / seconds


VARLEN_LENGTHS = [128, 256, 384, 512, 640, 768, 896, 512]  # 4096 tokens, 8 sequences


def varlen_leg(zsaa, weights, cfg, shape, accel, flush, stream, max_over_ranks, world, steps):
    """zsaa_forward_varlen on 8 sequences of 128..896 tokens (4096 in all, the
    headline's token count), against the fixed-length forward of the same batch
    padded to the longest sequence (B=8, L=896: the cost of padding; its
    outputs are not those of the unpadded sequences).  A model made for
    max_L=896 on the same weights; CUDA events on the launch stream, L2 flushed
    between steps; the variable-length forward launches eagerly."""
    import numpy as np
    import torch
    from paper_2509_01190_gb300 import inputs as I
    lengths = VARLEN_LENGTHS
    T, B, Lp = sum(lengths), len(lengths), max(lengths)
    dev = flush.device
    model = zsaa.Model(cfg, weights, B, Lp)
    toks = I.make_tokens(B, Lp, shape.vocab, seed=11)
    packed = torch.from_numpy(np.concatenate([toks[b, :L] for b, L in enumerate(lengths)])).to(dev)
    padded = torch.from_numpy(toks).to(dev)
    sched, alpha = zsaa.zsaa_plan_varlen(model, lengths, accel)
    n_fin = sum(sc[-1] for sc in sched)
    lg_v = torch.empty(n_fin, shape.vocab, device=dev, dtype=torch.float32)
    psched, _ = zsaa.zsaa_plan(model, Lp, accel)
    lg_p = torch.empty(B, psched[-1], shape.vocab, device=dev, dtype=torch.float32)

    def timed(fn):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(steps)]
        for e0, e1 in evs:
            flush.zero_()
            e0.record(stream)
            fn()
            e1.record(stream)
        torch.cuda.synchronize()
        zsaa.zsaa_sync(model)
        return max_over_ranks(sum(a.elapsed_time(b) for a, b in evs) / steps)

    ms_v = timed(lambda: zsaa.zsaa_forward_varlen(model, packed, lengths, accel, lg_v, stream=stream))
    ms_p = timed(lambda: zsaa.zsaa_forward(model, padded, B, Lp, accel, lg_p, None, stream=stream))
    model.close()
    return {"lengths": lengths, "accel": accel, "alpha": alpha, "final_rows": n_fin,
            "ms_per_step": ms_v, "tokens_per_s": world * T / (ms_v / 1e3),
            "padded_ms_per_step": ms_p, "padded_real_tokens_per_s": world * T / (ms_p / 1e3),
            "speedup_vs_padded": ms_p / ms_v,
            "note": "packed rows, one alpha for the batch (zsaa_plan_varlen); eager launches"}


def decode_leg(zsaa, model, weights, shape, B, L, accel, tok_dev, stream, barrier, max_over_ranks,
               world, steps=48, warmup=8):
    """Decode steps after a pruned prefill (CUDA-graph replay, events on the
    launch stream), the same with an unpruned cache, and the weight-streaming
    roofline of a step: every weight is read once per step (2.5 GB > L2, no
    flush needed) plus the cached keys/values the step attends to."""
    import torch
    peaks, src = load_peaks()
    hbm = peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
    seen, wbytes = set(), 0
    for t in [weights["embed"], weights["final_norm"], weights["head"]] + \
            [v for lw in weights["layers"] for v in lw.values()]:
        if t.data_ptr() not in seen:
            seen.add(t.data_ptr())
            wbytes += t.numel() * t.element_size()
    wbytes -= weights["embed"].numel() * weights["embed"].element_size() \
        if weights["embed"].data_ptr() != weights["head"].data_ptr() else 0  # only B embedding rows are read
    g = torch.Generator(device=tok_dev.device).manual_seed(5)
    new_tok = torch.randint(0, shape.vocab, (steps + warmup, B), generator=g, device=tok_dev.device,
                            dtype=torch.int32)
    out = {}
    for name, a in (("pruned", accel), ("unpruned", 1.0)):
        cache = zsaa.Cache(model, B, L, a, steps + warmup)
        sched, _ = zsaa.zsaa_plan(model, L, a)
        logits = torch.empty(B, shape.vocab, device=tok_dev.device, dtype=torch.float32)
        step_tok = torch.empty(B, device=tok_dev.device, dtype=torch.int32)
        zsaa.zsaa_prefill(model, cache, tok_dev, logits)
        for t in range(warmup):
            step_tok.copy_(new_tok[t])
            zsaa.zsaa_decode_step(model, cache, step_tok, logits, stream=stream)
        barrier()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for t, (e0, e1) in enumerate(evs):
            step_tok.copy_(new_tok[warmup + t])
            e0.record(stream)
            zsaa.zsaa_decode_step(model, cache, step_tok, logits, stream=stream)
            e1.record(stream)
        torch.cuda.synchronize()
        zsaa.zsaa_sync(model)
        ms = max_over_ranks(sum(e0.elapsed_time(e1) for e0, e1 in evs) / steps)
        kv_rows = sum(sched[:-1]) + shape.n_layers * (warmup + steps / 2.0)  # mean rows attended
        kv_read = 2.0 * B * shape.n_kv_heads * shape.head_dim * 2 * kv_rows
        nbytes = wbytes + kv_read
        pruned_b, full_b = zsaa.zsaa_cache_bytes(cache)
        out[name] = {"accel": a, "ms_per_step": ms, "tokens_per_s": world * B / (ms / 1e3),
                     "algorithmic_bytes_per_step": nbytes, "gbs": nbytes / (ms * 1e6),
                     "frac_of_hbm": nbytes / (ms * 1e6) / hbm, "kv_cache_bytes": pruned_b,
                     "kv_cache_bytes_unpruned": full_b}
        cache.close()
    out["workload"] = (f"{steps} timed decode steps (after {warmup}) of B={B} sequences after a "
                       f"prefill of L={L}; teacher-forced random token ids")
    out["peak_gbs"] = hbm
    out["peak_source"] = f"{src} hbm_gbs"
    out["speedup_vs_unpruned_cache"] = out["unpruned"]["ms_per_step"] / out["pruned"]["ms_per_step"]
    return out


def r4(x):
    """x to 4 significant digits (short JSON)."""
    return None if x is None else float(f"{x:.4g}")


def gemm_class_bounds(shape, B, sched, peak_tflops, hbm_gbs):
    """Per GEMM class of one pruned forward: the modelled FLOPs and the bound
    sum over its launches of max(FLOPs / tensor peak, bytes / HBM bandwidth),
    with each launch's rows from the schedule (QKV and O-projection on the
    N_{l-1} rows a layer starts with; the MLP on the N_l rows kept before it;
    the LM head on the final rows).  Bytes as the library's trace counts them:
    activations in, weights, outputs (and the residual read)."""
    d, F, V = shape.d_model, shape.ffn_dim, shape.vocab
    dq = shape.n_heads * shape.head_dim
    qkv = dq + 2 * shape.n_kv_heads * shape.head_dim
    out = {}

    def add(name, flops, nbytes):
        t = max(flops / (peak_tflops * 1e12), nbytes / (hbm_gbs * 1e9))
        c = out.setdefault(name, {"flops": 0.0, "bound_ms": 0.0, "launches": 0})
        c["flops"] += flops
        c["bound_ms"] += 1e3 * t
        c["launches"] += 1

    for l in range(1, shape.n_layers + 1):
        M, Mm = B * sched[l - 1], B * sched[l]
        add("gemm_qkv_rope", 2.0 * M * qkv * d, 2.0 * (M * d + qkv * d + M * qkv))
        add("gemm_o_resid", 2.0 * M * d * dq, 2.0 * (M * dq + d * dq + 2 * M * d))
        add("gemm_gate_up_swiglu", 4.0 * Mm * F * d, 2.0 * (Mm * d + 2 * F * d + Mm * F))
        add("gemm_down_resid", 2.0 * Mm * d * F, 2.0 * (Mm * F + F * d + 2 * Mm * d))
    if not shape.n_classes:
        M = B * sched[-1]
        add("gemm_lm_head", 2.0 * M * V * d, 2.0 * (M * d + V * d) + 4.0 * M * V)
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="8b", choices=["1b", "1b_cls", "8b"])
    ap.add_argument("--accel", type=float, default=4.0)
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--no-extras", action="store_true", help="headline timing only")
    args = ap.parse_args()

    import numpy as np
    import torch

    from paper_2509_01190_gb300 import inputs as I

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    wl = I.WORKLOADS[args.workload]
    shape, B, L = wl["shape"], wl["B"], wl["L"]
    workload_name = f"{shape.name} B={B} L={L} accel={args.accel:g}"
    config = {"workload": workload_name, "model": shape.name, "global_batch": B * world, "seq_len": L,
              "accel": args.accel, "parallelism": f"replicas x{world} (independent sequences, no collective)",
              "l2": "flushed between timed steps (256 MiB write); weights exceed L2"}

    if args.impl == "reference":
        # reference arm: the CPU oracle, one decoder layer per step, rank 0 only
        if rank != 0:
            return
        weights = I.make_weights(shape, device="cpu")
        wnp = I.weights_to_numpy(weights)
        del weights
        tokens = I.make_tokens(B, L, shape.vocab)
        st = OracleStepper(shape, wnp, tokens, args.accel)
        for _ in range(args.warmup):
            st.step()
        work, secs = 0.0, 0.0
        for _ in range(args.steps):
            t0 = time.perf_counter()
            work += st.step()
            secs += time.perf_counter() - t0
        val = st.tokens_per_s(work, secs)
        cfg = dict(config)
        cfg["alpha"] = st.alpha
        line = {"impl": "reference", "metric": "prefill_tokens_per_s", "value": val, "unit": "tokens/s",
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": 1e3 * secs / args.steps, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded N(0,0.02) weights, uniform token ids)",
                "config": cfg,
                "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": cpu_threads(), "kind": "oracle",
                                 "sample": f"float64 NumPy oracle, sequence 0 of the batch, one decoder layer per "
                                           f"step ({args.warmup} untimed, then layers {args.warmup + 1}.. of the "
                                           f"chain), rated by modelled FLOPs: {work / st.total:.3f} of a "
                                           f"sequence in {secs:.1f} s"},
                "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    from paper_2509_01190_gb300 import replicas as R
    from paper_2509_01190_gb300 import zsaa

    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", init_method="env://")
    else:
        dist = None
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())
    stream = torch.cuda.current_stream()
    peaks, peak_src = load_peaks()
    hbm = peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
    sust = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    SPEC_TFLOPS, SPEC_GBS = 2250.0, 8000.0  # nominal dense bf16 and HBM3e rates, for context

    def barrier():
        R.barrier(dist, torch.cuda.synchronize)

    def max_over_ranks(x):
        return R.max_over_ranks(x, dist, dev)

    flush = torch.empty(256 * 1024 * 1024 // 4, device=dev, dtype=torch.float32)

    class Workload:
        def __init__(self, name):
            w = I.WORKLOADS[name]
            self.name, self.shape, self.B, self.L, self.accels = name, w["shape"], w["B"], w["L"], w["accels"]
            self.weights = I.make_weights(self.shape, device=dev)
            self.tokens = I.make_tokens(self.B, self.L, self.shape.vocab,
                                        seed=R.rank_token_seed(I.TOKEN_SEED, rank))
            self.tok_dev = torch.from_numpy(self.tokens).to(dev)
            self.cfg = zsaa.config_from_shape(self.shape)
            self.model = zsaa.Model(self.cfg, self.weights, self.B, self.L)
            n_out = self.B * (self.shape.n_classes if self.shape.n_classes else self.L * self.shape.vocab)
            self.logits = torch.empty(n_out, device=dev, dtype=torch.float32)

        def run(self, accel):
            zsaa.zsaa_forward(self.model, self.tok_dev, self.B, self.L, accel, self.logits, None, stream=stream)

        def timed(self, accel, steps, warmup, sampler=None):
            for _ in range(warmup):
                self.run(accel)
            zsaa.zsaa_sync(self.model)
            barrier()
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(steps)]
            if sampler:
                sampler.__enter__()
            try:
                for a, b in evs:
                    flush.zero_()
                    a.record(stream)
                    self.run(accel)
                    b.record(stream)
                torch.cuda.synchronize()
            finally:
                if sampler:
                    sampler.__exit__(None, None, None)
            zsaa.zsaa_sync(self.model)
            ms = sum(a.elapsed_time(b) for a, b in evs)
            barrier()
            return max_over_ranks(ms) / steps

        def sweep(self, steps, known=None):
            from oracle import zsaa_oracle as O
            ocfg = oracle_config(self.shape)
            sched1, _ = zsaa.zsaa_plan(self.model, self.L, 1.0)
            full = O.model_cost(ocfg, sched1)
            out = {}
            for a in self.accels:
                ms = known[a] if known and a in known else self.timed(a, steps, 3)
                s_a, al = zsaa.zsaa_plan(self.model, self.L, a)
                out[a] = {"ms": ms, "alpha": al, "final_rows": s_a[-1],
                          "flop_red": full / O.model_cost(ocfg, s_a)}
            base = out[1.0]["ms"] if 1.0 in out else None
            for v in out.values():
                v["x"] = base / v["ms"] if base else None
            return out

        def close(self):
            self.model.close()
            del self.weights, self.logits

    main_wl = Workload(args.workload)
    sched, alpha = zsaa.zsaa_plan(main_wl.model, L, args.accel)
    config["alpha"] = alpha
    config["schedule"] = sched

    # ---- headline (plain forwards replay from the library's CUDA graphs)
    sampler = ClockSampler(local) if rank == 0 else None
    ms_head = main_wl.timed(args.accel, args.steps, args.warmup, sampler)
    value = R.job_tokens_per_s(world, B, L, ms_head)
    clocks = sampler.summary() if sampler else None

    line = {"metric": "prefill_tokens_per_s", "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_head, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if shape.dtype == "bf16" else "f32",
            "data": "synthetic (seeded N(0,0.02) weights, uniform token ids)", "config": config,
            "clocks": clocks}
    tail = {}

    if not args.no_extras:
        # ---- accel sweep (speedup over the same library's unpruned forward)
        sw = main_wl.sweep(args.steps, known={args.accel: ms_head})
        # the same headline forward without graph replay (every launch from the host)
        zsaa.zsaa_model_set_graphs(main_wl.model, False)
        line["ms_per_step_eager"] = main_wl.timed(args.accel, args.steps, 3)
        zsaa.zsaa_model_set_graphs(main_wl.model, True)

        # ---- per-kernel trace of the headline forward (separate traced steps)
        zsaa.zsaa_trace_begin(main_wl.model)
        n_tr = 3
        for _ in range(n_tr):
            flush.zero_()
            main_wl.run(args.accel)
        rows = zsaa.zsaa_trace_end(main_wl.model)
        zsaa.zsaa_sync(main_wl.model)
        tot_ms = sum(r["ms"] for r in rows)
        kern = {}
        for r in rows:
            kern[r["name"]] = {"launches": r["launches"] / n_tr, "ms": r4(r["ms"] / n_tr),
                               "share": r4(r["ms"] / tot_ms) if tot_ms else None,
                               "tflops": r4(r["flops"] / (r["ms"] / 1e3) / 1e12) if r["ms"] and r["flops"] else None,
                               "gbs": r4(r["bytes"] / (r["ms"] / 1e3) / 1e9) if r["ms"] else None}
        line["kernels"] = kern
        line["gpu_launches"] = int(sum(r["launches"] for r in rows) // n_tr) * args.steps
        gemms = [r for r in rows if r["name"].startswith("gemm")]
        dom = max(gemms, key=lambda r: r["ms"])
        per_launch = dom["ms"] / dom["launches"]
        ach = dom["flops"] / (dom["ms"] / 1e3) / 1e12
        bounds = gemm_class_bounds(shape, B, sched, sust, hbm)
        tr = measured_traffic(dom["name"], args.workload)
        line["roofline"] = {
            "bound": "tensor", "achieved": ach, "peak": sust, "unit": "TFLOP/s", "frac": ach / sust,
            "traffic": tr["bytes"] if tr else None, "kernel": dom["name"],
            "per_launch_ms": per_launch,
            "peak_source": f"{peak_src} bf16_tflops_sustained (kernel inside a long step)",
            "frac_of_spec_2250": ach / SPEC_TFLOPS,
            "frac_of_own_bound": bounds[dom["name"]]["bound_ms"] * n_tr / dom["ms"]}
        if tr:
            line["roofline"]["traffic_launch"] = tr["launch"]
            line["roofline"]["traffic_algorithmic_bytes"] = tr["algorithmic_bytes"]
        gc = {}
        for r in gemms:
            b_ = bounds.get(r["name"])
            if b_ is None:
                continue
            ms = r["ms"] / n_tr
            gc[r["name"]] = {"ms": r4(ms), "bound_ms": r4(b_["bound_ms"]), "frac_of_bound": r4(b_["bound_ms"] / ms),
                             "tflops": r4(r["flops"] / (r["ms"] / 1e3) / 1e12),
                             "frac_of_sustained": r4(r["flops"] / (r["ms"] / 1e3) / 1e12 / sust)}
        gms = sum(r["ms"] for r in gemms) / n_tr
        gc["all"] = {"ms": r4(gms), "bound_ms": r4(sum(v["bound_ms"] for v in bounds.values())),
                     "tflops": r4(sum(r["flops"] for r in gemms) / n_tr / (gms / 1e3) / 1e12),
                     "share_of_device_time": r4(gms * n_tr / tot_ms)}
        line["gemm_classes"] = {"bound": "per launch max(FLOPs / sustained bf16 peak, bytes / measured HBM)",
                                "by_class": gc}

        # ---- end to end through the host-buffer entry point
        n_fin = sched[-1]
        n_logit = B * (shape.n_classes if shape.n_classes else n_fin * shape.vocab)
        tok_h = torch.from_numpy(main_wl.tokens).pin_memory()
        log_h = torch.empty(n_logit, dtype=torch.float32).pin_memory()
        for _ in range(2):
            zsaa.zsaa_forward_host(main_wl.model, tok_h, B, L, args.accel, log_h, None, stream=stream)
        barrier()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            flush.zero_()
            zsaa.zsaa_forward_host(main_wl.model, tok_h, B, L, args.accel, log_h, None, stream=stream)
        torch.cuda.synchronize()
        e2e_s = max_over_ranks(time.perf_counter() - t0) / args.steps
        line["e2e"] = {"value": world * B * L / e2e_s, "unit": "tokens/s", "h2d_bytes_per_step": B * L * 4,
                       "d2h_bytes_per_step": n_logit * 4, "ms_per_step": e2e_s * 1e3,
                       "note": "zsaa_forward_host: pinned host tokens in, host float32 logits out; "
                               "the 256 MiB L2 flush runs inside this span"}

        # ---- CPU oracle on the host cores (rank 0, N=1 only)
        if rank == 0 and world == 1:
            wnp = I.weights_to_numpy(main_wl.weights)
            st = OracleStepper(shape, wnp, main_wl.tokens, args.accel)
            work, t0 = 0.0, time.perf_counter()
            while True:
                work += st.step()
                if time.perf_counter() - t0 > args.cpu_budget:
                    break
            secs = time.perf_counter() - t0
            line["cpu_baseline"] = {
                "value": st.tokens_per_s(work, secs), "unit": "tokens/s", "cores": cpu_threads(), "kind": "oracle",
                "sample": f"float64 NumPy oracle on sequence 0 at accel {args.accel:g}, layers 1-{st.layer or st.cfg.n_layers}"
                          f" of the chain in {secs:.1f} s ({work / st.total:.3f} of a sequence by modelled FLOPs)"}
            del wnp, st

        # ---- the 1B workloads: sweeps, and on the LM shape decode / varlen / masked mode
        others = {}
        for name in ("1b", "1b_cls"):
            if name == args.workload:
                continue
            ow = Workload(name)
            osw = ow.sweep(max(5, args.steps // 3))
            others[name] = {f"{a:g}": {"ms": r4(v["ms"]), "x": r4(v["x"])} for a, v in osw.items()}
            if name == "1b":
                acc = 4.0
                lg_m = torch.empty_like(ow.logits)

                def run_masked():
                    zsaa.zsaa_forward_masked(ow.model, ow.tok_dev, ow.B, ow.L, acc, lg_m, None, stream=stream)
                for _ in range(3):
                    run_masked()
                torch.cuda.synchronize()
                evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                       for _ in range(10)]
                for e0, e1 in evs:
                    flush.zero_()
                    e0.record(stream)
                    run_masked()
                    e1.record(stream)
                torch.cuda.synchronize()
                zsaa.zsaa_sync(ow.model)
                ms_m = max_over_ranks(sum(a.elapsed_time(b) for a, b in evs) / len(evs))
                line["masked_mode_1b"] = {"accel": acc, "ms_per_step": ms_m, "vs_compacted": ms_m / osw[acc]["ms"],
                                          "note": "zsaa_forward_masked, eager launches"}
                line["varlen_1b"] = varlen_leg(zsaa, ow.weights, ow.cfg, ow.shape, acc, flush, stream,
                                               max_over_ranks, world, 10)
                line["decode_1b"] = decode_leg(zsaa, ow.model, ow.weights, ow.shape, ow.B, ow.L, acc, ow.tok_dev,
                                               stream, barrier, max_over_ranks, world)
            ow.close()
            del ow
            torch.cuda.empty_cache()

        # ---- isolated score + select + compaction on [32, 4096, 4096] bf16 (1 GiB,
        # larger than L2): algorithmic bytes = read every row once + write the
        # kept rows = 2*B*L*d + 2*B*k*d
        mb = I.WORKLOADS["microbench"]
        mB, mL, md = mb["B"], mb["L"], mb["d"]
        hidden = I.make_hidden(mB, mL, md, device=dev)
        micro = {}
        for a in mb["accels"]:
            k = int(mL // a)
            idx = torch.empty(mB, k, device=dev, dtype=torch.int32)
            rws = torch.empty(mB, k, md, device=dev, dtype=torch.bfloat16)
            for _ in range(3):
                zsaa.zsaa_score_select(hidden, mB, mL, md, k, idx, rws, stream=stream)
            torch.cuda.synchronize()
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(10)]
            for e0, e1 in evs:
                flush.zero_()
                e0.record(stream)
                zsaa.zsaa_score_select(hidden, mB, mL, md, k, idx, rws, stream=stream)
                e1.record(stream)
            torch.cuda.synchronize()
            us = 1e3 * sum(e0.elapsed_time(e1) for e0, e1 in evs) / len(evs)
            nbytes = 2.0 * mB * mL * md + 2.0 * mB * k * md
            # the kept rows are read again once the selection is known: at 1 GiB
            # the first pass has long left L2, so that re-read comes from HBM
            moved = nbytes + 2.0 * mB * k * md
            micro[f"{a:g}"] = {"us": r4(us), "gbs": r4(nbytes / (us * 1e3)), "frac": r4(nbytes / (us * 1e3) / hbm),
                               "frac_8tbs": r4(nbytes / (us * 1e3) / SPEC_GBS),
                               "frac_with_reread": r4(moved / (us * 1e3) / hbm)}
            del idx, rws
        del hidden

        # short summaries last on the line
        tail["sweep"] = {f"{a:g}": {"ms": r4(v["ms"]), "tok_s": r4(R.job_tokens_per_s(world, B, L, v["ms"])),
                                    "x": r4(v["x"]), "flop_red": r4(v["flop_red"])} for a, v in sw.items()}
        tail["microbench_score_select"] = {"shape": [mB, mL, md], "peak_gbs": hbm, "by_accel": micro}
        tail["other_workloads"] = others
    if rank == 0:
        line.update(tail)
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
