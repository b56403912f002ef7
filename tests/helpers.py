"""Shared pieces of the GPU parity tests: device checks, oracle configs from
model shapes, and the comparison rules (tolerances are stated here once)."""

import numpy as np
import pytest
import torch

from oracle import zsaa_oracle as O

# bf16 logits tolerance (max-abs / mean-abs) and fp32 relative tolerance of the
# forward pass, as the acceptance criteria state them.
BF16_MAX_ABS = 2e-2
BF16_MEAN_ABS = 2e-3
F32_REL = 1e-4


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")


def oracle_cfg(shape, prune_layers=None, n_layers=None):
    return O.OracleConfig(
        n_layers=shape.n_layers if n_layers is None else n_layers, d_model=shape.d_model,
        n_heads=shape.n_heads, n_kv_heads=shape.n_kv_heads, head_dim=shape.head_dim,
        ffn_dim=shape.ffn_dim, vocab=shape.vocab, n_classes=shape.n_classes,
        rope_theta=shape.rope_theta, rms_eps=shape.rms_eps, dtype=shape.dtype,
        prune_layers=shape.prune_layers() if prune_layers is None else prune_layers,
        plan_mode=shape.plan_mode, causal=not getattr(shape, "bidirectional", False),
        score_mode=getattr(shape, "score_mode", "softscore_vnorm"))


def bf16_ulp_close(got, ref, ulps=1, atol=0.0):
    """|got - ref| within `ulps` bf16 units of the larger magnitude plus atol
    (ref given in float64, already rounded to bf16 by the caller).  atol carries
    the float32 accumulation error of the device, e.g. ``accum_bound``."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    mag = np.maximum(np.abs(got), np.abs(ref))
    ulp = np.where(mag > 0, 2.0 ** (np.floor(np.log2(np.maximum(mag, 1e-38))) - 7), 2.0 ** -133)
    return np.abs(got - ref) <= ulps * ulp + atol + 1e-30


def accum_bound(A, W):
    """Worst-case error of a float32 dot product of length K summed in any
    order: K * 2^-24 * sum_k |a_k w_k| (recursive-summation bound), per output
    element of A[M, K] @ W[N, K]^T."""
    K = A.shape[1]
    return K * 2.0 ** -24 * (np.abs(A) @ np.abs(W).T)


def logits_report(got, ref):
    d = np.abs(np.asarray(got, np.float64) - np.asarray(ref, np.float64))
    return float(d.max()), float(d.mean())
