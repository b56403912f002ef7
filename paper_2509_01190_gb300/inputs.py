"""Seeded synthetic inputs shared by the tests, the bench and the oracle checks.

This module only draws random numbers and lays them out; it holds none of the
pruned-prefill arithmetic.  It imports torch (for seeded device generation and
bf16 casting) but nothing from the CUDA library or from the oracle.

Recipes (all seeded):

* weights: every linear and embedding matrix N(0, 0.02), norm weights 1.
  Linear weights are stored ``[out_features, in_features]`` row-major.
* token ids: uniform on [0, vocab) from ``numpy.random.Generator(PCG64(seed))``.
* microbench hidden state: ``N(0, 1) * exp(z)`` with one ``z ~ N(0, 1)`` per
  row (a log-normal per-position scale, sigma = 1), so row norms are well
  separated.
"""

from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional

import numpy as np
import torch

WEIGHT_SEED = 1234
TOKEN_SEED = 42
MICROBENCH_SEED = 7


@dataclasses.dataclass(frozen=True)
class ModelShape:
    """A named decoder shape and the options the library is created with."""

    name: str
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int
    vocab: int
    n_classes: int = 0
    rope_theta: float = 500000.0
    rms_eps: float = 1e-5
    dtype: str = "bf16"
    tie_embeddings: bool = False
    prune: str = "all_but_last"  # or a comma list of 1-based layers, e.g. "1"
    plan_mode: str = "cost"
    bidirectional: bool = False  # encoder variant: Eq. 1 without the causal mask
    score_mode: str = "softscore_vnorm"  # or "softscore" (column mass alone)

    def prune_layers(self) -> List[int]:
        if self.prune == "all_but_last":
            return list(range(1, self.n_layers))
        if self.prune == "none":
            return []
        return [int(x) for x in self.prune.split(",") if x]


# The five workloads: their shapes and batch/sequence sizes.
TINY_F32 = ModelShape("tiny-f32-2L-d128", 2, 128, 4, 4, 32, 512, 1000, rope_theta=10000.0,
                      dtype="f32", prune="1", plan_mode="rate")
LLAMA_1B = ModelShape("llama-3.2-1b-shape", 16, 2048, 32, 8, 64, 8192, 128256,
                      tie_embeddings=True)
LLAMA_1B_CLS = dataclasses.replace(LLAMA_1B, name="llama-3.2-1b-shape-cls4", n_classes=4,
                                   tie_embeddings=False)
LLAMA_8B = ModelShape("llama-3-8b-shape", 32, 4096, 32, 8, 128, 14336, 128256)

WORKLOADS = {
    "tiny": dict(shape=TINY_F32, B=2, L=64, accels=[2.0]),
    "1b": dict(shape=LLAMA_1B, B=8, L=512, accels=[1.0, 2.0, 4.0, 8.0]),
    "1b_cls": dict(shape=LLAMA_1B_CLS, B=64, L=256, accels=[1.0, 3.0, 6.0, 11.0]),
    "8b": dict(shape=LLAMA_8B, B=4, L=2048, accels=[1.0, 2.0, 4.0, 8.0, 11.0]),
    "microbench": dict(B=32, L=4096, d=4096, accels=[1.5, 2.0, 4.0, 8.0, 11.0]),
}


def torch_dtype(shape: ModelShape):
    return torch.bfloat16 if shape.dtype == "bf16" else torch.float32


def make_weights(shape: ModelShape, device="cpu", seed: int = WEIGHT_SEED) -> Dict:
    """Random-init weights of ``shape`` as torch tensors on ``device``.

    Returns ``{"embed", "layers": [ {attn_norm, wq, wk, wv, wo, mlp_norm, wg,
    wu, wd} ], "final_norm", "head"}``; ``head`` is the embedding itself when
    the shape ties them, and ``[n_classes, d]`` for a classifier.
    """
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    dt = torch_dtype(shape)
    d, hd = shape.d_model, shape.head_dim

    def normal(*size):
        t = torch.randn(*size, generator=g, device=device, dtype=torch.float32)
        return (t * 0.02).to(dt)

    def ones(n):
        return torch.ones(n, device=device, dtype=dt)

    embed = normal(shape.vocab, d)
    layers = []
    for _ in range(shape.n_layers):
        layers.append({
            "attn_norm": ones(d),
            "wq": normal(shape.n_heads * hd, d),
            "wk": normal(shape.n_kv_heads * hd, d),
            "wv": normal(shape.n_kv_heads * hd, d),
            "wo": normal(d, shape.n_heads * hd),
            "mlp_norm": ones(d),
            "wg": normal(shape.ffn_dim, d),
            "wu": normal(shape.ffn_dim, d),
            "wd": normal(d, shape.ffn_dim),
        })
    if shape.n_classes > 0:
        head = normal(shape.n_classes, d)
    elif shape.tie_embeddings:
        head = embed
    else:
        head = normal(shape.vocab, d)
    return {"embed": embed, "layers": layers, "final_norm": ones(d), "head": head}


def weights_to_numpy(w: Dict, layers: Optional[List[int]] = None) -> Dict:
    """Copy weights to host float32 numpy arrays (bf16 values are exact in f32).

    ``layers`` restricts which layer dicts are copied (others become None)."""

    def cv(t):
        return t.detach().to("cpu", torch.float32).numpy()

    out = {"embed": cv(w["embed"]), "final_norm": cv(w["final_norm"]), "head": cv(w["head"])}
    out["layers"] = [
        ({k: cv(v) for k, v in lw.items()} if layers is None or i in layers else None)
        for i, lw in enumerate(w["layers"])
    ]
    return out


def make_tokens(B: int, L: int, vocab: int, seed: int = TOKEN_SEED) -> np.ndarray:
    """Token ids [B, L] int32, uniform on [0, vocab)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.integers(0, vocab, size=(B, L), dtype=np.int64).astype(np.int32)


def make_hidden(B: int, L: int, d: int, seed: int = MICROBENCH_SEED, device="cpu",
                dtype=torch.bfloat16) -> torch.Tensor:
    """Hidden state [B, L, d]: N(0, 1) times a per-row log-normal scale exp(z)."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    z = torch.randn(B, L, 1, generator=g, device=device, dtype=torch.float32)
    x = torch.randn(B, L, d, generator=g, device=device, dtype=torch.float32)
    return (x * torch.exp(z)).to(dtype)


def make_positions(B: int, N: int, L: int, seed: int) -> np.ndarray:
    """Original positions [B, N] int32 of N rows kept out of L, as a compaction
    leaves them: per sequence a sorted uniform sample of [0, L) without
    repeats that always holds the last position L - 1."""
    rng = np.random.Generator(np.random.PCG64(seed))
    out = np.empty((B, N), dtype=np.int32)
    for b in range(B):
        rest = rng.choice(L - 1, size=N - 1, replace=False) if N > 1 else np.zeros(0, np.int64)
        out[b] = np.sort(np.append(rest, L - 1))
    return out
