"""CPU oracle for Zero-Shot Adjustable Acceleration (arXiv 2509.01190).

TEST INFRASTRUCTURE ONLY.  This module is a plain, slow restatement of what the
pruned prefill computes, used to check the CUDA library.  Only the test suite,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it.  It shares no code with the CUDA path and imports nothing from it.

Every function follows one passage of the paper:

* ``attention_probs`` / ``attention_output`` -- Eq. 1 (Sec. 3.2): the soft-score
  ``softmax(QK^T/sqrt(d_k) + M)`` with a causal mask M (or none, for the
  bidirectional-encoder variant), then multiplied by V.
* ``column_mass`` / ``position_scores`` -- Sec. 3.2 and Sec. 3.3: the soft-score
  times V gives each V row's contribution to the layer output; rows with the
  lowest contribution are eliminated from the following layers.
* ``select_topk`` -- Sec. 3.3 (keep the highest-contribution rows).
* ``schedule`` -- Eq. 2 (Sec. 3.3) with tau = 5 (Sec. 4.2).
* ``plan`` -- Sec. 3.4 / Sec. 4.4: the preservation rate is picked at inference
  time, per requested acceleration, without retraining; ``plan_varlen`` picks
  one rate for a batch of different lengths (R17) and ``forward_varlen`` runs it.
* ``forward`` -- Appendix A: a pre-norm decoder (RMSNorm, GQA, RoPE, SwiGLU),
  with the Sec. 3.3 elimination applied after each pruning layer.
* ``forward_masked`` -- Appendix B: the "marked as pruned but not removed"
  formulation, an independent second route to the same kept-row outputs.
* ``forward_marked`` -- Appendix B's figure, where marked rows may be
  reactivated at a later layer (reading R18: nothing is removed or hidden).
* ``decode_step`` / ``generate`` -- Sec. 3.3 carried into generation: a row
  eliminated before layer l is absent from layer l, so a generated token
  attends, in layer l, to the keys and values of the rows that layer kept.

Readings of points the paper leaves open (each is listed in the design notes):

* R1 score: ``s_j = sum_g C[g, j] * ||v_{g, j}||_2`` where ``C[g, j]`` sums the
  soft-score column j over all queries and all query heads of KV group g
  ("softscore_vnorm"); ``"softscore"`` drops the norm factor.
* R2 unnormalised column sums (no division by the number of queries).
* R3 pruning happens after the whole layer: layer l scores its own rows and its
  output rows are compacted; layer l+1 runs on the kept rows.  With
  ``prune_point="attention"`` the compaction happens between attention and
  MLP instead; the kept rows are the same (the MLP acts on each row alone).
* R5 acceleration -> alpha: bisection on the modelled per-sequence FLOPs.
* R6 ``N_l = min(N_{l-1}, max(floor(alpha N_{l-1}), min(tau, N_{l-1})))``.
* R7 ties by lower index; NaN scores rank lowest.
* R8 the last position may be force-kept; it counts toward k.
* R11 bf16 models keep activations in bf16 at fixed storage points (listed in
  ``_Store``); arithmetic between storage points is exact here (float64).
"""

from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence

import numpy as np

# --------------------------------------------------------------------------
# configuration
# --------------------------------------------------------------------------


@dataclasses.dataclass
class OracleConfig:
    """Shape and options of one decoder (Appendix A, Table 1 columns)."""

    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int
    vocab: int
    n_classes: int = 0  # 0 -> language-model head over the vocabulary
    rope_theta: float = 500000.0
    rms_eps: float = 1e-5
    tau: int = 5  # Sec. 4.2: minimum number of preserved activations
    dtype: str = "bf16"  # storage type of activations: "bf16" or "f32"
    prune_layers: Sequence[int] = ()  # 1-based layers whose output is compacted
    force_keep_last: bool = True
    score_mode: str = "softscore_vnorm"  # or "softscore"
    plan_mode: str = "cost"  # "cost" (R5 bisection) or "rate" (alpha = 1/accel)
    # where a pruning layer compacts its rows: "layer" (after the MLP, R3) or
    # "attention" (between attention and MLP; the MLP then runs on kept rows only)
    prune_point: str = "layer"
    # Eq. 1's mask M: causal (decoder) or none (bidirectional encoder)
    causal: bool = True
    # arithmetic between the storage points: "f64" (the oracle proper) or
    # "f32" (a control: the same storage points, float32 sums and products,
    # to measure how far two correct bf16-storage implementations drift apart)
    arith: str = "f64"


# --------------------------------------------------------------------------
# storage rounding (R11)
# --------------------------------------------------------------------------


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 value (ties to even), returned as float64.

    The value is first rounded to float32 (as a device accumulator would hold
    it), then its low 16 bits are rounded away.  NaN stays NaN.
    """
    f = np.asarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + lsb) & np.uint64(0xFFFF0000)).astype(np.uint32)
    out = r.view(np.float32).astype(np.float64)
    return np.where(np.isnan(f), np.nan, out)


class _Store:
    """Where a bf16 model rounds: x (normed), q/k (after RoPE), v, attention
    output, residual after each branch, SwiGLU product, final normed x."""

    def __init__(self, dtype: str):
        if dtype not in ("bf16", "f32"):
            raise ValueError(dtype)
        self.bf16 = dtype == "bf16"

    def __call__(self, x: np.ndarray) -> np.ndarray:
        return bf16_round(x) if self.bf16 else np.asarray(x, dtype=np.float64)


# --------------------------------------------------------------------------
# model pieces (Appendix A: pre-norm decoder; Eq. 1)
# --------------------------------------------------------------------------


def _ft(cfg: "OracleConfig"):
    """numpy type of the arithmetic between storage points (``cfg.arith``)."""
    if cfg.arith == "f64":
        return np.float64
    if cfg.arith == "f32":
        return np.float32
    raise ValueError(cfg.arith)


def rmsnorm(h: np.ndarray, w: np.ndarray, eps: float, ft=np.float64) -> np.ndarray:
    """Root-mean-square normalisation of each row, scaled by w (pre-norm)."""
    h = np.asarray(h, dtype=ft)
    ms = np.mean(h * h, axis=-1, keepdims=True)
    return h / np.sqrt(ms + ft(eps)) * np.asarray(w, dtype=ft)


def rope_angles(pos: np.ndarray, head_dim: int, theta: float):
    """cos/sin of RoPE for original positions pos; frequency i is theta^(-2i/hd)."""
    half = head_dim // 2
    inv = theta ** (-(2.0 * np.arange(half, dtype=np.float64)) / head_dim)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]
    return np.cos(ang), np.sin(ang)


def apply_rope(x: np.ndarray, cos: np.ndarray, sin: np.ndarray) -> np.ndarray:
    """Rotate pairs (c, c + hd/2) of x[n, H, hd] by the angles of each row."""
    half = x.shape[-1] // 2
    x1 = x[..., :half]
    x2 = x[..., half:]
    c = cos[:, None, :].astype(x.dtype)
    s = sin[:, None, :].astype(x.dtype)
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def attention_probs(q: np.ndarray, k: np.ndarray, key_mask: Optional[np.ndarray] = None,
                    causal: bool = True) -> np.ndarray:
    """Soft-score of Eq. 1 for one head: softmax(q k^T / sqrt(d_k) + M).

    q: [n, hd], k: [n, hd].  M is causal (-inf above the diagonal), or zero
    for a bidirectional encoder (``causal=False``); if ``key_mask`` (bool [n])
    is given, keys where it is False are also -inf.
    Returns P [n, n] with rows summing to one.
    """
    n, hd = q.shape
    logits = (q @ k.T) / math.sqrt(hd)
    allowed = np.tril(np.ones((n, n), dtype=bool)) if causal else np.ones((n, n), dtype=bool)
    if key_mask is not None:
        allowed = allowed & key_mask[None, :]
    logits = np.where(allowed, logits, -np.inf)
    m = np.max(logits, axis=1, keepdims=True)
    m = np.where(np.isfinite(m), m, 0.0)
    e = np.where(allowed, np.exp(logits - m), 0.0)
    z = np.sum(e, axis=1, keepdims=True)
    return e / np.where(z > 0, z, 1.0)


def column_mass(P: np.ndarray, n_kv_heads: int) -> np.ndarray:
    """C[g, j] = sum over the query heads h of group g and all queries i of P^h[i, j].

    P: [H, n, n].  Heads are grouped contiguously: head h uses KV head
    h // (H / n_kv_heads).  Unnormalised (R2); the diagonal is included (R10).
    """
    H, n, _ = P.shape
    per = H // n_kv_heads
    col = P.sum(axis=1)  # [H, n]: sum over queries
    return col.reshape(n_kv_heads, per, n).sum(axis=1)


def position_scores(C: np.ndarray, v: np.ndarray, mode: str) -> np.ndarray:
    """Contribution of each position (R1).

    C: [G, n] column mass, v: [n, G, hd].  "softscore_vnorm" weights each
    group's column mass by the norm of that group's value row; "softscore"
    sums the column mass alone.
    """
    if mode == "softscore":
        return C.sum(axis=0)
    if mode != "softscore_vnorm":
        raise ValueError(mode)
    vnorm = np.sqrt(np.sum(np.asarray(v, np.float64) ** 2, axis=-1))  # [n, G]
    return np.sum(C * vnorm.T, axis=0)


def select_topk(scores: np.ndarray, k: int, force_last: bool) -> np.ndarray:
    """Indices of the k highest scores, ascending (Sec. 3.3, R7, R8).

    Ranking is by score descending, then index ascending; NaN ranks below
    every number.  With ``force_last`` the last index is always kept and the
    other k-1 come from the ranking of the rest.
    """
    s = np.asarray(scores, dtype=np.float64)
    n = s.shape[0]
    if not 1 <= k <= n:
        raise ValueError("k out of range")
    cand = list(range(n - 1)) if force_last else list(range(n))
    need = k - 1 if force_last else k

    def rank_key(j):
        x = s[j]
        return (1, 0.0, j) if np.isnan(x) else (0, -x, j)

    chosen = sorted(cand, key=rank_key)[:need]
    if force_last:
        chosen.append(n - 1)
    return np.array(sorted(chosen), dtype=np.int64)


# --------------------------------------------------------------------------
# schedule and planning (Eq. 2, Sec. 3.4)
# --------------------------------------------------------------------------


def schedule(L: int, alpha: float, n_layers: int, prune_layers: Sequence[int], tau: int) -> List[int]:
    """[N_0, ..., N_n] with N_0 = L and Eq. 2 applied after each pruning layer.

    N_l = min(N_{l-1}, max(floor(alpha * N_{l-1}), min(tau, N_{l-1}))) (R6);
    a layer that does not prune passes its count through.
    """
    pl = set(int(x) for x in prune_layers)
    out = [int(L)]
    for layer in range(1, n_layers + 1):
        prev = out[-1]
        if layer in pl:
            nl = max(int(math.floor(alpha * prev)), min(tau, prev))
            out.append(min(prev, nl))
        else:
            out.append(prev)
    return out


def layer_flops_per_row(cfg: OracleConfig) -> int:
    """Multiply-add FLOPs (2 per MAC) of the linear layers for one row of one layer."""
    d, hd = cfg.d_model, cfg.head_dim
    qkv = 2 * d * (cfg.n_heads * hd + 2 * cfg.n_kv_heads * hd)
    o = 2 * cfg.n_heads * hd * d
    mlp = 2 * 3 * d * cfg.ffn_dim
    return qkv + o + mlp


def model_cost(cfg: OracleConfig, sched: Sequence[int]) -> int:
    """Modelled FLOPs of one sequence (R5): linear + causal attention + head."""
    f = layer_flops_per_row(cfg)
    dq = cfg.n_heads * cfg.head_dim
    total = 0
    for layer in range(cfg.n_layers):
        n = sched[layer]
        total += n * f + 2 * n * n * dq
    if cfg.n_classes > 0:
        total += 2 * cfg.d_model * cfg.n_classes
    else:
        total += sched[-1] * 2 * cfg.d_model * cfg.vocab
    return total


def plan(cfg: OracleConfig, L: int, accel: float):
    """Acceleration factor -> (alpha, schedule) (Sec. 3.4, R5).

    "rate": alpha = 1/accel.  "cost": the largest alpha found by 60 bisection
    steps on [0, 1] whose modelled cost is at most cost(alpha=1)/accel.
    """
    if not accel >= 1.0:
        raise ValueError("accel must be >= 1")
    if cfg.plan_mode == "rate":
        alpha = 1.0 / accel
        return alpha, schedule(L, alpha, cfg.n_layers, cfg.prune_layers, cfg.tau)
    if cfg.plan_mode != "cost":
        raise ValueError(cfg.plan_mode)
    full = model_cost(cfg, schedule(L, 1.0, cfg.n_layers, cfg.prune_layers, cfg.tau))
    target = full / accel
    if accel == 1.0:
        alpha = 1.0
    else:
        lo, hi = 0.0, 1.0
        for _ in range(60):
            mid = 0.5 * (lo + hi)
            c = model_cost(cfg, schedule(L, mid, cfg.n_layers, cfg.prune_layers, cfg.tau))
            if c <= target:
                lo = mid
            else:
                hi = mid
        alpha = lo
    return alpha, schedule(L, alpha, cfg.n_layers, cfg.prune_layers, cfg.tau)


def plan_varlen(cfg: OracleConfig, lengths: Sequence[int], accel: float):
    """One preservation rate for a batch of sequences of different lengths (R17).

    Sec. 3.4 picks alpha per inference call; with several lengths in one call
    the "cost" mode bisects (60 steps, as ``plan``) for the largest alpha whose
    modelled FLOPs summed over the batch are at most 1/accel of the unpruned
    sum, and every sequence follows Eq. 2 from its own length with that alpha.
    "rate": alpha = 1/accel.  Returns (alpha, [schedule per sequence]).
    """
    lengths = [int(x) for x in lengths]
    if not lengths or min(lengths) < 1:
        raise ValueError("lengths must be >= 1")
    if not accel >= 1.0:
        raise ValueError("accel must be >= 1")

    def scheds(a):
        return [schedule(L, a, cfg.n_layers, cfg.prune_layers, cfg.tau) for L in lengths]

    if cfg.plan_mode == "rate":
        alpha = 1.0 / accel
        return alpha, scheds(alpha)
    if cfg.plan_mode != "cost":
        raise ValueError(cfg.plan_mode)
    full = sum(model_cost(cfg, sc) for sc in scheds(1.0))
    target = full / accel
    if accel == 1.0:
        alpha = 1.0
    else:
        lo, hi = 0.0, 1.0
        for _ in range(60):
            mid = 0.5 * (lo + hi)
            if sum(model_cost(cfg, sc) for sc in scheds(mid)) <= target:
                lo = mid
            else:
                hi = mid
        alpha = lo
    return alpha, scheds(alpha)


# --------------------------------------------------------------------------
# forward pass
# --------------------------------------------------------------------------


def _as64(a) -> np.ndarray:
    return np.asarray(a, dtype=np.float64)


def attention_block(cfg: OracleConfig, lw: Dict[str, np.ndarray], h: np.ndarray, pos: np.ndarray,
                    store: _Store, key_mask: Optional[np.ndarray] = None,
                    kv_out: Optional[list] = None, detail: Optional[dict] = None):
    """Pre-norm attention branch of one layer on rows h [n, d].

    Returns (new residual h, P [H, n, n], v [n, Hkv, hd]).  If ``kv_out`` is a
    list, the layer's stored keys (after RoPE) and values are appended to it.
    If ``detail`` is a dict, the stored intermediates go into it: ``x``
    (normed rows), ``q``/``k``/``v``, ``o`` (attention output before the
    O-projection) and ``h1`` (the residual after the branch).
    """
    n = h.shape[0]
    H, G, hd = cfg.n_heads, cfg.n_kv_heads, cfg.head_dim
    ft = _ft(cfg)

    def W(name):
        return np.asarray(lw[name], dtype=ft)

    x = store(rmsnorm(h, lw["attn_norm"], cfg.rms_eps, ft))
    xf = np.asarray(x, dtype=ft)
    cos, sin = rope_angles(pos, hd, cfg.rope_theta)
    q = store(apply_rope((xf @ W("wq").T).reshape(n, H, hd), cos, sin))
    k = store(apply_rope((xf @ W("wk").T).reshape(n, G, hd), cos, sin))
    v = store((xf @ W("wv").T).reshape(n, G, hd))
    if kv_out is not None:
        kv_out.append((k, v))
    per = H // G
    P = np.empty((H, n, n), dtype=ft)
    o = np.empty((n, H, hd), dtype=ft)
    for hh in range(H):
        g = hh // per
        P[hh] = attention_probs(np.asarray(q[:, hh, :], dtype=ft), np.asarray(k[:, g, :], dtype=ft),
                               key_mask, cfg.causal)
        o[:, hh, :] = P[hh] @ np.asarray(v[:, g, :], dtype=ft)
    o = store(o.reshape(n, H * hd))
    h1 = store(np.asarray(h, dtype=ft) + np.asarray(o, dtype=ft) @ W("wo").T)
    if detail is not None:
        detail.update(x=x, q=q, k=k, v=v, o=o, h1=h1)
    return h1, P, v


def mlp_block(cfg: OracleConfig, lw: Dict[str, np.ndarray], h: np.ndarray, store: _Store,
              detail: Optional[dict] = None) -> np.ndarray:
    """Pre-norm SwiGLU branch: h + (silu(x Wg^T) * (x Wu^T)) Wd^T.

    If ``detail`` is a dict, ``x2`` (normed rows), ``a`` (the SwiGLU product)
    and ``h2`` (the residual after the branch) go into it."""
    ft = _ft(cfg)
    x = store(rmsnorm(h, lw["mlp_norm"], cfg.rms_eps, ft))
    xf = np.asarray(x, dtype=ft)
    a = store(silu(xf @ np.asarray(lw["wg"], ft).T) * (xf @ np.asarray(lw["wu"], ft).T))
    h2 = store(np.asarray(h, dtype=ft) + np.asarray(a, dtype=ft) @ np.asarray(lw["wd"], ft).T)
    if detail is not None:
        detail.update(x2=x, a=a, h2=h2)
    return h2


def head(cfg: OracleConfig, weights, h: np.ndarray, store: _Store) -> np.ndarray:
    """Final RMSNorm, then the LM head on every kept row, or the d x n_classes
    classifier on the last kept row (last-position pooling)."""
    ft = _ft(cfg)
    x = np.asarray(store(rmsnorm(h, weights["final_norm"], cfg.rms_eps, ft)), dtype=ft)
    W = np.asarray(weights["head"], dtype=ft)
    if cfg.n_classes > 0:
        return np.asarray(x[-1] @ W.T, dtype=np.float64)
    return np.asarray(x @ W.T, dtype=np.float64)


def decoder_layer(cfg: OracleConfig, lw: Dict[str, np.ndarray], layer: int, h: np.ndarray,
                  pos: np.ndarray, k_keep: int, store: _Store, forced: Optional[np.ndarray] = None,
                  kv_out: Optional[list] = None, detail: Optional[dict] = None):
    """One pre-norm decoder layer (Appendix A) on rows h [n, d] at original
    positions pos, with the Sec. 3.3 elimination when ``layer`` is a pruning
    layer: every row is scored (R1), the top ``k_keep`` are kept (ties by
    lower index, the last row forced when ``cfg.force_keep_last``) unless
    ``forced`` gives the kept indices, and the kept rows are compacted in
    order.  ``cfg.prune_point`` places the compaction after the MLP ("layer",
    R3) or between attention and MLP ("attention"); the kept rows come out
    the same either way.

    Returns (h, pos, idx, scores); idx and scores are None if the layer does
    not prune.  ``detail`` collects the blocks' intermediates (see
    ``attention_block`` / ``mlp_block``; the MLP's are on the rows it ran on).
    """
    if cfg.prune_point not in ("layer", "attention"):
        raise ValueError(cfg.prune_point)
    h, P, v = attention_block(cfg, lw, h, pos, store, kv_out=kv_out, detail=detail)
    if cfg.prune_point == "layer":
        h = mlp_block(cfg, lw, h, store, detail=detail)
    idx = s = None
    if layer in set(cfg.prune_layers):
        C = column_mass(P, cfg.n_kv_heads)
        s = position_scores(C, v, cfg.score_mode)
        if forced is not None:
            idx = np.asarray(forced, dtype=np.int64)
        elif k_keep == h.shape[0]:
            idx = np.arange(h.shape[0])
        else:
            idx = select_topk(s, k_keep, cfg.force_keep_last)
        h = h[idx]
        pos = pos[idx]
    if cfg.prune_point == "attention":
        h = mlp_block(cfg, lw, h, store, detail=detail)
    return h, pos, idx, s


def layer_rows(cfg: OracleConfig, lw: Dict[str, np.ndarray], h: np.ndarray, pos: np.ndarray,
               rows: Sequence[int], detail: Optional[dict] = None) -> np.ndarray:
    """Outputs of a layer that does not prune, for the listed rows only.

    Row i of a layer's output depends on row i and, through Eq. 1, on the keys
    and values of the rows it may attend to (rows 0..i for the causal mask,
    every row otherwise), so every row's key and value is computed and the
    attention, O-projection and MLP run for the listed query rows alone.
    Returns h_out [len(rows), d]; ``detail`` as ``attention_block`` /
    ``mlp_block``, for the listed rows.
    """
    rows = np.asarray(rows, dtype=np.int64)
    n = h.shape[0]
    H, G, hd = cfg.n_heads, cfg.n_kv_heads, cfg.head_dim
    ft = _ft(cfg)
    store = _Store(cfg.dtype)

    def W(name):
        return np.asarray(lw[name], dtype=ft)

    x = store(rmsnorm(h, lw["attn_norm"], cfg.rms_eps, ft)).astype(ft)
    cos, sin = rope_angles(pos, hd, cfg.rope_theta)
    k = store(apply_rope((x @ W("wk").T).reshape(n, G, hd), cos, sin))
    v = store((x @ W("wv").T).reshape(n, G, hd))
    q = store(apply_rope((x[rows] @ W("wq").T).reshape(len(rows), H, hd), cos[rows], sin[rows]))
    per = H // G
    o = np.empty((len(rows), H, hd), dtype=ft)
    for r, i in enumerate(rows):
        nk = i + 1 if cfg.causal else n
        for hh in range(H):
            g = hh // per
            logits = (k[:nk, g, :].astype(ft) @ q[r, hh].astype(ft)) / math.sqrt(hd)
            e = np.exp(logits - np.max(logits))
            o[r, hh] = (e / np.sum(e)) @ v[:nk, g, :].astype(ft)
    o = store(o.reshape(len(rows), H * hd))
    h1 = store(np.asarray(h[rows], dtype=ft) + o.astype(ft) @ W("wo").T)
    if detail is not None:
        detail.update(x=store(x[rows]), q=q, k=k[rows], v=v[rows], o=o, h1=h1)
    return mlp_block(cfg, lw, h1, store, detail=detail)


def forward(cfg: OracleConfig, weights, tokens: np.ndarray, accel: Optional[float] = None,
            alpha: Optional[float] = None, forced_idx: Optional[Dict[int, np.ndarray]] = None,
            collect: bool = False, collect_cache: bool = False):
    """Pruned prefill of a batch of token sequences [B, L].

    The preservation schedule comes from ``accel`` (via ``plan``) or from
    ``alpha`` directly.  ``forced_idx`` maps a 1-based pruning layer to kept
    indices [B, k] that replace the top-k choice there (scores are still
    computed and returned).

    Returns a dict with ``logits`` ([B, N_n, V] or [B, n_classes]),
    ``kept_pos`` [B, N_n], ``schedule``, ``alpha`` and per pruning layer
    ``idx`` [B, k] and ``scores`` [B, N_{l-1}].  With ``collect`` it also has
    ``layer_inputs`` {l: (h [B, N_{l-1}, d], pos [B, N_{l-1}])} and
    ``final_hidden`` [B, N_n, d] (the residual rows entering the head).
    With ``collect_cache`` it also has ``cache`` (see ``decode_step``): per
    layer the stored keys and values of the rows that layer ran on.
    """
    tokens = np.asarray(tokens)
    B, L = tokens.shape
    if accel is not None:
        alpha, sched = plan(cfg, L, accel)
    else:
        if alpha is None:
            alpha = 1.0
        sched = schedule(L, alpha, cfg.n_layers, cfg.prune_layers, cfg.tau)
    store = _Store(cfg.dtype)
    emb = _as64(weights["embed"])
    logits, kept_pos = [], []
    idx_all: Dict[int, list] = {}
    scores_all: Dict[int, list] = {}
    inputs_all: Dict[int, list] = {}
    cache_all: Dict[int, list] = {}
    finals = []
    for b in range(B):
        h = store(emb[tokens[b]])
        pos = np.arange(L)
        for layer in range(1, cfg.n_layers + 1):
            lw = weights["layers"][layer - 1]
            if collect:
                inputs_all.setdefault(layer, []).append((h, pos))
            kv: list = []
            fi = forced_idx[layer][b] if forced_idx is not None and layer in forced_idx else None
            h, pos_new, idx, s = decoder_layer(cfg, lw, layer, h, pos, sched[layer], store, forced=fi,
                                               kv_out=kv)
            if collect_cache:
                cache_all.setdefault(layer, []).append((kv[0][0], kv[0][1], pos))
            pos = pos_new
            if idx is not None:
                idx_all.setdefault(layer, []).append(idx)
                scores_all.setdefault(layer, []).append(s)
        logits.append(head(cfg, weights, h, store))
        kept_pos.append(pos)
        finals.append(h)
    out = {
        "logits": np.stack(logits),
        "kept_pos": np.stack(kept_pos),
        "schedule": sched,
        "alpha": alpha,
        "idx": {k: np.stack(v) for k, v in idx_all.items()},
        "scores": {k: np.stack(v) for k, v in scores_all.items()},
    }
    if collect:
        out["layer_inputs"] = {k: (np.stack([a for a, _ in v]), np.stack([p for _, p in v]))
                               for k, v in inputs_all.items()}
        out["final_hidden"] = np.stack(finals)
    if collect_cache:
        out["cache"] = {"L": L, "layers": {
            layer: {"k": np.stack([a for a, _, _ in v]), "v": np.stack([b for _, b, _ in v]),
                    "pos": np.stack([p for _, _, p in v])}
            for layer, v in cache_all.items()}}
    return out


def forward_masked(cfg: OracleConfig, weights, tokens: np.ndarray, sched: Sequence[int]):
    """Appendix B formulation: pruned rows stay in place but are marked.

    Every layer runs on all L rows.  Marked rows are never used as keys again
    and their own outputs are ignored; at a pruning layer the scores come from
    unmarked queries only and the top-N_l unmarked rows stay unmarked.
    Returns logits of the rows unmarked at the end, their positions, and the
    kept positions after each pruning layer.
    """
    tokens = np.asarray(tokens)
    B, L = tokens.shape
    store = _Store(cfg.dtype)
    emb = _as64(weights["embed"])
    G = cfg.n_kv_heads
    logits, kept_pos, kept_by_layer = [], [], {}
    for b in range(B):
        h = store(emb[tokens[b]])
        active = np.ones(L, dtype=bool)
        for layer in range(1, cfg.n_layers + 1):
            lw = weights["layers"][layer - 1]
            h, P, v = attention_block(cfg, lw, h, np.arange(L), store, key_mask=active)
            h = mlp_block(cfg, lw, h, store)
            if layer in set(cfg.prune_layers):
                act_idx = np.nonzero(active)[0]
                Pa = P[:, act_idx][:, :, act_idx]  # active queries x active keys
                C = column_mass(Pa, G)
                s = position_scores(C, v[act_idx], cfg.score_mode)
                k_keep = sched[layer]
                if k_keep < act_idx.shape[0]:
                    keep = act_idx[select_topk(s, k_keep, cfg.force_keep_last)]
                    active = np.zeros(L, dtype=bool)
                    active[keep] = True
                kept_by_layer.setdefault(layer, []).append(np.nonzero(active)[0])
        rows = np.nonzero(active)[0]
        logits.append(head(cfg, weights, h[rows], store))
        kept_pos.append(rows)
    return {
        "logits": np.stack(logits),
        "kept_pos": np.stack(kept_pos),
        "kept_by_layer": {k: np.stack(v) for k, v in kept_by_layer.items()},
    }


def forward_marked(cfg: OracleConfig, weights, tokens: np.ndarray, sched: Sequence[int]):
    """Appendix B's figure: every hidden activation stays, including those
    marked as pruned, and a row marked at one layer can be reactivated at a
    later one.

    Reading (R18): a row hidden as a key receives soft-score zero in every
    later layer (Eq. 1 gives it no probability), so under the R1 score it
    could never come back; reactivation needs the marked rows to stay in the
    computation.  So nothing is removed or hidden: every layer runs on all L
    rows as the unpruned decoder does, and each pruning layer marks as
    preserved the top N_l of ALL L rows by that layer's scores (R1, ties and
    the forced last row as ``select_topk``), whatever the earlier marks.  The
    output is the logits of the rows preserved at the last pruning layer,
    i.e. the unpruned forward's logits at those positions.

    Returns ``logits``, ``kept_pos`` [B, N_n], and per pruning layer
    ``kept_by_layer`` [B, N_l] and ``scores`` [B, L].
    """
    tokens = np.asarray(tokens)
    B, L = tokens.shape
    store = _Store(cfg.dtype)
    emb = _as64(weights["embed"])
    G = cfg.n_kv_heads
    logits, kept_pos, kept_by_layer, scores_by_layer = [], [], {}, {}
    for b in range(B):
        h = store(emb[tokens[b]])
        pos = np.arange(L)
        keep = pos
        for layer in range(1, cfg.n_layers + 1):
            lw = weights["layers"][layer - 1]
            h, P, v = attention_block(cfg, lw, h, pos, store)
            if layer in set(cfg.prune_layers):
                s = position_scores(column_mass(P, G), v, cfg.score_mode)
                k_keep = sched[layer]
                keep = select_topk(s, k_keep, cfg.force_keep_last) if k_keep < L else np.arange(L)
                kept_by_layer.setdefault(layer, []).append(keep)
                scores_by_layer.setdefault(layer, []).append(s)
            h = mlp_block(cfg, lw, h, store)
        logits.append(head(cfg, weights, h[keep], store))
        kept_pos.append(keep)
    return {
        "logits": np.stack(logits),
        "kept_pos": np.stack(kept_pos),
        "kept_by_layer": {k: np.stack(v) for k, v in kept_by_layer.items()},
        "scores": {k: np.stack(v) for k, v in scores_by_layer.items()},
    }


def forward_varlen(cfg: OracleConfig, weights, seqs: Sequence[np.ndarray], accel: Optional[float] = None,
                   alpha: Optional[float] = None, forced_idx: Optional[Dict[int, list]] = None):
    """Pruned prefill of sequences of different lengths in one call.

    The rate comes from ``plan_varlen`` (or ``alpha``); each sequence then
    runs ``forward`` on its own (a sequence never attends to another one).
    ``forced_idx`` maps a pruning layer to a list of per-sequence index arrays.
    Returns a dict of per-sequence lists (``logits``, ``kept_pos``,
    ``schedule``, ``idx`` {layer: [..]}, ``scores`` {layer: [..]}) and ``alpha``.
    """
    lengths = [len(t) for t in seqs]
    if alpha is None:
        alpha, _ = plan_varlen(cfg, lengths, 1.0 if accel is None else accel)
    out = {"alpha": alpha, "logits": [], "kept_pos": [], "schedule": [], "idx": {}, "scores": {}}
    for b, t in enumerate(seqs):
        fi = None if forced_idx is None else {l: np.asarray(v[b])[None] for l, v in forced_idx.items()}
        r = forward(cfg, weights, np.asarray(t)[None], alpha=alpha, forced_idx=fi)
        out["logits"].append(r["logits"][0])
        out["kept_pos"].append(r["kept_pos"][0])
        out["schedule"].append(r["schedule"])
        for l, v in r["idx"].items():
            out["idx"].setdefault(l, []).append(v[0])
        for l, v in r["scores"].items():
            out["scores"].setdefault(l, []).append(v[0])
    return out


# --------------------------------------------------------------------------
# generation over the pruned KV cache
# --------------------------------------------------------------------------


def attention_probs_one(q: np.ndarray, k: np.ndarray) -> np.ndarray:
    """Eq. 1 for one query that comes after every key: softmax(q k^T / sqrt(d_k)).

    q: [hd], k: [n, hd].  The causal mask hides nothing here (every cached key
    is at an earlier position, or is the query's own).  Returns p [n]."""
    logits = (k @ q) / math.sqrt(q.shape[0])
    e = np.exp(logits - np.max(logits))
    return e / np.sum(e)


def decode_step(cfg: OracleConfig, weights, cache, tokens: np.ndarray):
    """One generated token per sequence after a pruned prefill.

    Sec. 3.3 removes a pruned row from every later layer, so in layer l the
    new token attends to the rows layer l ran on during the prefill (their
    stored keys and values, RoPE at their original positions) plus the tokens
    generated so far and itself; generated tokens are never pruned.

    cache: ``{"L": L, "layers": {l: {"k": [B, n_l, Hkv, hd], "v": ..., "pos": [B, n_l]}}}``
    as returned by ``forward(..., collect_cache=True)`` or a previous call.
    tokens: [B] ids of the new tokens, at position L + (tokens generated so far).
    Returns (logits [B, V] of the new tokens, the cache with their keys and values appended).
    """
    if cfg.n_classes > 0:
        raise ValueError("generation needs the language-model head")
    if not cfg.causal:
        raise ValueError("generation needs causal attention")
    tokens = np.asarray(tokens)
    B = tokens.shape[0]
    H, G, hd = cfg.n_heads, cfg.n_kv_heads, cfg.head_dim
    per = H // G
    store = _Store(cfg.dtype)
    emb = _as64(weights["embed"])
    layers = cache["layers"]
    position = cache["L"] + cache.get("generated", 0)
    new_layers = {}
    logits = []
    for layer in range(1, cfg.n_layers + 1):
        new_layers[layer] = {"k": [], "v": [], "pos": []}
    for b in range(B):
        h = store(emb[tokens[b]])[None, :]
        for layer in range(1, cfg.n_layers + 1):
            lw = weights["layers"][layer - 1]
            c = layers[layer]
            x = store(rmsnorm(h, lw["attn_norm"], cfg.rms_eps))
            cos, sin = rope_angles(np.array([position]), hd, cfg.rope_theta)
            q = store(apply_rope((x @ _as64(lw["wq"]).T).reshape(1, H, hd), cos, sin))[0]
            k = store(apply_rope((x @ _as64(lw["wk"]).T).reshape(1, G, hd), cos, sin))
            v = store((x @ _as64(lw["wv"]).T).reshape(1, G, hd))
            K = np.concatenate([c["k"][b], k], axis=0)
            V = np.concatenate([c["v"][b], v], axis=0)
            o = np.empty((H, hd))
            for hh in range(H):
                g = hh // per
                o[hh] = attention_probs_one(q[hh], K[:, g, :]) @ V[:, g, :]
            o = store(o.reshape(1, H * hd))
            h = store(h + o @ _as64(lw["wo"]).T)
            h = mlp_block(cfg, lw, h, store)
            new_layers[layer]["k"].append(K)
            new_layers[layer]["v"].append(V)
            new_layers[layer]["pos"].append(np.append(c["pos"][b], position))
        logits.append(head(cfg, weights, h, store)[0])
    out_cache = {"L": cache["L"], "generated": cache.get("generated", 0) + 1,
                 "layers": {layer: {kk: np.stack(vv) for kk, vv in d.items()}
                            for layer, d in new_layers.items()}}
    return np.stack(logits), out_cache


def generate(cfg: OracleConfig, weights, tokens: np.ndarray, new_tokens: np.ndarray,
             accel: Optional[float] = None, alpha: Optional[float] = None,
             forced_idx: Optional[Dict[int, np.ndarray]] = None):
    """Pruned prefill of tokens [B, L], then one ``decode_step`` per column of
    new_tokens [B, T] (teacher-forced ids).  Returns a dict with the prefill's
    output (``prefill``), ``logits`` [B, T, V] of the generated tokens and the
    final ``cache``."""
    pre = forward(cfg, weights, tokens, accel=accel, alpha=alpha, forced_idx=forced_idx,
                  collect_cache=True)
    cache = pre["cache"]
    out = []
    for t in range(np.asarray(new_tokens).shape[1]):
        lg, cache = decode_step(cfg, weights, cache, np.asarray(new_tokens)[:, t])
        out.append(lg)
    T = np.asarray(new_tokens).shape[1]
    logits = np.stack(out, axis=1) if T else np.zeros((tokens.shape[0], 0, cfg.vocab))
    return {"prefill": pre, "logits": logits, "cache": cache}


# --------------------------------------------------------------------------
# isolated score + select + gather (no attention: C = 1, one group)
# --------------------------------------------------------------------------


def score_select(hidden: np.ndarray, k: int, force_last: bool = False):
    """Score every row of hidden [B, L, d] by its L2 norm (the R1 score with
    unit column mass and a single group), keep the top k per sequence.

    Returns (scores [B, L], idx [B, k] ascending, gathered [B, k, d])."""
    hidden = np.asarray(hidden)
    B = hidden.shape[0]
    scores = np.sqrt(np.sum(_as64(hidden) ** 2, axis=-1))
    idx = np.stack([select_topk(scores[b], k, force_last) for b in range(B)])
    gathered = np.stack([hidden[b][idx[b]] for b in range(B)])
    return scores, idx, gathered
