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


def rand_bf16(shape, seed, scale=1.0):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    return (torch.randn(*shape, generator=g, device="cuda") * scale).to(torch.bfloat16)


def np64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def linear_case(z, epi, M, N, K, seed, hd=64, rope_cols=0):
    """One zsaa_op_linear call on seeded bf16 operands; returns (output, float64
    reference of the same operands and epilogue, per-element tolerance)."""
    A = rand_bf16((M, K), seed)
    W = rand_bf16((N, K), seed + 1, 0.05)
    An, Wn = np64(A), np64(W)
    tol = accum_bound(An, Wn)
    if epi == "swiglu":
        W2 = rand_bf16((N, K), seed + 2, 0.05)
        out = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
        z.zsaa_op_linear(A, W, W2, None, out, M, N, K, z.ZSAA_BF16, z.EPI_SWIGLU)
        g, u = An @ Wn.T, An @ np64(W2).T
        ref = O.bf16_round(O.silu(g) * u)
        tol = 1.1 * np.abs(u) * tol + np.abs(O.silu(g)) * accum_bound(An, np64(W2))
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
        H = rand_bf16((M, N), seed + 3)
        h0 = np64(H)
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


def check_linear(out, ref, tol, epi, what):
    """float32 outputs within the accumulation bound; bf16 within 2 ulps plus the
    bound, 99.5% within 1 ulp."""
    got = np64(out)
    if epi == "store_f32":
        assert np.all(np.abs(got - ref) <= tol + 1e-6 * np.abs(ref)), what
    else:
        assert np.all(bf16_ulp_close(got, ref, 2, tol)), what
        assert np.mean(bf16_ulp_close(got, ref, 1)) > 0.995, what


def bf16_ulp(x):
    """One bf16 unit in the last place of each |x| (2^-133 at zero)."""
    mag = np.abs(np.asarray(x, np.float64))
    return np.where(mag > 0, 2.0 ** (np.floor(np.log2(np.maximum(mag, 1e-38))) - 7), 2.0 ** -133)


def layer_noise_scale(det, lw):
    """Rounding-noise scale of each element of a decoder layer's output rows.

    A bf16-storage layer computed with float32 sums differs from the float64
    oracle only through 1-ulp flips at its storage points, which propagate
    through the next product.  For the output h2 = round(h1 + a Wd^T) with
    h1 = round(h + o Wo^T) (from identical inputs h), each flip of o or a moves
    an output by one ulp times its weight, with an arbitrary sign, so the
    scale of the difference is
        sigma^2 = ulp(h2)^2 + ulp(h1)^2 + ulp(o)^2 (Wo^2)^T + ulp(a)^2 (Wd^2)^T
    per element (the upstream flips of x, q, k, v and x2 surface as flips of
    o and a).  ``det`` holds the oracle's o, h1, a, h2 for the compared rows."""
    wo = np.asarray(lw["wo"], np.float64)
    wd = np.asarray(lw["wd"], np.float64)
    s2 = bf16_ulp(det["h2"]) ** 2 + bf16_ulp(det["h1"]) ** 2
    s2 = s2 + (bf16_ulp(det["o"]) ** 2) @ (wo * wo).T + (bf16_ulp(det["a"]) ** 2) @ (wd * wd).T
    return np.sqrt(s2)


def layer_error_stats(got, ref, sigma):
    """Per-element comparison of layer outputs: z = |got - ref| / sigma, and
    the fractions of elements within 0, 1 and 2 bf16 ulps."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    err = np.abs(got - ref)
    z = err / sigma
    ulp = bf16_ulp(np.maximum(np.abs(got), np.abs(ref)))
    return dict(z_max=float(z.max()), z_mean=float(z.mean()), exact=float(np.mean(err == 0)),
                ulp1=float(np.mean(err <= ulp)), ulp2=float(np.mean(err <= 2 * ulp)),
                rel_mean=float(err.mean() / max(np.abs(ref).mean(), 1e-30)), n=int(err.size))


def oracle_pruning_layer_at(cfg, lw, h, pos, ks, rows_for_k, store, forced=None):
    """decoder_layer with the compaction between attention and MLP, for
    several kept counts at once: the attention branch and the scores (Sec. 3.2,
    R1) do not depend on k, the top-k (Sec. 3.3) and the compaction do, and the
    MLP acts on each kept row alone, so it runs for the kept rows
    ``rows_for_k(k, idx)`` (indices into the kept set) only.

    ``forced`` ({k: idx}) replaces the top-k choice (the scores are still
    computed).  Returns (scores [n], {k: (idx [k], rows, h_out [len(rows), d],
    det)}) where det holds o, h1, a, h2 of those rows (``layer_noise_scale``)."""
    det = {}
    h1, P, v = O.attention_block(cfg, lw, h, pos, store, detail=det)
    s = O.position_scores(O.column_mass(P, cfg.n_kv_heads), v, cfg.score_mode)
    del P
    out = {}
    for k in ks:
        if forced is not None and k in forced:
            idx = np.asarray(forced[k], dtype=np.int64)
        elif k == h.shape[0]:
            idx = np.arange(h.shape[0])
        else:
            idx = O.select_topk(s, k, cfg.force_keep_last)
        rows = np.asarray(rows_for_k(k, idx), dtype=np.int64)
        sel = idx[rows]
        dm = {}
        h2 = O.mlp_block(cfg, lw, h1[sel], store, detail=dm)
        out[k] = (idx, rows, h2, dict(o=det["o"][sel], h1=h1[sel], a=dm["a"], h2=h2))
    return s, out


def sample_rows(n, count, seed):
    """``count`` distinct row indices of [0, n), always with the last one, sorted."""
    if n <= count:
        return np.arange(n)
    rng = np.random.default_rng(seed)
    return np.sort(np.append(rng.choice(n - 1, count - 1, replace=False), n - 1))
