"""Pins for the CPU oracle: each check compares it with something other than
itself (a library routine, a closed form, an invariant, brute force or a
hand-worked example from the paper), so that a dropped term, a wrong sign or
index, or a transposed operand fails at least one test."""

import dataclasses
import itertools
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import zsaa_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- bf16 storage

def test_bf16_round_matches_torch_cast():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        rng.standard_normal(20000) * 10.0 ** rng.integers(-40, 38, 20000),
        np.array([0.0, -0.0, np.inf, -np.inf, 1e-45, -3e-39, 3.3895e38, 1.0 + 2.0 ** -8,
                  1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -8 + 2.0 ** -20]),
    ]).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    got = O.bf16_round(x)
    assert np.array_equal(got, ref)
    assert np.isnan(O.bf16_round(np.array([np.nan], np.float32)))[0]


# ---------------------------------------------------------------- RMSNorm

def test_rmsnorm_matches_torch_and_unit_rms():
    rng = np.random.default_rng(1)
    h = rng.standard_normal((7, 48)) * 3.0
    w = rng.standard_normal(48)
    got = O.rmsnorm(h, w, 1e-5)
    ref = F.rms_norm(torch.from_numpy(h), (48,), weight=torch.from_numpy(w), eps=1e-5).numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)
    unit = O.rmsnorm(h, np.ones(48), 0.0)
    np.testing.assert_allclose(np.mean(unit ** 2, axis=-1), 1.0, rtol=1e-12)


# ---------------------------------------------------------------- RoPE

def _rope_complex(x, pos, theta):
    """Same rotation written as complex multiplication z * exp(i * pos * f)."""
    hd = x.shape[-1]
    half = hd // 2
    f = np.array([theta ** (-2.0 * i / hd) for i in range(half)])
    z = x[..., :half] + 1j * x[..., half:]
    z = z * np.exp(1j * pos[:, None, None] * f[None, None, :])
    return np.concatenate([z.real, z.imag], axis=-1)


def test_rope_matches_complex_rotation_and_is_relative():
    rng = np.random.default_rng(2)
    n, H, hd, theta = 9, 3, 16, 10000.0
    pos = rng.integers(0, 5000, n)
    x = rng.standard_normal((n, H, hd))
    cos, sin = O.rope_angles(pos, hd, theta)
    got = O.apply_rope(x, cos, sin)
    np.testing.assert_allclose(got, _rope_complex(x, pos, theta), rtol=1e-10, atol=1e-10)
    # rotation: norms preserved; position 0 is the identity
    np.testing.assert_allclose(np.linalg.norm(got, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-12)
    c0, s0 = O.rope_angles(np.zeros(n), hd, theta)
    np.testing.assert_allclose(O.apply_rope(x, c0, s0), x, atol=0)
    # relative: <rope(q, m), rope(k, n)> depends on m - n only
    q, k = rng.standard_normal((1, 1, hd)), rng.standard_normal((1, 1, hd))

    def dot(m, nn):
        cq, sq = O.rope_angles(np.array([m]), hd, theta)
        ck, sk = O.rope_angles(np.array([nn]), hd, theta)
        return float(np.sum(O.apply_rope(q, cq, sq) * O.apply_rope(k, ck, sk)))

    assert abs(dot(10, 3) - dot(110, 103)) < 1e-9
    assert abs(dot(10, 3) - dot(11, 3)) > 1e-6


def test_silu_matches_torch():
    x = np.linspace(-30, 30, 1001)
    np.testing.assert_allclose(O.silu(x), F.silu(torch.from_numpy(x)).numpy(), rtol=1e-12, atol=1e-300)


# ---------------------------------------------------------------- Eq. 1

@pytest.mark.parametrize("n,hd", [(1, 8), (13, 16), (40, 32)])
def test_attention_eq1_matches_sdpa(n, hd):
    rng = np.random.default_rng(n)
    q = rng.standard_normal((n, hd)) * 2
    k = rng.standard_normal((n, hd)) * 2
    v = rng.standard_normal((n, hd))
    P = O.attention_probs(q, k)
    ref = F.scaled_dot_product_attention(
        torch.from_numpy(q)[None, None], torch.from_numpy(k)[None, None],
        torch.from_numpy(v)[None, None], is_causal=True)[0, 0].numpy()
    np.testing.assert_allclose(P @ v, ref, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(P.sum(axis=1), 1.0, rtol=1e-12)
    assert np.all(P[np.triu_indices(n, 1)] == 0.0)


def test_attention_key_mask_excludes_keys():
    rng = np.random.default_rng(5)
    n, hd = 10, 8
    q, k = rng.standard_normal((n, hd)), rng.standard_normal((n, hd))
    mask = np.array([1, 0, 1, 1, 0, 1, 0, 1, 1, 1], bool)
    P = O.attention_probs(q, k, mask)
    assert np.all(P[:, ~mask] == 0.0)
    idx = np.nonzero(mask)[0]
    # restricted to the unmasked rows it is the plain causal softmax on the compacted sequence
    np.testing.assert_allclose(P[np.ix_(idx, idx)], O.attention_probs(q[idx], k[idx]), rtol=1e-12)


# ---------------------------------------------------------------- column mass

def test_column_mass_closed_form_uniform_attention():
    # q = 0 makes every allowed logit equal, so P[i, j] = 1/(i+1) for j <= i and
    # C_j = heads_per_group * (H_N - H_j) with H_m the m-th harmonic number.
    n, H, G, hd = 17, 6, 2, 8
    rng = np.random.default_rng(3)
    k = rng.standard_normal((n, hd))
    P = np.stack([O.attention_probs(np.zeros((n, hd)), k) for _ in range(H)])
    C = O.column_mass(P, G)
    harm = np.concatenate([[0.0], np.cumsum(1.0 / np.arange(1, n + 1))])
    expect = (H // G) * (harm[n] - harm[np.arange(n)])
    for g in range(G):
        np.testing.assert_allclose(C[g], expect, rtol=1e-12)


def test_column_mass_brute_force_and_total():
    rng = np.random.default_rng(4)
    H, G, n = 4, 2, 6
    P = np.stack([O.attention_probs(rng.standard_normal((n, 4)), rng.standard_normal((n, 4)))
                  for _ in range(H)])
    C = O.column_mass(P, G)
    for g in range(G):
        for j in range(n):
            tot = 0.0
            for h in range(H):
                if h // (H // G) != g:
                    continue
                for i in range(n):
                    tot += P[h, i, j]
            assert abs(C[g, j] - tot) < 1e-12
    # every row of P sums to one, so a group's columns total heads_per_group * n
    np.testing.assert_allclose(C.sum(axis=1), (H // G) * n, rtol=1e-12)


def test_position_scores_reduce_to_row_norm():
    rng = np.random.default_rng(6)
    v = rng.standard_normal((11, 1, 24))
    s = O.position_scores(np.ones((1, 11)), v, "softscore_vnorm")
    np.testing.assert_allclose(s, np.linalg.norm(v[:, 0, :], axis=1), rtol=1e-12)
    C = rng.random((3, 11))
    np.testing.assert_allclose(O.position_scores(C, rng.standard_normal((11, 3, 4)), "softscore"),
                               C.sum(axis=0), rtol=1e-12)
    # linear in each group's value row: scaling group 1's v by 3 adds 2*C[1]*|v1|
    v3 = rng.standard_normal((11, 3, 4))
    v3b = v3.copy()
    v3b[:, 1, :] *= 3.0
    diff = O.position_scores(C, v3b, "softscore_vnorm") - O.position_scores(C, v3, "softscore_vnorm")
    np.testing.assert_allclose(diff, 2.0 * C[1] * np.linalg.norm(v3[:, 1, :], axis=1), rtol=1e-10)


# ---------------------------------------------------------------- top-k

def _brute_keep(s, k, force_last):
    """j is kept iff fewer than `need` candidates beat it (greater score, or equal
    score and lower index; NaN beaten by everything numeric)."""
    n = len(s)
    cand = list(range(n - 1)) if force_last else list(range(n))
    need = k - 1 if force_last else k

    def beats(a, b):
        if math.isnan(s[b]) and not math.isnan(s[a]):
            return True
        if math.isnan(s[a]):
            return math.isnan(s[b]) and a < b
        return s[a] > s[b] or (s[a] == s[b] and a < b)

    kept = [j for j in cand if sum(beats(a, j) for a in cand if a != j) < need]
    if force_last:
        kept.append(n - 1)
    return sorted(kept)


def test_select_topk_brute_force_with_ties():
    rng = np.random.default_rng(7)
    for trial in range(400):
        n = int(rng.integers(1, 9))
        s = rng.integers(0, 4, n).astype(float)
        if trial % 5 == 0:
            s[rng.integers(0, n)] = np.nan
        for k in range(1, n + 1):
            for fl in (False, True):
                got = O.select_topk(s, k, fl)
                assert list(got) == _brute_keep(s, k, fl)
                assert len(got) == k and len(set(got.tolist())) == k
                assert np.all(np.diff(got) > 0)


def test_select_topk_exhaustive_small():
    # every score vector over {0,1,2} of length 5: the kept set maximises the
    # score sum and, among maximisers, is lexicographically smallest.
    for s in itertools.product([0.0, 1.0, 2.0], repeat=5):
        s = np.array(s)
        for k in range(1, 6):
            best = max(itertools.combinations(range(5), k), key=lambda c: (sum(s[list(c)]), [-x for x in c]))
            assert list(O.select_topk(s, k, False)) == list(best)


# ---------------------------------------------------------------- Eq. 2

def _golden_schedules():
    rows = []
    with open(os.path.join(GOLDEN, "eq2_schedule.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            lhs, rhs = line.split(":")
            L, alpha, tau, n, pl = lhs.split()
            rows.append((int(L), float(alpha), int(tau), int(n), [int(x) for x in pl.split(",")],
                         [int(x) for x in rhs.split()]))
    return rows


@pytest.mark.parametrize("row", _golden_schedules())
def test_schedule_matches_hand_worked_eq2(row):
    L, alpha, tau, n, pl, expect = row
    assert O.schedule(L, alpha, n, pl, tau) == expect


def _cfg(**kw):
    base = dict(n_layers=4, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16, ffn_dim=96,
                vocab=50, rope_theta=10000.0, dtype="f32", prune_layers=[1, 2, 3])
    base.update(kw)
    return O.OracleConfig(**base)


def test_plan_meets_cost_target_and_is_tight():
    cfg = _cfg(n_layers=16, d_model=2048, n_heads=32, n_kv_heads=8, head_dim=64, ffn_dim=8192,
               vocab=128256, prune_layers=list(range(1, 16)))
    L = 512
    full = O.model_cost(cfg, O.schedule(L, 1.0, 16, cfg.prune_layers, 5))
    a1, s1 = O.plan(cfg, L, 1.0)
    assert a1 == 1.0 and s1 == [L] * 17
    prev = 1.0
    for accel in (1.5, 2.0, 4.0, 8.0):
        alpha, sched = O.plan(cfg, L, accel)
        assert O.model_cost(cfg, sched) <= full / accel
        # a slightly larger alpha would break the target (bisection is tight)
        worse = O.schedule(L, min(1.0, alpha + 1e-9), 16, cfg.prune_layers, 5)
        assert O.model_cost(cfg, worse) > full / accel or worse == sched
        assert alpha < prev
        prev = alpha


def test_plan_rate_mode():
    cfg = _cfg(n_layers=2, prune_layers=[1], plan_mode="rate")
    alpha, sched = O.plan(cfg, 64, 2.0)
    assert alpha == 0.5 and sched == [64, 32, 32]
    with pytest.raises(ValueError):
        O.plan(cfg, 64, 0.5)


# ---------------------------------------------------------------- forward

def _tiny_weights(cfg, seed=0, scale=0.3):
    rng = np.random.default_rng(seed)
    d, hd = cfg.d_model, cfg.head_dim

    def nrm(*s):
        return rng.standard_normal(s) * scale

    layers = []
    for _ in range(cfg.n_layers):
        layers.append(dict(attn_norm=1 + 0.1 * nrm(d), wq=nrm(cfg.n_heads * hd, d),
                           wk=nrm(cfg.n_kv_heads * hd, d), wv=nrm(cfg.n_kv_heads * hd, d),
                           wo=nrm(d, cfg.n_heads * hd) * 0.3, mlp_norm=1 + 0.1 * nrm(d),
                           wg=nrm(cfg.ffn_dim, d), wu=nrm(cfg.ffn_dim, d), wd=nrm(d, cfg.ffn_dim) * 0.3))
    heads = cfg.n_classes if cfg.n_classes else cfg.vocab
    return dict(embed=nrm(cfg.vocab, d), layers=layers, final_norm=1 + 0.1 * nrm(d), head=nrm(heads, d))


def _torch_forward_unpruned(cfg, w, tokens, key_alive=None, all_rows=False):  # noqa: C901
    """Unpruned decoder composed from torch library routines (float64).

    ``key_alive[l]`` (bool [B, n], 0-based layer l) hides keys from layer l on
    top of the causal mask; ``all_rows`` returns logits of every row."""
    T = lambda a: torch.from_numpy(np.asarray(a, np.float64))  # noqa: E731
    H, G, hd, d = cfg.n_heads, cfg.n_kv_heads, cfg.head_dim, cfg.d_model
    out = []
    for b in range(tokens.shape[0]):
        n = tokens.shape[1]
        h = T(w["embed"])[torch.from_numpy(tokens[b].astype(np.int64))]
        pos = np.arange(n)
        for li, lw in enumerate(w["layers"]):
            x = F.rms_norm(h, (d,), weight=T(lw["attn_norm"]), eps=cfg.rms_eps)
            q = F.linear(x, T(lw["wq"])).view(n, H, hd).numpy()
            k = F.linear(x, T(lw["wk"])).view(n, G, hd).numpy()
            v = F.linear(x, T(lw["wv"])).view(n, G, hd)
            q = T(_rope_complex(q, pos, cfg.rope_theta)).transpose(0, 1)[None]
            k = T(_rope_complex(k, pos, cfg.rope_theta)).transpose(0, 1)[None]
            if key_alive is None:
                o = F.scaled_dot_product_attention(q, k, v.transpose(0, 1)[None], is_causal=cfg.causal,
                                                   enable_gqa=True)
            else:
                allowed = torch.tril(torch.ones(n, n, dtype=torch.bool))
                allowed &= torch.from_numpy(np.asarray(key_alive[li][b], bool))[None, :]
                o = F.scaled_dot_product_attention(q, k, v.transpose(0, 1)[None], attn_mask=allowed,
                                                   enable_gqa=True)
            h = h + F.linear(o[0].transpose(0, 1).reshape(n, H * hd), T(lw["wo"]))
            x = F.rms_norm(h, (d,), weight=T(lw["mlp_norm"]), eps=cfg.rms_eps)
            h = h + F.linear(F.silu(F.linear(x, T(lw["wg"]))) * F.linear(x, T(lw["wu"])), T(lw["wd"]))
        x = F.rms_norm(h, (d,), weight=T(w["final_norm"]), eps=cfg.rms_eps)
        logits = F.linear(x, T(w["head"]))
        out.append(logits[-1] if cfg.n_classes and not all_rows else logits)
    return torch.stack(out).numpy()


@pytest.mark.parametrize("n_classes", [0, 3])
def test_unpruned_forward_matches_torch_composition(n_classes):
    cfg = _cfg(n_classes=n_classes, prune_layers=[])
    w = _tiny_weights(cfg)
    tokens = np.random.default_rng(8).integers(0, cfg.vocab, (2, 19))
    got = O.forward(cfg, w, tokens, accel=1.0)
    ref = _torch_forward_unpruned(cfg, w, tokens)
    np.testing.assert_allclose(got["logits"], ref, rtol=1e-9, atol=1e-9)


def test_accel_one_equals_unpruned():
    cfg = _cfg()
    w = _tiny_weights(cfg, seed=1)
    tokens = np.random.default_rng(9).integers(0, cfg.vocab, (2, 23))
    a = O.forward(cfg, w, tokens, accel=1.0)
    b = O.forward(_cfg(prune_layers=[]), w, tokens, accel=1.0)
    assert a["schedule"] == [23] * 5
    np.testing.assert_array_equal(a["logits"], b["logits"])
    np.testing.assert_array_equal(a["kept_pos"], np.tile(np.arange(23), (2, 1)))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_compacted_equals_masked_formulation(dtype):
    # Appendix B: keeping pruned rows in place but masked must give the same kept
    # rows, positions and logits as physically removing them.
    cfg = _cfg(dtype=dtype, prune_layers=[1, 2, 3], n_layers=4)
    w = _tiny_weights(cfg, seed=2)
    tokens = np.random.default_rng(10).integers(0, cfg.vocab, (2, 37))
    alpha = 0.6
    sched = O.schedule(37, alpha, cfg.n_layers, cfg.prune_layers, cfg.tau)
    assert sched[-1] < 37
    a = O.forward(cfg, w, tokens, alpha=alpha)
    m = O.forward_masked(cfg, w, tokens, sched)
    np.testing.assert_array_equal(a["kept_pos"], m["kept_pos"])
    if dtype == "f32":
        np.testing.assert_allclose(a["logits"], m["logits"], rtol=1e-9, atol=1e-9)
    else:  # different matmul shapes may flip a rare bf16 rounding
        assert np.max(np.abs(a["logits"] - m["logits"])) < 2e-2


def test_forced_indices_reproduce_natural_choice_and_last_kept():
    cfg = _cfg()
    w = _tiny_weights(cfg, seed=3)
    tokens = np.random.default_rng(11).integers(0, cfg.vocab, (2, 30))
    a = O.forward(cfg, w, tokens, alpha=0.5)
    b = O.forward(cfg, w, tokens, alpha=0.5, forced_idx=a["idx"])
    np.testing.assert_array_equal(a["logits"], b["logits"])
    for layer, idx in a["idx"].items():
        n_in = a["schedule"][layer - 1]
        assert idx.shape == (2, a["schedule"][layer])
        assert np.all(idx[:, -1] == n_in - 1)  # force-kept last row
        assert np.all(np.diff(idx, axis=1) > 0)
    assert np.all(a["kept_pos"][:, -1] == 29)


def test_late_positions_pruned_more_under_causal_attention():
    # Appendix B: with causal attention pruning accumulates toward the end of
    # the sequence (later keys are seen by fewer queries).
    cfg = _cfg(n_layers=2, prune_layers=[1], force_keep_last=False)
    w = _tiny_weights(cfg, seed=4, scale=0.05)
    tokens = np.random.default_rng(12).integers(0, cfg.vocab, (4, 64))
    out = O.forward(cfg, w, tokens, alpha=0.5)
    kept = out["kept_pos"]
    assert kept.mean() < 0.8 * 63 / 2


def test_score_select_norms_and_gather():
    rng = np.random.default_rng(13)
    hid = (rng.standard_normal((3, 20, 16)) * np.exp(rng.standard_normal((3, 20, 1)))).astype(np.float32)
    s, idx, g = O.score_select(hid, 7)
    np.testing.assert_allclose(s, np.linalg.norm(hid.astype(np.float64), axis=-1), rtol=1e-12)
    for b in range(3):
        assert np.array_equal(g[b], hid[b][idx[b]])
        order = np.argsort(-s[b], kind="stable")[:7]
        assert sorted(order.tolist()) == idx[b].tolist()


# ---------------------------------------------------------------- generation

def test_attention_one_query_is_last_row_of_causal_attention():
    rng = np.random.default_rng(21)
    q, k = rng.standard_normal((9, 16)), rng.standard_normal((9, 16))
    P = O.attention_probs(q, k)
    np.testing.assert_allclose(O.attention_probs_one(q[-1], k), P[-1], rtol=1e-13, atol=1e-15)


def test_decode_unpruned_equals_full_forward_of_longer_sequence():
    # accel = 1: prefill L tokens, then generate T; every generated token's
    # logits equal the plain causal decoder's on the L + T sequence.
    cfg = _cfg(prune_layers=[])
    w = _tiny_weights(cfg, seed=5)
    rng = np.random.default_rng(14)
    L, T = 13, 4
    seq = rng.integers(0, cfg.vocab, (2, L + T))
    out = O.generate(cfg, w, seq[:, :L], seq[:, L:], accel=1.0)
    ref = _torch_forward_unpruned(cfg, w, seq, all_rows=True)
    np.testing.assert_allclose(out["prefill"]["logits"][:, -1], ref[:, L - 1], rtol=1e-9, atol=1e-9)
    np.testing.assert_allclose(out["logits"], ref[:, L:], rtol=1e-9, atol=1e-9)
    assert out["cache"]["layers"][1]["k"].shape == (2, L + T, cfg.n_kv_heads, cfg.head_dim)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_decode_over_pruned_cache_equals_masked_longer_sequence(dtype):
    # Sec. 3.3 / Appendix B: a row pruned before layer l is a hidden key in
    # layer l and later.  Generating after a pruned prefill must equal one
    # causal pass over the L + T tokens with exactly those keys hidden (the
    # generated tokens are never hidden).
    cfg = _cfg(dtype=dtype)
    w = _tiny_weights(cfg, seed=6)
    rng = np.random.default_rng(15)
    L, T = 29, 3
    seq = rng.integers(0, cfg.vocab, (2, L + T))
    out = O.generate(cfg, w, seq[:, :L], seq[:, L:], alpha=0.55)
    pre = out["prefill"]
    assert pre["schedule"][-1] < L // 2
    alive = []
    kept = np.tile(np.arange(L), (2, 1))
    for layer in range(1, cfg.n_layers + 1):
        a = np.zeros((2, L + T), bool)
        a[:, L:] = True
        for b in range(2):
            a[b, kept[b]] = True
        alive.append(a)
        np.testing.assert_array_equal(out["cache"]["layers"][layer]["pos"][:, :-T], kept)
        if layer in pre["idx"]:
            kept = np.stack([kept[b][pre["idx"][layer][b]] for b in range(2)])
    if dtype == "f32":
        ref = _torch_forward_unpruned(cfg, w, seq, key_alive=alive, all_rows=True)
        np.testing.assert_allclose(out["logits"], ref[:, L:], rtol=1e-9, atol=1e-9)
    else:
        # the torch composition has no bf16 storage points; compare with the
        # compacted prefill of the L + T tokens in which every layer keeps the
        # prefix rows the prefill kept plus all generated rows
        forced, n_in = {}, L
        for layer in sorted(pre["idx"]):
            idx = pre["idx"][layer]
            forced[layer] = np.concatenate([idx, np.tile(np.arange(n_in, n_in + T), (2, 1))], axis=1)
            n_in = idx.shape[1]
        full = O.forward(cfg, w, seq, alpha=1.0, forced_idx=forced)
        np.testing.assert_array_equal(full["kept_pos"][:, -T:], np.tile(np.arange(L, L + T), (2, 1)))
        assert np.max(np.abs(out["logits"] - full["logits"][:, -T:])) < 2e-2
    # the cache holds, per layer, exactly the rows that layer ran on, then the generated ones
    for layer in range(1, cfg.n_layers + 1):
        pos = out["cache"]["layers"][layer]["pos"]
        assert pos.shape[1] == pre["schedule"][layer - 1] + T
        np.testing.assert_array_equal(pos[:, -T:], np.tile(np.arange(L, L + T), (2, 1)))
        assert np.all(np.diff(pos, axis=1) > 0)


def test_decode_cache_keys_are_the_prefill_keys_of_the_kept_rows():
    # Layer 1 runs on every row; its cached keys must equal layer 1's keys of
    # an unpruned run on the same prefix (pruning only acts after layer 1).
    cfg = _cfg()
    w = _tiny_weights(cfg, seed=7)
    toks = np.random.default_rng(16).integers(0, cfg.vocab, (2, 21))
    a = O.forward(cfg, w, toks, alpha=0.5, collect_cache=True)["cache"]["layers"]
    b = O.forward(_cfg(prune_layers=[]), w, toks, accel=1.0, collect_cache=True)["cache"]["layers"]
    np.testing.assert_array_equal(a[1]["k"], b[1]["k"])
    np.testing.assert_array_equal(a[1]["v"], b[1]["v"])
    assert a[4]["k"].shape[1] < b[4]["k"].shape[1]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_pruning_between_attention_and_mlp_gives_the_same_rows(dtype):
    # The scores come from the layer's attention, and the MLP acts on each row
    # alone, so compacting before the MLP (which then runs on kept rows only)
    # must leave every kept row, index and logit unchanged.
    cfg = _cfg(dtype=dtype)
    w = _tiny_weights(cfg, seed=8)
    tokens = np.random.default_rng(17).integers(0, cfg.vocab, (2, 33))
    a = O.forward(cfg, w, tokens, alpha=0.6)
    cfg2 = _cfg(dtype=dtype, prune_point="attention")
    b = O.forward(cfg2, w, tokens, alpha=0.6)
    # (float64 products over a different number of rows may round differently
    # in the last bit, and in bf16 such a bit can flip a rounding)
    tol = 1e-12 if dtype == "f32" else 2e-2
    for layer in a["idx"]:
        np.testing.assert_array_equal(a["idx"][layer], b["idx"][layer])
        np.testing.assert_allclose(a["scores"][layer], b["scores"][layer], rtol=tol)
    np.testing.assert_array_equal(a["kept_pos"], b["kept_pos"])
    np.testing.assert_allclose(a["logits"], b["logits"], rtol=tol, atol=tol)
    with pytest.raises(ValueError):
        O.forward(_cfg(prune_point="mlp"), w, tokens, alpha=0.6)


# ---------------------------------------------------------------- bidirectional encoder variant

@pytest.mark.parametrize("n,hd", [(1, 8), (9, 16)])
def test_attention_without_mask_matches_sdpa(n, hd):
    rng = np.random.default_rng(30 + n)
    q, k = rng.standard_normal((n, hd)), rng.standard_normal((n, hd))
    P = O.attention_probs(q, k, causal=False)
    tq, tk = torch.from_numpy(q)[None, None], torch.from_numpy(k)[None, None]
    eye = torch.eye(n, dtype=torch.float64)[None, None]
    ref = F.scaled_dot_product_attention(tq, tk, eye, is_causal=False)[0, 0].numpy()
    np.testing.assert_allclose(P, ref, rtol=1e-12, atol=1e-14)
    assert np.all(P > 0)


def test_column_mass_closed_form_uniform_bidirectional():
    # q = 0: every query spreads 1/n over all n keys, so each key collects
    # exactly one unit per query head of its group.
    n, H, G = 10, 4, 2
    P = np.stack([O.attention_probs(np.zeros((n, 8)), np.ones((n, 8)), causal=False) for _ in range(H)])
    np.testing.assert_allclose(O.column_mass(P, G), np.full((G, n), H // G), rtol=1e-13)


def test_bidirectional_forward_matches_torch_composition():
    cfg = _cfg(prune_layers=[], causal=False)
    w = _tiny_weights(cfg, seed=9)
    tokens = np.random.default_rng(18).integers(0, cfg.vocab, (2, 15))
    got = O.forward(cfg, w, tokens, accel=1.0)
    ref = _torch_forward_unpruned(cfg, w, tokens)
    np.testing.assert_allclose(got["logits"], ref, rtol=1e-9, atol=1e-9)
    causal = O.forward(_cfg(prune_layers=[]), w, tokens, accel=1.0)
    # in one layer only the last row would see the same keys under both
    # masks; the first row sees all keys here and one key under the causal mask
    assert np.abs(got["logits"][:, 0] - causal["logits"][:, 0]).max() > 1e-6


def test_bidirectional_compacted_equals_masked_formulation():
    cfg = _cfg(causal=False)
    w = _tiny_weights(cfg, seed=10)
    tokens = np.random.default_rng(19).integers(0, cfg.vocab, (2, 31))
    sched = O.schedule(31, 0.6, cfg.n_layers, cfg.prune_layers, cfg.tau)
    a = O.forward(cfg, w, tokens, alpha=0.6)
    m = O.forward_masked(cfg, w, tokens, sched)
    np.testing.assert_array_equal(a["kept_pos"], m["kept_pos"])
    np.testing.assert_allclose(a["logits"], m["logits"], rtol=1e-9, atol=1e-9)
    with pytest.raises(ValueError):
        O.decode_step(cfg, w, O.forward(cfg, w, tokens, alpha=0.6, collect_cache=True)["cache"],
                      tokens[:, 0])


# ---------------------------------------------------------------- variable-length batches

def test_plan_varlen_reduces_to_plan_and_meets_target():
    cfg = _cfg(n_layers=16, d_model=2048, n_heads=32, n_kv_heads=8, head_dim=64, ffn_dim=8192,
               vocab=128256, prune_layers=list(range(1, 16)))
    for accel in (1.0, 2.0, 4.0, 8.0):
        a1, s1 = O.plan(cfg, 512, accel)
        a2, s2 = O.plan_varlen(cfg, [512], accel)
        assert a1 == a2 and s2 == [s1]
        a3, s3 = O.plan_varlen(cfg, [512] * 5, accel)
        assert s3 == [s1] * 5 and abs(a3 - a1) < 1e-12
    lengths = [512, 37, 2048, 1, 300]
    full = sum(O.model_cost(cfg, O.schedule(L, 1.0, 16, cfg.prune_layers, 5)) for L in lengths)
    prev = 1.0
    for accel in (1.5, 3.0, 6.0):
        alpha, scheds = O.plan_varlen(cfg, lengths, accel)
        cost = sum(O.model_cost(cfg, sc) for sc in scheds)
        assert cost <= full / accel
        worse = [O.schedule(L, min(1.0, alpha + 1e-9), 16, cfg.prune_layers, 5) for L in lengths]
        assert sum(O.model_cost(cfg, sc) for sc in worse) > full / accel or worse == scheds
        for L, sc in zip(lengths, scheds):
            assert sc == O.schedule(L, alpha, 16, cfg.prune_layers, 5)
        assert alpha < prev
        prev = alpha
    # the longest sequence dominates the batch cost: its rate is close to its own
    a_long, _ = O.plan(cfg, 2048, 3.0)
    a_mix, _ = O.plan_varlen(cfg, lengths, 3.0)
    assert abs(a_mix - a_long) < 0.05
    with pytest.raises(ValueError):
        O.plan_varlen(cfg, [10, 0], 2.0)


def test_forward_varlen_runs_each_sequence_at_the_batch_rate():
    cfg = _cfg()
    w = _tiny_weights(cfg, seed=11)
    rng = np.random.default_rng(20)
    seqs = [rng.integers(0, cfg.vocab, n) for n in (23, 5, 40)]
    out = O.forward_varlen(cfg, w, seqs, accel=3.0)
    alpha, scheds = O.plan_varlen(cfg, [23, 5, 40], 3.0)
    assert out["alpha"] == alpha and out["schedule"] == scheds
    for b, t in enumerate(seqs):
        r = O.forward(cfg, w, t[None], alpha=alpha)
        np.testing.assert_array_equal(out["logits"][b], r["logits"][0])
        np.testing.assert_array_equal(out["kept_pos"][b], r["kept_pos"][0])
        assert out["kept_pos"][b][-1] == len(t) - 1


# ---------------------------------------------------------------- sampled rows, per-layer entry, f32 control

@pytest.mark.parametrize("causal", [True, False])
def test_layer_rows_matches_torch_composition(causal):
    # A one-layer model: the head applied to layer_rows' outputs for a few rows
    # must equal those rows' logits from the torch-composed decoder.
    cfg = _cfg(n_layers=1, prune_layers=[], causal=causal)
    w = _tiny_weights(cfg, seed=21)
    tokens = np.random.default_rng(22).integers(0, cfg.vocab, (1, 17))
    ref = _torch_forward_unpruned(cfg, w, tokens, all_rows=True)[0]
    rows = [0, 5, 11, 16]
    h0 = w["embed"][tokens[0]]
    out = O.layer_rows(cfg, w["layers"][0], h0, np.arange(17), rows)
    got = O.head(cfg, w, out, O._Store("f32"))
    np.testing.assert_allclose(got, ref[rows], rtol=1e-9, atol=1e-9)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_layer_rows_equals_rows_of_the_full_layer(dtype):
    # At original positions that skip (as after a compaction), sampled rows of a
    # non-pruning layer equal the same rows of decoder_layer's full output.
    cfg = _cfg(dtype=dtype, prune_layers=[], n_layers=1)
    w = _tiny_weights(cfg, seed=23)
    rng = np.random.default_rng(24)
    h = O.bf16_round(rng.standard_normal((29, cfg.d_model)))
    pos = np.sort(rng.choice(200, 29, replace=False))
    full, pos_out, idx, s = O.decoder_layer(cfg, w["layers"][0], 1, h, pos, 29, O._Store(dtype))
    assert idx is None and s is None and np.array_equal(pos_out, pos)
    rows = [0, 3, 28, 14]
    det = {}
    got = O.layer_rows(cfg, w["layers"][0], h, pos, rows, detail=det)
    if dtype == "f32":
        np.testing.assert_allclose(got, full[rows], rtol=1e-12, atol=1e-12)
    else:  # a different matmul shape may flip a rare bf16 rounding
        assert np.mean(got == full[rows]) > 0.99
        assert np.max(np.abs(got - full[rows])) <= 2.0 ** -7 * np.max(np.abs(full[rows]))
    assert np.array_equal(det["h2"], got) and det["a"].shape == (4, cfg.ffn_dim)


def test_decoder_layer_is_the_forward_step():
    # forward() is decoder_layer applied layer by layer: running the layers by
    # hand from the embedded rows reproduces its logits, indices and scores.
    cfg = _cfg(dtype="bf16")
    w = _tiny_weights(cfg, seed=25)
    tokens = np.random.default_rng(26).integers(0, cfg.vocab, (1, 31))
    ref = O.forward(cfg, w, tokens, alpha=0.6)
    store = O._Store("bf16")
    h, pos = store(w["embed"][tokens[0]]), np.arange(31)
    for layer in range(1, cfg.n_layers + 1):
        h, pos, idx, s = O.decoder_layer(cfg, w["layers"][layer - 1], layer, h, pos, ref["schedule"][layer], store)
        if layer in cfg.prune_layers:
            np.testing.assert_array_equal(idx, ref["idx"][layer][0])
            np.testing.assert_array_equal(s, ref["scores"][layer][0])
    np.testing.assert_array_equal(O.head(cfg, w, h, store), ref["logits"][0])
    np.testing.assert_array_equal(pos, ref["kept_pos"][0])


def test_f32_arithmetic_control_drifts_within_the_format_floor():
    # The control keeps every bf16 storage point and sums in float32: it must
    # really compute in float32 (it differs from the float64 oracle), stay close
    # to it (a few bf16 ulps per layer), and pick the same rows where forced.
    cfg = _cfg(dtype="bf16", n_layers=4, d_model=128, n_heads=4, n_kv_heads=2, head_dim=32,
               ffn_dim=256, vocab=300)
    w = _tiny_weights(cfg, seed=27, scale=0.1)
    tokens = np.random.default_rng(28).integers(0, cfg.vocab, (2, 40))
    ref = O.forward(cfg, w, tokens, alpha=0.7)
    ctl = O.forward(dataclasses.replace(cfg, arith="f32"), w, tokens, alpha=0.7, forced_idx=ref["idx"])
    np.testing.assert_array_equal(ctl["kept_pos"], ref["kept_pos"])
    gap = np.abs(ctl["logits"] - ref["logits"])
    assert gap.max() > 0
    assert gap.mean() <= 2.0 ** -7 * np.sqrt(cfg.n_layers) * ref["logits"].std()
    with pytest.raises(ValueError):
        O.forward(dataclasses.replace(cfg, arith="f16"), w, tokens, alpha=0.7)


def test_pruning_layer_at_several_k_equals_decoder_layer():
    # The full-size tests run one attention branch for several kept counts and
    # the MLP on sampled kept rows; that must be decoder_layer's result.
    from tests.helpers import oracle_pruning_layer_at
    cfg = _cfg(dtype="bf16", prune_point="attention")
    w = _tiny_weights(cfg, seed=29, scale=0.2)
    rng = np.random.default_rng(30)
    h = O.bf16_round(rng.standard_normal((37, cfg.d_model)))
    pos = np.sort(rng.choice(90, 37, replace=False))
    store = O._Store("bf16")
    s, per_k = oracle_pruning_layer_at(cfg, w["layers"][0], h, pos, [37, 20, 7],
                                       lambda k, idx: np.arange(0, k, 2), store)
    for k, (idx, rows, h2, det) in per_k.items():
        ref, pref, iref, sref = O.decoder_layer(cfg, w["layers"][0], 1, h, pos, k, store)
        np.testing.assert_array_equal(idx, iref)
        np.testing.assert_array_equal(s, sref)
        np.testing.assert_array_equal(h2, ref[rows])
        np.testing.assert_array_equal(det["h2"], h2)


# ---------------------------------------------------------------- Appendix B figure mode (reactivation)

def test_marked_mode_logits_are_the_unpruned_decoders_at_the_kept_rows():
    cfg = _cfg(prune_layers=[1, 2, 3])
    w = _tiny_weights(cfg, seed=31)
    tokens = np.random.default_rng(32).integers(0, cfg.vocab, (2, 33))
    sched = O.schedule(33, 0.6, cfg.n_layers, cfg.prune_layers, cfg.tau)
    r = O.forward_marked(cfg, w, tokens, sched)
    ref = _torch_forward_unpruned(cfg, w, tokens, all_rows=True)
    for b in range(2):
        np.testing.assert_allclose(r["logits"][b], ref[b][r["kept_pos"][b]], rtol=1e-9, atol=1e-9)
    for layer in cfg.prune_layers:
        marks = r["kept_by_layer"][layer]
        assert marks.shape == (2, sched[layer])
        assert np.all(np.diff(marks, axis=1) > 0) and np.all(marks[:, -1] == 32)


def test_marked_mode_first_layer_matches_compaction_and_later_layers_reactivate():
    # The first pruning layer sees every row in both modes, so its marks are
    # the compacted forward's choice; later layers rank all rows again, and on
    # random inputs some row marked as pruned comes back.
    cfg = _cfg(prune_layers=[1, 2, 3], n_layers=4)
    w = _tiny_weights(cfg, seed=33)
    tokens = np.random.default_rng(34).integers(0, cfg.vocab, (3, 41))
    alpha = 0.7
    sched = O.schedule(41, alpha, cfg.n_layers, cfg.prune_layers, cfg.tau)
    r = O.forward_marked(cfg, w, tokens, sched)
    c = O.forward(cfg, w, tokens, alpha=alpha)
    np.testing.assert_array_equal(r["kept_by_layer"][1], c["idx"][1])
    np.testing.assert_array_equal(r["scores"][1], c["scores"][1])
    back = 0
    for b in range(3):
        for l in (2, 3):
            back += len(set(r["kept_by_layer"][l][b]) - set(r["kept_by_layer"][l - 1][b]))
    assert back > 0
    # accel 1: nothing is marked, every row's logits are the unpruned ones
    r1 = O.forward_marked(cfg, w, tokens, [41] * 5)
    np.testing.assert_allclose(r1["logits"], _torch_forward_unpruned(cfg, w, tokens, all_rows=True),
                               rtol=1e-9, atol=1e-9)
