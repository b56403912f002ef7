"""End-to-end parity of the pruned prefill (zsaa_forward / _ex / _host) on the
GPU against the oracle.

Protocol for each small case (the full sizes are in test_gpu_full_size.py):
1. the oracle runs the sampled sequences with its own top-k choices;
2. the GPU runs naturally (idx_out / scores_out hooks): at the first pruning
   layer (identical inputs there) its scores must agree closely with the
   oracle's and its kept set must equal the oracle's outside a narrow band
   around the k-th score;
3. the GPU runs again with forced_idx = the oracle's choices for the sampled
   sequences, so bf16 near-ties cannot flip a selection, and its logits must be
   within max-abs 2e-2 / mean-abs 2e-3 (bf16) or 1e-4 relative (fp32) of the
   oracle's, with identical kept positions.
"""

import dataclasses

import numpy as np
import pytest
import torch

from oracle import zsaa_oracle as O
from paper_2509_01190_gb300 import inputs as I
from tests.helpers import BF16_MAX_ABS, BF16_MEAN_ABS, F32_REL, logits_report, need_gpu, oracle_cfg

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def z(zlib):
    need_gpu()
    return zlib


SMALL_BF16 = I.ModelShape("small-bf16", 3, 256, 4, 2, 64, 512, 1008)
SMALL_BF16_128 = I.ModelShape("small-bf16-hd128", 2, 512, 4, 1, 128, 768, 2000 - 2000 % 16)
SMALL_CLS = dataclasses.replace(SMALL_BF16, name="small-cls", n_classes=4)


def _layers_run(shape, n_run):
    return shape.n_layers if not n_run else n_run


def run_case(z, shape, B, L, accel, seqs, n_run=0, seed_tok=42, oracle_dtype=None):
    """Returns a dict of GPU and oracle results for sequences `seqs`."""
    weights = I.make_weights(shape, device="cuda")
    tokens = I.make_tokens(B, L, shape.vocab, seed=seed_tok)
    tok_dev = torch.from_numpy(tokens).cuda()
    cfg = z.config_from_shape(shape)
    model = z.Model(cfg, weights, B, L)
    sched, alpha = z.zsaa_plan(model, L, accel)
    n_layers = _layers_run(shape, n_run)
    prune = [l for l in shape.prune_layers() if l <= n_layers]
    # --- oracle on the sampled sequences
    wnp = I.weights_to_numpy(weights, layers=list(range(n_layers)))
    ocfg = oracle_cfg(shape, prune_layers=prune, n_layers=n_layers)
    if oracle_dtype:
        ocfg.dtype = oracle_dtype
    ores = O.forward(ocfg, wnp, tokens[seqs], alpha=alpha)
    assert ores["schedule"] == sched[: n_layers + 1]
    # --- GPU natural run
    n_fin = sched[n_layers]
    out_shape = (B, shape.n_classes) if shape.n_classes else (B, n_fin, shape.vocab)
    logits = torch.empty(out_shape, device="cuda", dtype=torch.float32)
    kept = torch.empty(B, n_fin, device="cuda", dtype=torch.int32)
    idx_tot = sum(B * sched[l] for l in prune)
    sc_tot = sum(B * sched[l - 1] for l in prune)
    idx_out = torch.full((max(idx_tot, 1),), -1, device="cuda", dtype=torch.int32)
    sc_out = torch.zeros(max(sc_tot, 1), device="cuda", dtype=torch.float32)
    z.zsaa_forward_ex(model, tok_dev, B, L, accel, logits, kept, scores_out=sc_out, idx_out=idx_out,
                      n_layers_run=n_run)
    z.zsaa_sync(model)
    nat_idx, nat_sc = {}, {}
    oi = osc = 0
    for l in prune:
        nat_idx[l] = idx_out[oi: oi + B * sched[l]].view(B, sched[l]).cpu().numpy()
        nat_sc[l] = sc_out[osc: osc + B * sched[l - 1]].view(B, sched[l - 1]).cpu().numpy()
        oi += B * sched[l]
        osc += B * sched[l - 1]
    nat_logits = logits.cpu().numpy()
    # --- GPU forced run
    forced = []
    for l in prune:
        blk = nat_idx[l].copy()
        for r, b in enumerate(seqs):
            blk[b] = ores["idx"][l][r]
        forced.append(blk.reshape(-1))
    forced_dev = torch.from_numpy(np.concatenate(forced).astype(np.int32)).cuda() if forced else None
    logits2 = torch.empty_like(logits)
    kept2 = torch.empty_like(kept)
    z.zsaa_forward_ex(model, tok_dev, B, L, accel, logits2, kept2, forced_idx=forced_dev,
                      n_layers_run=n_run)
    z.zsaa_sync(model)
    res = dict(model=model, weights=weights, tokens=tokens, sched=sched, alpha=alpha, ores=ores,
               nat_idx=nat_idx, nat_sc=nat_sc, nat_logits=nat_logits, kept_nat=kept.cpu().numpy(),
               forced_logits=logits2.cpu().numpy(), forced_kept=kept2.cpu().numpy(), prune=prune,
               seqs=seqs, tok_dev=tok_dev)
    return res


def check_case(res, dtype):
    ores, seqs = res["ores"], res["seqs"]
    got = res["forced_logits"][seqs]
    ref = ores["logits"]
    np.testing.assert_array_equal(res["forced_kept"][seqs], ores["kept_pos"])
    if dtype == "bf16":
        mx, mean = logits_report(got, ref)
        assert mx <= BF16_MAX_ABS and mean <= BF16_MEAN_ABS, (mx, mean, float(np.std(ref)))
    else:
        scale = float(np.max(np.abs(ref)))
        np.testing.assert_allclose(got, ref, rtol=F32_REL, atol=F32_REL * scale)
    # natural selection at the first pruning layer (identical inputs there):
    # scores agree closely, and kept sets agree outside a band around the
    # k-th score where bf16 rounding may reorder near-ties.
    if not res["prune"]:
        return
    l = res["prune"][0]
    k = res["sched"][l]
    rtol, band = (1e-4, 1e-6) if dtype == "f32" else (2e-2, 1e-2)
    for r, b in enumerate(seqs):
        s_ref = ores["scores"][l][r]
        np.testing.assert_allclose(res["nat_sc"][l][b], s_ref, rtol=rtol, atol=rtol * s_ref.max())
        if k == len(s_ref):
            continue
        order = np.sort(s_ref[:-1])[::-1]
        thr = order[k - 2] if k >= 2 else np.inf
        amb = set(np.nonzero(np.abs(s_ref - thr) <= band * abs(thr))[0].tolist())
        got = set(res["nat_idx"][l][b].tolist()) - amb
        ref = set(ores["idx"][l][r].tolist()) - amb
        assert got == ref, (l, b, sorted(got ^ ref)[:10])


def test_tiny_f32_config(z):
    wl = I.WORKLOADS["tiny"]
    res = run_case(z, wl["shape"], wl["B"], wl["L"], wl["accels"][0], seqs=[0, 1])
    assert res["sched"] == [64, 32, 32]
    check_case(res, "f32")
    # fp32 has no near-tie ambiguity at these sizes: natural choice = oracle choice
    np.testing.assert_array_equal(res["nat_idx"][1], res["ores"]["idx"][1])
    np.testing.assert_allclose(res["nat_logits"], res["ores"]["logits"], rtol=F32_REL,
                               atol=F32_REL * np.abs(res["ores"]["logits"]).max())


@pytest.mark.parametrize("accel", [1.0, 2.0, 4.0, 50.0])
def test_small_bf16_lm(z, accel):
    res = run_case(z, SMALL_BF16, 3, 200, accel, seqs=[0, 1, 2])
    check_case(res, "bf16")
    if accel == 1.0:
        assert res["sched"] == [200] * 4
        np.testing.assert_array_equal(res["kept_nat"], np.tile(np.arange(200), (3, 1)))


def test_small_bf16_hd128(z):
    res = run_case(z, SMALL_BF16_128, 2, 333, 3.0, seqs=[0, 1])
    check_case(res, "bf16")


def test_small_bf16_classifier(z):
    res = run_case(z, SMALL_CLS, 4, 150, 3.0, seqs=[0, 3])
    check_case(res, "bf16")
    assert res["forced_logits"].shape == (4, 4)


def test_edge_lengths(z):
    for L, accel in [(1, 1.0), (1, 8.0), (5, 8.0), (6, 2.0), (65, 1e6)]:
        res = run_case(z, SMALL_BF16, 2, L, accel, seqs=[1])
        check_case(res, "bf16")


def test_forward_host_matches_device(z):
    res = run_case(z, SMALL_BF16, 2, 96, 2.0, seqs=[0])
    model, sched = res["model"], res["sched"]
    B, L = 2, 96
    logits_h = np.zeros((B, sched[-1], SMALL_BF16.vocab), np.float32)
    kept_h = np.zeros((B, sched[-1]), np.int32)
    z.zsaa_forward_host(model, res["tokens"], B, L, 2.0, logits_h, kept_h)
    np.testing.assert_array_equal(logits_h, res["nat_logits"])
    np.testing.assert_array_equal(kept_h, res["kept_nat"])


@pytest.mark.parametrize("vocab", [None, 256])
def test_forward_host_pinned_streams_head(z, vocab):
    # A pinned logits buffer: the LM head runs as column slabs copied to the
    # host while later slabs compute.  Eager, captured and replayed calls (the
    # forward is graph-cached) must all equal the device forward bit for bit;
    # with 256 columns, some of the four slabs are empty.
    shape = SMALL_BF16 if vocab is None else dataclasses.replace(SMALL_BF16, name="small-v256", vocab=vocab)
    res = run_case(z, shape, 2, 96, 2.0, seqs=[0])
    model, sched = res["model"], res["sched"]
    B, L = 2, 96
    tok = torch.from_numpy(np.ascontiguousarray(res["tokens"])).pin_memory()
    logits_h = torch.zeros(B, sched[-1], shape.vocab, dtype=torch.float32).pin_memory()
    kept_h = torch.zeros(B, sched[-1], dtype=torch.int32).pin_memory()
    for _ in range(3):
        logits_h.zero_()
        z.zsaa_forward_host(model, tok, B, L, 2.0, logits_h, kept_h)
        np.testing.assert_array_equal(logits_h.numpy(), res["nat_logits"])
        np.testing.assert_array_equal(kept_h.numpy(), res["kept_nat"])
