"""Variable-length batches on the GPU (zsaa_forward_varlen) against the
oracle's forward_varlen: one preservation rate for the batch, each sequence
pruned from its own length, packed rows.

Protocol as for fixed lengths: a natural run (scores and kept sets at the first
pruning layer against the oracle's, outside a narrow band around the k-th
score), then a run with the oracle's kept indices forced, whose logits must be
within the stated bf16 tolerance and whose kept positions must be exact.  With
equal lengths the packed forward must reproduce zsaa_forward_ex bit for bit.
"""

import numpy as np
import pytest
import torch

from oracle import zsaa_oracle as O
from paper_2509_01190_gb300 import inputs as I
from tests.helpers import BF16_MAX_ABS, BF16_MEAN_ABS, logits_report, need_gpu, oracle_cfg
from tests.test_gpu_forward import SMALL_BF16, SMALL_BF16_128, SMALL_CLS

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def z(zlib):
    need_gpu()
    return zlib


def _packed(arrs, dtype=np.int32):
    return torch.from_numpy(np.concatenate([np.asarray(a, dtype) for a in arrs])).cuda()


def run_varlen_case(z, shape, lengths, accel, seed=42):
    B, Lmax = len(lengths), max(lengths)
    weights = I.make_weights(shape, device="cuda")
    toks = I.make_tokens(B, Lmax, shape.vocab, seed=seed)
    seqs = [toks[b, :L] for b, L in enumerate(lengths)]
    model = z.Model(z.config_from_shape(shape), weights, B, Lmax)
    sched, alpha = z.zsaa_plan_varlen(model, lengths, accel)
    ocfg = oracle_cfg(shape)
    ores = O.forward_varlen(ocfg, I.weights_to_numpy(weights), seqs, accel=accel)
    assert ores["alpha"] == alpha and ores["schedule"] == sched
    n = shape.n_layers
    prune = shape.prune_layers()
    tok = _packed(seqs)
    n_fin = sum(sc[n] for sc in sched)
    out_shape = (B, shape.n_classes) if shape.n_classes else (n_fin, shape.vocab)
    idx_tot = sum(sum(sc[l] for sc in sched) for l in prune)
    sc_tot = sum(sum(sc[l - 1] for sc in sched) for l in prune)
    logits = torch.empty(out_shape, device="cuda", dtype=torch.float32)
    kept = torch.empty(n_fin, device="cuda", dtype=torch.int32)
    idx_out = torch.full((max(idx_tot, 1),), -1, device="cuda", dtype=torch.int32)
    sc_out = torch.zeros(max(sc_tot, 1), device="cuda", dtype=torch.float32)
    z.zsaa_forward_varlen(model, tok, lengths, accel, logits, kept, scores_out=sc_out, idx_out=idx_out)
    z.zsaa_sync(model)
    nat_idx, nat_sc = {}, {}
    oi = osc = 0
    for l in prune:
        ki = [sc[l] for sc in sched]
        ni = [sc[l - 1] for sc in sched]
        flat_i = idx_out[oi: oi + sum(ki)].cpu().numpy()
        flat_s = sc_out[osc: osc + sum(ni)].cpu().numpy()
        nat_idx[l] = np.split(flat_i, np.cumsum(ki)[:-1])
        nat_sc[l] = np.split(flat_s, np.cumsum(ni)[:-1])
        oi += sum(ki)
        osc += sum(ni)
    forced = [np.concatenate(ores["idx"][l]) for l in prune if l in ores["idx"]]
    forced_dev = _packed(forced) if forced else None
    logits2 = torch.empty_like(logits)
    kept2 = torch.empty_like(kept)
    z.zsaa_forward_varlen(model, tok, lengths, accel, logits2, kept2, forced_idx=forced_dev)
    z.zsaa_sync(model)
    return dict(model=model, sched=sched, ores=ores, nat_idx=nat_idx, nat_sc=nat_sc, prune=prune,
                nat_logits=logits.cpu().numpy(), forced_logits=logits2.cpu().numpy(),
                forced_kept=kept2.cpu().numpy(), tok=tok, weights=weights, seqs=seqs)


def check_varlen(res, shape):
    ores = res["ores"]
    if shape.n_classes:
        ref = np.stack(ores["logits"])
    else:
        ref = np.concatenate(ores["logits"], axis=0)
    np.testing.assert_array_equal(res["forced_kept"], np.concatenate(ores["kept_pos"]))
    mx, mean = logits_report(res["forced_logits"], ref)
    assert mx <= BF16_MAX_ABS and mean <= BF16_MEAN_ABS, (mx, mean)
    if not res["prune"]:
        return
    l = res["prune"][0]
    for b, s_ref in enumerate(ores["scores"][l]):
        np.testing.assert_allclose(res["nat_sc"][l][b], s_ref, rtol=2e-2, atol=2e-2 * s_ref.max())
        k = res["sched"][b][l]
        if k == len(s_ref):
            np.testing.assert_array_equal(res["nat_idx"][l][b], np.arange(k))
            continue
        order = np.sort(s_ref[:-1])[::-1]
        thr = order[k - 2] if k >= 2 else np.inf
        amb = set(np.nonzero(np.abs(s_ref - thr) <= 1e-2 * abs(thr))[0].tolist())
        got = set(res["nat_idx"][l][b].tolist()) - amb
        want = set(ores["idx"][l][b].tolist()) - amb
        assert got == want, (b, sorted(got ^ want)[:10])


@pytest.mark.parametrize("accel", [1.0, 3.0])
def test_varlen_small_lm(z, accel):
    lengths = [37, 150, 1, 90, 64]
    res = run_varlen_case(z, SMALL_BF16, lengths, accel)
    check_varlen(res, SMALL_BF16)
    if accel == 1.0:
        assert all(sc == [L] * (SMALL_BF16.n_layers + 1) for sc, L in zip(res["sched"], lengths))


def test_varlen_small_hd128_and_classifier(z):
    check_varlen(run_varlen_case(z, SMALL_BF16_128, [333, 129, 7], 2.5), SMALL_BF16_128)
    res = run_varlen_case(z, SMALL_CLS, [20, 77, 150, 5], 3.0)
    check_varlen(res, SMALL_CLS)
    assert res["forced_logits"].shape == (4, 4)


def test_varlen_equal_lengths_reproduces_fixed_forward(z):
    B, L, accel = 3, 130, 2.5
    weights = I.make_weights(SMALL_BF16, device="cuda")
    toks = I.make_tokens(B, L, SMALL_BF16.vocab, seed=5)
    model = z.Model(z.config_from_shape(SMALL_BF16), weights, B, L)
    sched, _ = z.zsaa_plan(model, L, accel)
    n_fin = sched[-1]
    a = torch.empty(B, n_fin, SMALL_BF16.vocab, device="cuda", dtype=torch.float32)
    ka = torch.empty(B, n_fin, device="cuda", dtype=torch.int32)
    tok = torch.from_numpy(toks).cuda()
    z.zsaa_forward_ex(model, tok, B, L, accel, a, ka)
    b = torch.empty(B * n_fin, SMALL_BF16.vocab, device="cuda", dtype=torch.float32)
    kb = torch.empty(B * n_fin, device="cuda", dtype=torch.int32)
    z.zsaa_forward_varlen(model, tok.reshape(-1), [L] * B, accel, b, kb)
    z.zsaa_sync(model)
    np.testing.assert_array_equal(ka.cpu().numpy().reshape(-1), kb.cpu().numpy())
    np.testing.assert_array_equal(a.cpu().numpy().reshape(B * n_fin, -1), b.cpu().numpy())


def test_varlen_rejects_bad_arguments(z):
    weights = I.make_weights(SMALL_BF16, device="cuda")
    model = z.Model(z.config_from_shape(SMALL_BF16), weights, 2, 50)
    tok = torch.zeros(100, device="cuda", dtype=torch.int32)
    out = torch.empty(100, SMALL_BF16.vocab, device="cuda", dtype=torch.float32)
    for lengths in ([10, 0], [51, 3], [10, 10, 10]):
        with pytest.raises(z.ZsaaError) as e:
            z.zsaa_forward_varlen(model, tok, lengths, 2.0, out)
        assert e.value.status == z.ZSAA_ERR_INVALID_ARG
    tiny = I.WORKLOADS["tiny"]["shape"]
    mt = z.Model(z.config_from_shape(tiny), I.make_weights(tiny, device="cuda"), 2, 50)
    with pytest.raises(z.ZsaaError) as e:
        z.zsaa_forward_varlen(mt, tok, [10, 20], 2.0, out)
    assert e.value.status == z.ZSAA_ERR_UNSUPPORTED
