"""The tiled GEMM's work decomposition, checked on the host through the C ABI
(zsaa_gemm_schedule runs the launch path's own tile plan and its units' work
iterator, without device work).

For every projection and LM-head shape of the 1B, classifier and 8B forwards
at each acceleration factor of their sweeps, on a GB300 (152 SMs, 76 CTA
pairs, the library's 256-slot split-K workspace), with the pair kernel or the
workspace taken away, and for seeded random shapes and device sizes:
* every k-block of every output tile is computed exactly once;
* a split tile has one final part, which adds exactly the partials of its
  other parts, each from its own slot, in ascending k order (so the sum order
  is fixed), and every slot and flag lies inside the workspace;
* no more units than the device runs at once, and no unit can wait forever:
  running every unit's items in order, each final part waiting for its
  partials, always completes (the kernels' flag waits are bounded, but a plan
  that needed the bound would be wrong).
"""

import numpy as np
import pytest

from paper_2509_01190_gb300 import inputs as I

GB300 = dict(sms=152, pair_slots=76, split_slots=256)
EPI = {"store": 0, "resid": 1, "swiglu": 2, "f32": 3, "rope": 4}
KINDS = ("whole", "partial", "final")


def check_schedule(z, epi, M, N, K, hd=64, sms=152, pair_slots=76, split_slots=256):
    plan, items = z.zsaa_gemm_schedule(epi, M, N, K, hd, sms, pair_slots, split_slots)
    BN, pairs, units, m_tiles, n_tiles, num_kb, total = plan[:7]
    tag = f"epi={epi} M={M} N={N} K={K} sms={sms} pairs={pair_slots} slots={split_slots}: {plan}"
    rows = 256 if pairs else 128
    vn = 2 * N if epi == EPI["swiglu"] else N
    assert m_tiles == -(-M // rows) and n_tiles == -(-vn // BN) and num_kb == K // 64, tag
    assert total == m_tiles * n_tiles, tag
    assert 1 <= units <= (pair_slots if pairs else sms), tag
    if pairs:
        assert BN == 256 and pair_slots > 0, tag

    cover = np.zeros((total, num_kb), np.int32)
    per_unit = [[] for _ in range(units)]
    by_tile = {}
    for it in items:
        u, t, kb0, kb1, kind, slot, count, stride = it
        assert 0 <= u < units and 0 <= t < total and 0 <= kb0 < kb1 <= num_kb, (tag, it)
        assert kind in (0, 1, 2), (tag, it)
        cover[t, kb0:kb1] += 1
        per_unit[u].append(it)
        by_tile.setdefault(t, []).append(it)
    assert np.all(cover == 1), tag

    # split tiles: one final part adding exactly the other parts' slots, in k order
    written = {}
    for t, its in by_tile.items():
        kinds = sorted(i[4] for i in its)
        if kinds == [0]:
            assert its[0][2] == 0 and its[0][3] == num_kb, (tag, its)
            continue
        assert split_slots > 0, (tag, its)
        assert 0 not in kinds and kinds.count(2) == 1 and kinds.count(1) == len(its) - 1, (tag, its)
        final = next(i for i in its if i[4] == 2)
        parts = {i[5]: i for i in its if i[4] == 1}
        assert len(parts) == len(its) - 1, (tag, its)  # one slot per part
        awaited = [final[5] + c * final[7] for c in range(final[6])]
        assert sorted(awaited) == sorted(parts), (tag, its)
        ks = [parts[s][2] for s in awaited]
        assert ks == sorted(ks), (tag, its)
        for s, i in parts.items():
            assert s not in written, (tag, i, written[s])
            written[s] = i
    # every slot and its four flags inside the workspace (a pair's CTA r uses slot 2s + r)
    cap = min(split_slots, 256)
    for s in written:
        top = 2 * s + 1 if pairs else s
        assert 0 <= top < cap, (tag, s)

    # run the units: a final part proceeds once all its partials are written
    done_slots, pos = set(), [0] * units
    progress = True
    while progress:
        progress = False
        for u in range(units):
            while pos[u] < len(per_unit[u]):
                _, t, kb0, kb1, kind, slot, count, stride = per_unit[u][pos[u]]
                if kind == 2 and not all(slot + c * stride in done_slots for c in range(count)):
                    break
                if kind == 1:
                    done_slots.add(slot)
                pos[u] += 1
                progress = True
    assert all(pos[u] == len(per_unit[u]) for u in range(units)), (tag, pos)
    return plan, items


def forward_shapes(z):
    """(epilogue, M, N, K, hd) of every GEMM of the bench's forwards."""
    out = set()
    for name in ("1b", "1b_cls", "8b"):
        wl = I.WORKLOADS[name]
        sh, B, L = wl["shape"], wl["B"], wl["L"]
        cfg = z.config_from_shape(sh)
        d, hd, F = sh.d_model, sh.head_dim, sh.ffn_dim
        qkv = (sh.n_heads + 2 * sh.n_kv_heads) * hd
        for accel in wl["accels"]:
            sched, _ = z.zsaa_plan_config(cfg, L, accel)
            for n in sorted(set(sched)):
                M = B * n
                out |= {(EPI["rope"], M, qkv, d, hd), (EPI["resid"], M, d, sh.n_heads * hd, hd),
                        (EPI["swiglu"], M, F, d, hd), (EPI["resid"], M, d, F, hd)}
            if not sh.n_classes:
                out.add((EPI["f32"], B * sched[-1], sh.vocab, d, hd))
    return sorted(out)


@pytest.mark.parametrize("device", ["gb300", "no_pairs", "no_workspace"])
def test_forward_gemm_schedules(zlib, device):
    dev = dict(GB300)
    if device == "no_pairs":
        dev["pair_slots"] = 0
    if device == "no_workspace":
        dev["split_slots"] = 0
    shapes = forward_shapes(zlib)
    assert len(shapes) > 100
    kinds = set()
    for epi, M, N, K, hd in shapes:
        _, items = check_schedule(zlib, epi, M, N, K, hd, **dev)
        kinds |= {i[4] for i in items}
    # the GB300 plans exercise whole tiles and both splits' partial hand-offs
    assert kinds == ({0} if device == "no_workspace" else {0, 1, 2})


def test_gb300_plans_of_known_shapes(zlib):
    # 8B down projection at 1536 rows: 96 pair tiles on 76 pairs, the 20 of
    # the ragged last wave cut into 3 aligned parts of the 224 k-blocks
    plan, items = check_schedule(zlib, EPI["resid"], 1536, 4096, 14336)
    assert plan[:11] == [256, 1, 76, 6, 16, 224, 96, 76, 0, 20, 3]
    assert sum(1 for i in items if i[4] == 2) == 20
    # 8B O projection at 744 rows: one wave of 48 whole pair tiles
    plan, items = check_schedule(zlib, EPI["resid"], 744, 4096, 4096)
    assert plan[:11] == [256, 1, 48, 3, 16, 64, 48, 48, 0, 0, 1]
    assert all(i[4] == 0 for i in items)
    # 1B QKV + RoPE at 4096 rows (short K): whole tiles only
    plan, items = check_schedule(zlib, EPI["rope"], 4096, 3072, 2048, 64)
    assert all(i[4] == 0 for i in items)


def test_random_shapes_and_devices(zlib):
    rng = np.random.default_rng(2509)
    for _ in range(400):
        epi = int(rng.integers(0, 5))
        M = int(rng.choice([rng.integers(1, 600), rng.integers(1, 9000)]))
        N = 16 * int(rng.integers(1, 1200))
        K = 64 * int(rng.integers(1, 260))
        hd = int(rng.choice([32, 64, 128]))
        sms = int(rng.choice([1, 3, 16, 100, 132, 152]))
        pair_slots = int(rng.choice([0, 1, 5, 66, 76]))
        split_slots = int(rng.choice([0, 7, 64, 256]))
        check_schedule(zlib, epi, M, N, K, hd, sms, pair_slots, split_slots)


def test_schedule_rejects_bad_arguments(zlib):
    with pytest.raises(zlib.ZsaaError):
        zlib.zsaa_gemm_schedule(0, 100, 100, 4096, 0, 152, 76, 256)  # N % 16
    with pytest.raises(zlib.ZsaaError):
        zlib.zsaa_gemm_schedule(0, 100, 256, 100, 0, 152, 76, 256)  # K % 64
    with pytest.raises(zlib.ZsaaError):
        zlib.zsaa_gemm_schedule(4, 100, 256, 256, 48, 152, 76, 256)  # RoPE head size
    with pytest.raises(zlib.ZsaaError):
        zlib.zsaa_gemm_schedule(0, 100, 256, 256, 0, 0, 76, 256)  # no SMs
    with pytest.raises(zlib.ZsaaError):
        zlib.zsaa_gemm_schedule(5, 100, 256, 256, 0, 152, 76, 256)  # epilogue
    with pytest.raises(zlib.ZsaaError):
        zlib.zsaa_gemm_schedule(0, 2 ** 31 - 1, 2 ** 30, 64, 0, 152, 76, 256)  # tile count
