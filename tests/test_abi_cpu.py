"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every entry point the header declares, its planner agrees exactly with the
oracle's Eq. 2 / Sec. 3.4 planner, and bad arguments are rejected before any
device work."""

import os
import re

import numpy as np
import pytest

from oracle import zsaa_oracle as O
from paper_2509_01190_gb300 import inputs as I

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "zsaa.h")


def test_library_exports_every_declared_entry_point(zlib):
    text = open(HEADER).read()
    declared = set(re.findall(r"^\s*(?:zsaa_status|void|const char\*)\s+(zsaa_\w+)\s*\(", text, re.M))
    assert declared, "no declarations parsed"
    L = zlib.lib()
    for name in sorted(declared):
        assert hasattr(L, name), name
    assert declared == set(zlib.EXPORTED)
    assert zlib.zsaa_version().startswith("zsaa")


def _oracle_cfg(shape, prune=None):
    return O.OracleConfig(
        n_layers=shape.n_layers, d_model=shape.d_model, n_heads=shape.n_heads,
        n_kv_heads=shape.n_kv_heads, head_dim=shape.head_dim, ffn_dim=shape.ffn_dim,
        vocab=shape.vocab, n_classes=shape.n_classes, rope_theta=shape.rope_theta,
        dtype=shape.dtype, prune_layers=shape.prune_layers() if prune is None else prune,
        plan_mode=shape.plan_mode)


@pytest.mark.parametrize("name", ["tiny", "1b", "1b_cls", "8b"])
def test_planner_matches_oracle_on_workloads(zlib, name):
    wl = I.WORKLOADS[name]
    shape, L = wl["shape"], wl["L"]
    cfg = zlib.config_from_shape(shape)
    ocfg = _oracle_cfg(shape)
    for accel in wl["accels"] + [1.25, 3.0, 16.0, 100.0]:
        sched, alpha = zlib.zsaa_plan_config(cfg, L, accel)
        oalpha, osched = O.plan(ocfg, L, accel)
        assert sched == osched, (name, accel)
        assert alpha == oalpha, (name, accel)
        assert sched[0] == L and all(a >= b for a, b in zip(sched, sched[1:]))


def test_planner_matches_oracle_random_configs(zlib):
    rng = np.random.default_rng(0)
    for _ in range(60):
        n = int(rng.integers(1, 9))
        prune = sorted(set(int(x) for x in rng.integers(1, n + 1, rng.integers(0, n + 1))))
        shape = I.ModelShape("r", n, 64 * int(rng.integers(1, 5)), 4, 2, 16 * int(rng.integers(1, 5)),
                             64 * int(rng.integers(1, 9)), int(rng.integers(16, 5000)),
                             n_classes=int(rng.integers(0, 2)) * 3, dtype="f32",
                             prune=",".join(map(str, prune)) if prune else "none",
                             plan_mode=["cost", "rate"][int(rng.integers(0, 2))])
        cfg = zlib.config_from_shape(shape, tau=int(rng.integers(1, 8)))
        ocfg = _oracle_cfg(shape)
        ocfg.tau = cfg.tau
        L = int(rng.integers(1, 3000))
        accel = float(1 + rng.random() * rng.integers(0, 20))
        sched, alpha = zlib.zsaa_plan_config(cfg, L, accel)
        oalpha, osched = O.plan(ocfg, L, accel)
        assert sched == osched and alpha == oalpha


def test_eq2_golden_via_c_planner(zlib):
    # alpha = 0.3 worked example through the library's rate planner (accel = 1/0.3)
    shape = I.ModelShape("g", 6, 64, 4, 2, 16, 64, 100, dtype="f32", prune="1,2,3,4,5,6",
                         plan_mode="rate")
    sched, alpha = zlib.zsaa_plan_config(zlib.config_from_shape(shape), 1000, 1 / 0.3)
    assert sched[:4] == [1000, 300, 90, 27] and sched[-1] == 5


def test_bad_arguments_rejected_without_device_work(zlib):
    shape = I.LLAMA_1B
    cfg = zlib.config_from_shape(shape)
    with pytest.raises(zlib.ZsaaError) as e:
        zlib.zsaa_plan_config(cfg, 512, 0.5)
    assert e.value.status == zlib.ZSAA_ERR_INVALID_ARG
    with pytest.raises(zlib.ZsaaError) as e:
        zlib.zsaa_plan_config(cfg, 0, 2.0)
    assert e.value.status == zlib.ZSAA_ERR_INVALID_ARG
    bad = zlib.config_from_shape(shape, n_kv_heads=3)
    with pytest.raises(zlib.ZsaaError) as e:
        zlib.zsaa_plan_config(bad, 512, 2.0)
    assert e.value.status == zlib.ZSAA_ERR_INVALID_ARG
    odd = zlib.config_from_shape(shape, head_dim=96)
    with pytest.raises(zlib.ZsaaError) as e:
        zlib.zsaa_plan_config(odd, 512, 2.0)
    assert e.value.status == zlib.ZSAA_ERR_UNSUPPORTED
    fake = 1 << 20  # aligned, never dereferenced: validation fails first
    for B, L, d, k in [(4, 100, 64, 0), (4, 100, 64, 101), (0, 100, 64, 5), (4, 100, 12, 5)]:
        with pytest.raises(zlib.ZsaaError) as e:
            zlib.zsaa_score_select(fake, B, L, d, k, fake, None, stream=0)
        assert e.value.status == zlib.ZSAA_ERR_INVALID_ARG
    with pytest.raises(zlib.ZsaaError) as e:
        zlib.zsaa_score_select(fake + 8, 4, 100, 64, 5, fake, None, stream=0)
    assert e.value.status == zlib.ZSAA_ERR_INVALID_ARG
    with pytest.raises(zlib.ZsaaError):
        zlib.zsaa_op_linear(None, fake, None, None, fake, 4, 16, 64, zlib.ZSAA_BF16, 0, stream=0)


def test_generation_entry_points_reject_null_handles(zlib):
    import ctypes as C
    L = zlib.lib()
    h = C.c_void_p()
    assert L.zsaa_cache_create(None, 1, 16, 2.0, 4, C.byref(h)) == zlib.ZSAA_ERR_INVALID_ARG
    assert h.value is None
    assert L.zsaa_cache_create(None, 1, 16, 2.0, 4, None) == zlib.ZSAA_ERR_INVALID_ARG
    assert L.zsaa_prefill(None, None, None, None, None, None) == zlib.ZSAA_ERR_INVALID_ARG
    assert L.zsaa_decode_step(None, None, None, None, None) == zlib.ZSAA_ERR_INVALID_ARG
    assert L.zsaa_cache_layer(None, 1, None, None, None, None, None, None) == zlib.ZSAA_ERR_INVALID_ARG
    assert L.zsaa_cache_bytes(None, None, None) == zlib.ZSAA_ERR_INVALID_ARG
    L.zsaa_cache_destroy(None)  # no-op


def test_varlen_planner_matches_oracle_exactly(zlib):
    rng = np.random.default_rng(3)
    for name in ("1b", "1b_cls", "8b", "tiny"):
        shape = I.WORKLOADS[name]["shape"]
        cfg = zlib.config_from_shape(shape)
        ocfg = _oracle_cfg(shape)
        for _ in range(6):
            B = int(rng.integers(1, 9))
            lengths = [int(x) for x in rng.integers(1, 2049, B)]
            for accel in (1.0, 1.7, 4.0, 11.0):
                sched, alpha = zlib.zsaa_plan_varlen_config(cfg, lengths, accel)
                oalpha, osched = O.plan_varlen(ocfg, lengths, accel)
                assert alpha == oalpha and sched == osched, (name, lengths, accel)
    with pytest.raises(zlib.ZsaaError) as e:
        zlib.zsaa_plan_varlen_config(zlib.config_from_shape(I.LLAMA_1B), [5, 0], 2.0)
    assert e.value.status == zlib.ZSAA_ERR_INVALID_ARG
