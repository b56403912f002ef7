"""Host-side logic of bench.py, checked without a GPU:
* the per-class GEMM bounds of a forward against the oracle's own FLOP model
  (Sec. 3.4 cost, R5) and their monotonicity in the kept rows;
* the nvidia-smi clock summary on a recorded sample file (median clock,
  maximum, throttle reasons that were active in any sample);
* the DRAM-traffic record, reported only while its sources are unchanged.
"""

import hashlib
import os

import numpy as np

import bench
from oracle import zsaa_oracle as O
from paper_2509_01190_gb300 import inputs as I

GEMM_CLASSES = ("gemm_qkv_rope", "gemm_o_resid", "gemm_gate_up_swiglu", "gemm_down_resid")


def test_class_flops_at_accel_one_equal_the_oracle_linear_flops():
    for name in ("1b", "8b", "1b_cls"):
        wl = I.WORKLOADS[name]
        sh, B, L = wl["shape"], wl["B"], wl["L"]
        cfg = bench.oracle_config(sh)
        sched = [L] * (sh.n_layers + 1)
        cls = bench.gemm_class_bounds(sh, B, sched, 1000.0, 5000.0)
        got = sum(cls[c]["flops"] for c in GEMM_CLASSES)
        assert got == B * sh.n_layers * L * O.layer_flops_per_row(cfg), name
        if sh.n_classes:
            assert "gemm_lm_head" not in cls
        else:
            # the oracle's cost minus its attention term is the linear layers plus the head
            attn = sh.n_layers * 2 * L * L * sh.n_heads * sh.head_dim
            head = B * (O.model_cost(cfg, sched) - attn) - got
            assert cls["gemm_lm_head"]["flops"] == head, name
        for c in cls.values():
            assert c["launches"] in (1, sh.n_layers)


def test_class_bounds_are_roofline_maxima_and_shrink_with_the_kept_rows():
    wl = I.WORKLOADS["8b"]
    sh, B, L = wl["shape"], wl["B"], wl["L"]
    cfg = bench.oracle_config(sh)
    prev = None
    for accel in (1.0, 2.0, 4.0, 8.0, 11.0):
        _, sched = O.plan(cfg, L, accel)
        cls = bench.gemm_class_bounds(sh, B, sched, 1722.0, 6776.0)
        for c in cls.values():
            # never below the tensor-core time of its FLOPs
            assert c["bound_ms"] >= c["flops"] / 1722e12 * 1e3 * (1 - 1e-12)
        # a compute-only peak gives the FLOP time exactly
        inf_bw = bench.gemm_class_bounds(sh, B, sched, 1722.0, 1e30)
        for k, c in inf_bw.items():
            assert np.isclose(c["bound_ms"], c["flops"] / 1722e12 * 1e3, rtol=1e-12), k
        if prev is not None:
            for k in cls:
                assert cls[k]["flops"] <= prev[k]["flops"] and cls[k]["bound_ms"] <= prev[k]["bound_ms"] + 1e-12
        prev = cls


def test_clock_summary_of_a_recorded_sample(tmp_path):
    rows = [
        "0, 1980, 2070, 950.5, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 1935, 2070, 1012.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 2070, 2070, 600.25, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "garbled line",
    ]
    p = tmp_path / "clocks.csv"
    p.write_text("\n".join(rows) + "\n")
    s = bench.ClockSampler(0)
    s.path = str(p)
    out = s.summary()
    assert out["sm_mhz"] == 1980.0 and out["sm_max_mhz"] == 2070.0
    assert out["reasons"] == ["sw_power_cap"] and out["samples"] == 3
    assert out["power_w_max"] == 1012.0
    assert not p.exists()  # the sample file is removed after reading

    p.write_text("0, 1500, 2070, 700, 0x8, Not Active, Active, Not Active, Not Active\n")
    s.path = str(p)
    assert bench.ClockSampler.summary(s)["reasons"] == ["hw_thermal_slowdown"]

    s.path = str(tmp_path / "missing.csv")
    assert s.summary()["reasons"] == ["no nvidia-smi samples"]


def test_traffic_record_only_while_its_sources_are_unchanged(tmp_path, monkeypatch):
    src = tmp_path / "kernel.cu"
    src.write_text("// kernel source\n")
    rec = {"launch": "a launch", "bytes": 123.0, "algorithmic_bytes": 100.0,
           "sources": {str(src): hashlib.sha256(src.read_bytes()).hexdigest()}}
    monkeypatch.setattr(bench, "TRAFFIC", {("k", "w"): rec})
    assert bench.measured_traffic("k", "w") == {"bytes": 123.0, "launch": "a launch", "algorithmic_bytes": 100.0}
    assert bench.measured_traffic("k", "other") is None
    src.write_text("// kernel source, changed\n")
    assert bench.measured_traffic("k", "w") is None
    os.remove(src)
    assert bench.measured_traffic("k", "w") is None
