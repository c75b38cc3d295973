"""The benchmark's host-side arithmetic, without a GPU: the algorithmic FLOPs and bytes
of each workload (the roofline's numerators), the roofline fractions, the committed DRAM
traffic lookup and the clock-record parsing that decides whether a run is kept."""
import json
import os

import numpy as np
import pytest

import bench
import workloads


@pytest.mark.parametrize("name,gflops", [("c0", 2.43), ("c1", 172.9), ("c2", 38.9), ("c3", 631.4), ("c4", 1507.5)])
def test_layer_flops(name, gflops):
    """router 2 T d E + experts 4 T k d h + shared 4 T d h_s (GELU workloads)."""
    c = workloads.CONFIGS[name]
    w = bench.layer_work(c, np.ones(c.E, np.int64))
    assert w["flops"] / 1e9 == pytest.approx(gflops, rel=2e-3)   # the values printed to 4 digits
    assert w["flops_up_gemm"] == w["flops_down_gemm"] == 2.0 * c.T * c.k * c.d * c.h


def test_layer_bytes_count_touched_experts_only():
    """Only experts that receive rows are read: an empty expert drops 2 d h bf16 weights."""
    c = workloads.CONFIGS["c2"]
    full = bench.layer_work(c, np.ones(c.E, np.int64))
    counts = np.ones(c.E, np.int64)
    counts[:3] = 0
    part = bench.layer_work(c, counts)
    assert full["bytes"] - part["bytes"] == 3 * 2 * c.d * c.h * 2
    assert part["touched_experts"] == c.E - 3
    # c2 streams its 302 MB of expert weights: the layer's bytes are about 309 MB
    assert 300e6 < full["bytes"] < 315e6


def test_swiglu_and_folded_shared_expert_flops():
    c = workloads.CONFIGS["pB"]   # SwiGLU, h_s = h: one always-on group in the routed launches
    w = bench.layer_work(c, np.ones(c.E, np.int64), shared_groups=1)
    assert w["flops_up_gemm"] == 4.0 * c.T * c.k * c.d * c.h + 2 * 2.0 * c.T * c.d * c.h
    assert w["flops_down_gemm"] == 2.0 * c.T * c.k * c.d * c.h + 2.0 * c.T * c.d * c.h
    assert w["flops"] == 2.0 * c.T * c.d * c.E + 6.0 * c.T * c.k * c.d * c.h + 6.0 * c.T * c.d * c.h_s


def test_summarise_fractions():
    c = workloads.CONFIGS["c4"]
    work = bench.layer_work(c, np.ones(c.E, np.int64))
    stages = {"route": 0.3, "permute": 0.05, "y_init": 0.002, "up_gemm": 0.65, "down_gemm": 0.95, "finalize": 0.1}
    pk = {"hbm_gbs": 6682.5, "bf16_tflops": 1916.0, "bf16_tflops_sustained": 1732.6, "source": "measured"}
    roof, layer, value = bench.summarise(c, {"stages": stages, "work": work, "ms": 2.0}, pk, 1)
    assert roof["kernel"].endswith("(down_gemm)") and roof["bound"] == "tensor" and roof["unit"] == "TFLOP/s"
    assert roof["achieved"] == pytest.approx(work["flops_down_gemm"] / 0.95e-3 / 1e12)
    assert roof["frac"] == pytest.approx(roof["achieved"] / 1916.0)
    assert layer["frac"] == pytest.approx(layer["roofline_us"] * 1e-6 / 2.0e-3)
    assert value == pytest.approx(c.T / 2.0e-3)
    assert bench.summarise(c, {"stages": stages, "work": work, "ms": 2.0}, pk, 4)[2] == pytest.approx(4 * value)


def test_committed_traffic_lookup():
    """profiles/grouped_gemm_dram_traffic.json holds per-launch DRAM bytes for the GEMM
    sources it names: the bench reports them while those sources are unchanged, and null
    once they differ (the counters then describe another kernel)."""
    rec = json.load(open(bench.TRAFFIC_FILE))
    current = rec["sources_sha256"] == bench.gemm_sources_hash()
    for name in ("c1", "c2", "c3", "c4"):
        for stage in ("up_gemm", "down_gemm"):
            t = bench.captured_traffic(name, stage)
            if current:
                assert t == float(rec["workloads"][name][stage]["dram_bytes"]) and t > 0
            else:
                assert t is None
    assert bench.captured_traffic("c0", "up_gemm") is None


def test_clock_record_parsing(tmp_path):
    s = bench.ClockSampler(0)
    s.proc = object()   # a sampler that ran
    s.path = str(tmp_path / "clocks.csv")
    rows = ["0, 2070, 2070, 900, 0x0, Not Active, Not Active, Not Active, Not Active",
            "0, 2070, 2070, 1100, 0x4, Not Active, Not Active, Not Active, Active",
            "0, 345, 2070, 100, 0x0, Not Active, Not Active, Not Active, Not Active"]
    with open(s.path, "w") as f:
        f.write("\n".join(rows) + "\n")
    out = s.summary()
    assert out["sm_mhz"] == 2070.0 and out["sm_max_mhz"] == 2070.0   # idle samples left out
    assert out["reasons"] == ["sw_power_cap"]
    assert not os.path.exists(s.path)
