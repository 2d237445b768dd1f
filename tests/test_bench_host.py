"""Host-side logic of bench.py (no GPU): an extra row that fails is reported in the JSON line and
does not take the headline measurement down with it."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_failing_extra_is_reported_and_the_others_kept():
    result = {"metric": "m", "value": 1.0}

    def ok():
        return {"row_a": {"GB_s": 1.0}}

    def broken():
        raise RuntimeError("device error in the measurement")

    bench._extra(result, "a", ok)
    bench._extra(result, "b", broken)
    assert result["row_a"] == {"GB_s": 1.0}
    assert result["value"] == 1.0
    assert "RuntimeError: device error" in result["extra_errors"]["b"]
    json.dumps(result)  # still one JSON line


def test_reference_arm_line_on_the_host_cores():
    """The reference arm (the oracle on the host cores, one bounded sample per timed step) prints
    the contract's keys, the same config dict as the GPU arm, no host/device copies, and a step
    time that is the time it actually measured."""
    import argparse

    from paper_2607_15456_gb300 import workloads as W

    args = argparse.Namespace(workload="ouro14_rho4", steps=1, warmup=0, cpu_seconds=2.0)
    line = bench.run_reference(args, 0, 1)
    json.dumps(line)
    w = W.WORKLOADS["ouro14_rho4"]
    lens = W.context_lengths(w)
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["config"] == bench.config_dict(w, lens, 1)
    assert line["unit"] == "tokens/s" and line["higher_is_better"] is True
    assert line["steps"] == 1 and line["warmup"] == 0 and line["extrapolated"] is True
    assert line["value"] > 0 and line["cpu_baseline"]["value"] == line["value"]
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    # steps x ms_per_step is measured time, within the arm's own wall clock
    assert 0 < line["ms_per_step"] * line["steps"] / 1e3 <= line["wall_seconds"] * 1.01
    # the extrapolated full step is longer than the sample it came from
    assert line["full_step_seconds_extrapolated"] > line["ms_per_step"] / 1e3


def test_algorithmic_bytes_per_decode_launch():
    """The roofline's numerator: one decode launch reads every cached token's latents of every
    head once ((r_k + r_v) bf16 values), this loop's W_up^K and W_up^V, and q, k_cur, v_cur, out.
    On the headline batch (H = 16, (96, 160), sum of contexts 54987) that is
    16 * 256 * 2 * 54987 + 16 * 128 * 256 * 2 + 4 * 16 * 16 * 128 * 2 = 451,764,224 bytes; the
    committed DRAM counters are compared with the same figure for each workload."""
    from types import SimpleNamespace

    from paper_2607_15456_gb300 import workloads as W

    with open(os.path.join(ROOT, "profiles", "decode_traffic.json")) as f:
        traffic = json.load(f)
    w = W.WORKLOADS["ouro14_rho4"]
    lens = W.context_lengths(w)
    assert sum(lens) == 54987 and len(lens) == 16
    head = SimpleNamespace(w=w, lens=lens, B=len(lens))
    assert bench.DecodeBench.decode_bytes_per_launch(head) == 451_764_224
    for name, entry in traffic.items():
        w = W.WORKLOADS[name]
        lens = W.context_lengths(w)
        ns = SimpleNamespace(w=w, lens=lens, B=len(lens))
        assert bench.DecodeBench.decode_bytes_per_launch(ns) == entry["algorithmic_bytes_per_launch"], name
        # the measured traffic is within a few percent above the algorithmic bytes: no re-reads
        assert 1.0 <= entry["dram_bytes_per_launch"] / entry["algorithmic_bytes_per_launch"] < 1.05, name
