"""Host logic of bench.py that needs no GPU: the clock record of the timed
region (median SM clock, maximum clock, throttle reasons seen)."""

import bench


def _sampler(lines):
    c = bench.ClockSampler(0)
    c.lines = list(lines)
    return c.summary()


def test_clock_summary_median_max_and_reasons():
    na, act = "Not Active", "Active"
    lines = [
        f"0, 2070, 2070, 900.1, 0x0, {na}, {na}, {na}, {na}",
        f"0, 1980, 2070, 1400.0, 0x4, {na}, {na}, {na}, {act}",
        f"0, 2070, 2070, 1390.5, 0x0, {na}, {na}, {na}, {na}",
        "garbled line",
        "0, [N/A], 2070, 1.0, 0x0, x, x, x, x",
    ]
    s = _sampler(lines)
    assert s == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}


def test_clock_summary_flags_every_slowdown_kind():
    act = "Active"
    s = _sampler([f"0, 1200, 2070, 700, 0x68, {act}, {act}, {act}, Not Active"])
    assert s["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"]
    assert s["sm_mhz"] == 1200.0


def test_clock_summary_without_samples():
    assert _sampler([]) == {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}


def test_reference_arm_line_on_the_cpu(capsys):
    """The reference arm (the CPU oracle) on the tiny workload: it prints the
    GPU arm's config dict, a measured per-step sample time, and marks the
    extrapolation to the whole step."""
    import argparse
    import json
    args = argparse.Namespace(config="tiny", steps=2, warmup=0, ratio=None, no_graph=False,
                              statistic="mean", value_norm="v", full_context=False,
                              selection="global", reference_step_seconds=0.2)
    bench.run_reference(args)
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["extrapolated"] is True
    assert line["config"] == bench.run_config(args, 256, 25, 1)
    assert 0 < line["ms_per_step"] <= line["extrapolated_full_step_ms"] * 1.5
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["value"] > 0


def test_traffic_lines_match_the_committed_kernels():
    """Every DRAM-traffic line under profiles/ names the source it was captured
    from; the bench reports it only while that source is unchanged, so every
    line must have been captured from the current kernel sources."""
    import os
    src = {"score": "score_tc.cu", "refresh": "refresh_tc.cu"}
    seen = set()
    for line in open(os.path.join(bench.ROOT, "profiles", "traffic.txt")):
        if line.startswith("#") or not line.strip():
            continue
        call, workload, nbytes, digest = line.split()[:4]
        assert float(nbytes) > 0
        got = bench._traffic(call, workload, src[call])
        assert got == (float(nbytes) if digest == bench._src_hash(src[call]) else None)
        if got is not None:
            seen.add((call, workload))
    # the four workloads' refresh lines and the scoring lines of the large ones
    # were all captured from the current sources
    for key in [("refresh", w) for w in ("batched", "multi", "single", "longdoc@0.1")] + \
               [("score", w) for w in ("batched", "multi", "longdoc@0.1")]:
        assert key in seen, key
    assert bench._traffic("refresh", "batched@0.3", "refresh_tc.cu") is None   # no capture at that ratio
