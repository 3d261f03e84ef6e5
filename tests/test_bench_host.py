"""Host logic of bench.py that needs no GPU: the reference arm's JSON line, the clock record and
the validity of stored DRAM-traffic figures."""
import os


def test_reference_arm_rank0_prints_one_contract_line(capsys):
    """Rank 0 times the oracle on the host and prints one JSON line with the contract's keys."""
    import argparse
    import json

    import bench
    args = argparse.Namespace(steps=1, warmup=0, impl="reference", gpus=1)
    bench.reference_arm(args, world=1, rank=0)
    lines = [x for x in capsys.readouterr().out.splitlines() if x.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["n_gpus"] == 1 and d["steps"] == 1 and d["warmup"] == 0 and d["higher_is_better"] is True
    assert d["value"] > 0 and d["ms_per_step"] > 0
    assert d["config"] == {"workload": bench.WORKLOAD}
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] == 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_clock_record_summary_from_a_fake_nvidia_smi_log(tmp_path, monkeypatch):
    """The clock record of the timed window: median SM clock, the maximum, and the throttle
    reasons seen active in any sample; malformed or N/A samples are skipped."""
    import bench
    monkeypatch.setenv("FQT1_CLOCKS_DIR", str(tmp_path))
    cs = bench.ClockSampler(3)
    assert cs.path == str(tmp_path / "clocks_gpu3.csv")
    (tmp_path / "clocks_gpu3.csv").write_text(
        "3, 2070, 2070, 410.2, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n"
        "3, 1995, 2070, 1398.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n"
        "3, [N/A], 2070, 400.0, 0x0, Not Active, Not Active, Not Active, Not Active\n"
        "garbage line\n"
        "3, 2070, 2070, 420.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n")
    cs.proc = object()  # stands for the nvidia-smi process that wrote the log
    s = cs.summary()
    assert s == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    (tmp_path / "clocks_gpu3.csv").write_text(
        "3, 1200, 2070, 300.0, 0x0000000000000048, Not Active, Active, Not Active, Not Active\n")
    assert bench.ClockSampler(3).summary()["reasons"] == ["nvidia-smi unavailable"]
    cs2 = bench.ClockSampler(3)
    cs2.proc = object()
    assert cs2.summary()["reasons"] == ["hw_thermal_slowdown"]


def test_stage_traffic_is_null_once_its_kernel_sources_change(tmp_path, monkeypatch):
    """A stored DRAM-traffic figure stands only for the kernel sources it was captured on."""
    import shutil

    import bench
    csrc = tmp_path / "paper_2408_14267_gb300" / "csrc"
    shutil.copytree(os.path.join(bench.ROOT, "paper_2408_14267_gb300", "csrc"), csrc,
                    ignore=shutil.ignore_patterns("*.o", "_build"))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    sha = bench.sources_sha("scq")
    monkeypatch.setitem(bench.TRAFFIC_SOURCES, "scq", sha)
    assert bench.stage_traffic("scq_quantize") == bench.TRAFFIC_BYTES["scq_quantize"]
    assert bench.stage_traffic("no_such_stage") is None
    # one byte more in a file of the group: a new hash, and no traffic figure
    with open(csrc / "quantize.cu", "ab") as f:
        f.write(b"\n")
    assert bench.sources_sha("scq") != sha
    assert bench.stage_traffic("scq_quantize") is None
    # files outside the group do not matter
    monkeypatch.setitem(bench.TRAFFIC_SOURCES, "scq", bench.sources_sha("scq"))
    with open(csrc / "gemm_tc.cu", "ab") as f:
        f.write(b"\n")
    assert bench.stage_traffic("scq_quantize") == bench.TRAFFIC_BYTES["scq_quantize"]


def test_all_cores_oracle_timing():
    """The all-cores CPU baseline: one single-threaded oracle process per core, started together."""
    import bench
    assert bench.host_cores() >= 1
    r = bench.run_oracle_parallel(batch=4, procs=2)
    assert r["cores"] == 2 and r["value"] > 0 and r["wall_s"] > 0
    assert (r["M"], r["K"], r["D"]) == (4 * 64, 2304, 256)
