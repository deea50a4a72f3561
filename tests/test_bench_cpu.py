"""The benchmark's arithmetic, on the CPU: the algorithmic bytes and FLOPs of
a c4 step (both frames read in full, the commit of changed pixels, the fp32
z read-modify-write of the open blocks, the weights; 2 FLOPs per MAC of the
open blocks), the roofline time they give, the replica aggregation, the
lookup of a kernel's DRAM traffic in its ncu summary, and the summary of the
clock samples taken during the timed steps."""
import bench


def test_algorithmic_bytes_and_flops_of_a_c4_step():
    x = 8 * 128 * 128 * 256 * 2                     # one bf16 frame of the 8 streams
    z_block = 8 * 8 * 256 * 4                         # fp32 z of one 8x8 block
    w = 256 * 256 * 3 * 3 * 2
    macs = 8 * 8 * 256 * 256 * 3 * 3
    for active, changed in ((0, 0), (208, 7488), (2048, 131072)):
        b, f, g = bench.algorithmic(active, changed, macs)
        assert b == 2 * x + changed * 512 + 2 * active * z_block + w
        assert g == 2 * x + changed * 512
        assert f == 2.0 * macs * active
    # the 10 % step the bench times: 166.49 MB and 15.70 GFLOP, a 24.9 us roofline at the measured peaks
    b, f, _ = bench.algorithmic(208, 7488, macs)
    assert abs(b / 1e6 - 166.49) < 0.01 and abs(f / 1e9 - 15.70) < 0.01
    t_roof = max(f / (1926.3e12), b / (6691.1e9))
    assert abs(t_roof * 1e6 - 24.88) < 0.01


def test_replica_value_counts_every_rank():
    # stream-frames per second of the whole job: 8 streams per step on every rank
    assert abs(bench.replica_value(1, 30, 1.5) - 8 * 30 / 1.5e-3) < 1e-6
    assert abs(bench.replica_value(4, 30, 1.5) - 4 * 8 * 30 / 1.5e-3) < 1e-6


def test_reference_arm_prints_the_contract_line():
    """`bench.py --impl reference` times the oracle on the host cores for the same metric and prints one
    JSON line with the reference-arm keys."""
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--steps", "1",
                          "--warmup", "0"], capture_output=True, text=True, timeout=300, cwd=root)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC and line["unit"] == bench.UNIT
    assert line["higher_is_better"] is True and line["value"] > 0
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["cpu_baseline"]["value"] == line["value"]


def test_traffic_is_read_only_while_the_profiled_sources_are_unchanged(tmp_path, monkeypatch):
    """The roofline's `traffic` comes from a committed ncu summary, and only while the sha256 it records
    is that of the kernel's current source files; otherwise (or with no summary) it is None."""
    import hashlib
    name, srcs = bench.PROFILE_FILES["step_fused"]
    csrc = tmp_path / "paper_2104_11487_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for i, f in enumerate(srcs):
        (csrc / f).write_bytes(b"source %d\n" % i)
    (tmp_path / "profiles").mkdir()
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_from_profiles("step_fused") is None        # no summary
    digest = hashlib.sha256(b"".join(b"source %d\n" % i for i in range(len(srcs)))).hexdigest()
    summary = tmp_path / "profiles" / ("%s_c4_d10.md" % name)
    summary.write_text("# x\n\nsource_sha256: %s (files)\ndram_bytes_per_launch: 158153472 (read + write)\n" % digest)
    assert bench.traffic_from_profiles("step_fused") == 158153472.0
    (csrc / srcs[0]).write_bytes(b"source 0, edited\n")             # the kernel changed since the capture
    assert bench.traffic_from_profiles("step_fused") is None
    assert bench.traffic_from_profiles("no_such_kernel") is None


def test_clock_samples_summary():
    """The clocks key of the bench line: the median SM clock under load, the highest maximum clock, and
    every throttle reason nvidia-smi reported active in any sample (a run that saw a thermal or hardware
    slowdown is one to reject); samples it could not measure are skipped, a missing power reading only
    drops the power."""
    lines = [
        "0, 2070, 2070, 455.1, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n",
        "0, 1980, 2070, 601.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n",
        "0, 2055, 2070, [N/A], 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n",
        "0, [N/A], [N/A], [N/A], [N/A], [N/A], [N/A], [N/A], [N/A]\n",
        "garbage\n",
    ]
    c = bench.Clocks.summarise(lines)
    assert c["samples"] == 3 and c["sm_mhz"] == 2055.0 and c["sm_max_mhz"] == 2070.0
    assert c["power_w_max"] == 601.0 and c["reasons"] == ["sw_power_cap"]
    hot = bench.Clocks.summarise(["0, 1500, 2070, 700, 0x48, Active, Active, Not Active, Not Active\n"])
    assert hot["reasons"] == ["hw_slowdown", "hw_thermal_slowdown"]
    assert bench.Clocks.summarise([])["sm_mhz"] is None
