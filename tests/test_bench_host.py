"""Host logic of bench.py that needs no GPU: the ncu traffic record is used
only while the kernel source it was taken on is unchanged, and the clock
samples taken during the timed region are reduced to the median SM clock and
the throttle reasons seen."""
import hashlib

import bench


def _record(path, sha, traffic=1234.0):
    with open(path, "w") as f:
        f.write("# a summary\n\n| kernel | bytes |\n|---|---|\n\n")
        f.write(f"traffic_bytes_per_launch_at_bench_size: {traffic:.0f}\n")
        f.write(f"source_sha256: {sha}\n")
        f.write("note: summed over the kernels of one call\n")


def test_traffic_record_used_while_the_source_is_unchanged(tmp_path, monkeypatch):
    src = tmp_path / "kernel.cu"
    src.write_bytes(b"__global__ void k() {}\n")
    prof = tmp_path / "traffic.md"
    _record(prof, hashlib.sha256(src.read_bytes()).hexdigest(), 6.5e9)
    monkeypatch.setattr(bench, "KERNEL_SRC", str(src))
    monkeypatch.setattr(bench, "PROFILE_TRAFFIC", str(prof))
    traffic, note = bench._traffic_record()
    assert traffic == 6.5e9 and "summed" in note

    src.write_bytes(b"__global__ void k() { /* changed */ }\n")
    traffic, note = bench._traffic_record()
    assert traffic is None and "changed" in note


def test_traffic_record_missing(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "PROFILE_TRAFFIC", str(tmp_path / "absent.md"))
    traffic, note = bench._traffic_record()
    assert traffic is None and "no ncu capture" in note


def test_committed_record_names_a_source_hash():
    with open(bench.PROFILE_TRAFFIC) as f:
        text = f.read()
    assert "source_sha256:" in text and "traffic_bytes_per_launch_at_bench_size:" in text


class _FakeProc:
    def terminate(self):
        pass

    def wait(self, timeout=None):
        return 0

    def kill(self):
        pass


def _reduce(lines):
    s = bench.ClockSampler(0)
    s.proc = _FakeProc()
    s.lines = lines
    return s.stop()


def test_clock_samples_reduced_to_median_and_reasons():
    rows = [
        "0, 2070, 2070, 900.1, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "0, 1980, 2070, 1390.5, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 2055, 2070, 1200.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "garbage line",
        "0, [N/A], 2070, 0, 0x0, Not Active, Not Active, Not Active, Not Active",
    ]
    out = _reduce(rows)
    assert out == {"sm_mhz": 2055.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}


def test_clock_samples_report_thermal_slowdown():
    rows = ["0, 1500, 2070, 1400, 0x40, Not Active, Active, Not Active, Not Active"] * 3
    out = _reduce(rows)
    assert out["reasons"] == ["hw_thermal_slowdown"] and out["sm_mhz"] == 1500.0


def test_clock_sampler_without_samples():
    assert _reduce([]) is None
    assert bench.ClockSampler(0).stop() is None  # never started


def test_end_to_end_block_count_has_a_single_median():
    assert bench.E2E_BLOCKS >= 3 and bench.E2E_BLOCKS % 2 == 1
