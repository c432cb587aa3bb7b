"""Host-side logic of bench.py on CPU: clock-record decoding (against a fake
NVML), the traffic record's source-hash check, algorithmic bytes per element
and the roofline peak lookup."""
import ctypes
import hashlib
import json
import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


def sampler(samples, max_mhz=2070, ok=True):
    s = bench.ClockSampler.__new__(bench.ClockSampler)
    s.samples, s.max_mhz, s.ok = list(samples), max_mhz, ok
    return s


def test_clock_summary_median_and_reasons():
    s = sampler([(2070, 0x0), (2070, 0x1), (1980, 0x4), (2070, 0x0)])
    out = s.summary()
    assert out["sm_mhz"] == 2070 and out["sm_max_mhz"] == 2070 and out["samples"] == 4
    assert out["reasons"] == ["sw_power_cap"]            # gpu_idle is not reported
    out = sampler([(1500, 0x8 | 0x40), (1600, 0x20)]).summary()
    assert out["sm_mhz"] == 1550
    assert set(out["reasons"]) == {"hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"}


def test_clock_summary_without_samples():
    out = sampler([], max_mhz=None, ok=False).summary()
    assert out["sm_mhz"] is None and out["samples"] == 0 and out["source"] == "unavailable"


class FakeNvml:
    """Stands in for libnvidia-ml: read-only queries answered from a script."""

    def __init__(self, clocks, reasons, new_api=True):
        self.clocks, self.reasons, self.new_api = list(clocks), list(reasons), new_api

    def nvmlDeviceGetClockInfo(self, h, kind, ref):
        assert kind == 1                                   # SM clock
        ref._obj.value = self.clocks.pop(0)
        return 0

    def nvmlDeviceGetCurrentClocksEventReasons(self, h, ref):
        if not self.new_api:
            return 13                                      # not supported by this driver
        ref._obj.value = self.reasons.pop(0)
        return 0

    def nvmlDeviceGetCurrentClocksThrottleReasons(self, h, ref):
        ref._obj.value = self.reasons.pop(0)
        return 0


@pytest.mark.parametrize("new_api", [True, False])
def test_clock_read_through_fake_nvml(new_api):
    s = sampler([])
    s.nvml = FakeNvml([2070, 1995], [0x4, 0x0], new_api=new_api)
    s.h = ctypes.c_void_p()
    assert s._read() == (2070, 0x4)
    assert s._read() == (1995, 0x0)


def test_clock_read_failure_gives_no_sample():
    class Broken(FakeNvml):
        def nvmlDeviceGetClockInfo(self, h, kind, ref):
            return 999
    s = sampler([])
    s.nvml, s.h = Broken([], []), ctypes.c_void_p()
    assert s._read() is None


def test_traffic_record_is_dropped_when_sources_change(tmp_path, monkeypatch):
    src = tmp_path / "k.cu"
    src.write_bytes(b"kernel v1")
    (tmp_path / "profiles").mkdir()
    rec = {"source_files": ["k.cu"], "source_sha256": hashlib.sha256(b"kernel v1").hexdigest(),
           "dram_bytes_per_element": 4.25}
    (tmp_path / "profiles" / "r.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_per_launch("r.json", 1000) == 4250
    src.write_bytes(b"kernel v2")
    assert bench.traffic_per_launch("r.json", 1000) is None
    assert bench.traffic_per_launch("missing.json", 1000) is None


def test_committed_traffic_records_are_well_formed():
    for name in ("quantize_group_pipelined_qwen72b_traffic.json",):
        with open(os.path.join(bench.ROOT, "profiles", name)) as f:
            rec = json.load(f)
        assert rec["source_files"] and len(rec["source_sha256"]) == 64
        assert rec["dram_bytes_per_element"] == pytest.approx(
            (rec["dram_read_bytes"] + rec["dram_write_bytes"]) / rec["elements"])
        assert 1.0 < rec["dram_bytes_per_element"] < 6.0
        for fn in rec["source_files"]:
            assert os.path.exists(os.path.join(bench.ROOT, fn)), fn
        if "per_launch" in rec:                # the step's launches add up to the totals
            rd = sum(x["bytes"] for x in rec["per_launch"] if x["metric"] == "dram__bytes_read.sum")
            wr = sum(x["bytes"] for x in rec["per_launch"] if x["metric"] == "dram__bytes_write.sum")
            assert (rd, wr) == (rec["dram_read_bytes"], rec["dram_write_bytes"])


def test_step_schedule_threshold_matches_the_library():
    """QuantizeStep.pipelined describes the library's automatic choice; its
    element threshold is the one the library's grouped launch uses."""
    import re
    from paper_2606_07618_gb300 import step as ST
    src = open(os.path.join(bench.ROOT, "paper_2606_07618_gb300", "csrc", "group_kernels.h")).read()
    m = re.search(r"kPipelineMinElements\s*=\s*int64_t\(1\)\s*<<\s*(\d+);", src)
    assert m is not None
    shift = int(m.group(1))
    step_src = open(ST.__file__).read()
    assert f"self.numel >= 1 << {shift}" in step_src


def test_workload_roofline_terms():
    """Candidates per block, FP32 ops per element and algorithmic HBM bytes of a
    step with in-launch scales (two input reads, codes, scales, weights)."""
    from paper_2606_07618_gb300 import workloads as W

    class T:                                 # stand-in for a device tensor: shape, numel, element size
        def __init__(self, r, c):
            self.shape = (r, c)

        def numel(self):
            return self.shape[0] * self.shape[1]

        def element_size(self):
            return 2
    wl = W.workload("qwen72b-b16-wmse")
    xs = [T(t.rows, t.cols) for t in wl.tensors]
    assert bench.candidates(wl) == 16 and bench.alu_ops_per_elem(wl) == 64
    n = 2 * 8192 * 29568
    assert bench.hbm_bytes(wl, xs) == n * (2 + 2 + 0.5 + 2 / 16) + 4 * (29568 + 8192)
    wl = W.workload("qwen72b-b16-mse")
    assert bench.candidates(wl) == 11 and bench.alu_ops_per_elem(wl) == 33
    wl = W.workload("qwen72b-b64-mse")
    assert bench.candidates(wl) == 16 and bench.alu_ops_per_elem(wl) == 48
    assert bench.hbm_bytes(wl, xs) == n * (2 + 2 + 0.5 + 1 / 64)
    assert bench.WORKLOAD == "qwen72b-b16-wmse"
    assert sorted(bench.LEG_CONFIGS + [bench.WORKLOAD]) == sorted(W.ALL_CONFIGS)


def test_algorithmic_bytes_per_element():
    assert bench.alg_bytes_per_elem() == 2.625                     # bf16, block 16, both scale layouts
    assert bench.alg_bytes_per_elem(both_layouts=False) == 2.5625
    assert bench.alg_bytes_per_elem(block=64, in_bytes=4) == 4.5 + 2 / 64


def test_peak_lookup(tmp_path, monkeypatch):
    (tmp_path / "MEASURED_PEAKS.json").write_text(json.dumps({"hbm_gbs": 6784.8}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.peaks() == (6784.8, "measured")
    os.remove(tmp_path / "MEASURED_PEAKS.json")
    assert bench.peaks() == (6800.0, "fallback")
