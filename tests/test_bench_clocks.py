"""bench.py's clock and traffic records on the host: the NVML sampler against a fake NVML
library (read-only queries: clocks, power, clock-event reasons), the nvidia-smi fallback's CSV
parsing, and the committed ncu traffic record's tie to the kernel sources. No GPU and no driver
library are touched."""
import os
import sys
import time

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


class FakeNvml:
    """The NVML entry points the sampler calls, answering from fixed readings."""

    def __init__(self, sm=(2070, 1965), power_mw=612000, reasons=0x1 | 0x4, max_sm=2070):
        self.sm = list(sm)
        self.i = 0
        self.power_mw = power_mw
        self.reasons = reasons
        self.max_sm = max_sm
        self.handle_index = None
        self.shut = False

    @staticmethod
    def _set(ref, v):
        ref._obj.value = v
        return 0

    def nvmlInit_v2(self):
        return 0

    def nvmlShutdown(self):
        self.shut = True
        return 0

    def nvmlDeviceGetHandleByIndex_v2(self, idx, ref):
        self.handle_index = idx.value
        return self._set(ref, 0x1234)

    def nvmlDeviceGetMaxClockInfo(self, dev, kind, ref):
        assert kind == 1  # the SM clock
        return self._set(ref, self.max_sm)

    def nvmlDeviceGetClockInfo(self, dev, kind, ref):
        assert kind == 1
        v = self.sm[self.i % len(self.sm)]
        self.i += 1
        return self._set(ref, v)

    def nvmlDeviceGetPowerUsage(self, dev, ref):
        return self._set(ref, self.power_mw)

    def nvmlDeviceGetCurrentClocksEventReasons(self, dev, ref):
        return self._set(ref, self.reasons)


def _sample(lib, idx=0, seconds=0.05):
    s = bench.NvmlSampler(idx, lib=lib)
    s.start()
    time.sleep(seconds)
    return s.stop()


def test_nvml_sampler_reports_median_power_and_reasons(monkeypatch):
    monkeypatch.delenv("CUDA_VISIBLE_DEVICES", raising=False)
    lib = FakeNvml(sm=(2070, 2070, 1965), reasons=0x1 | 0x4 | 0x40)
    r = _sample(lib)
    assert r["samples"] >= 3
    assert r["sm_mhz"] in (2070.0, 1965.0) and r["sm_max_mhz"] == 2070.0
    assert r["power_w_max"] == pytest.approx(612.0)
    # idle (0x1) is not a slowdown; power cap and hardware thermal slowdown are named
    assert r["reasons"] == ["hw_thermal_slowdown", "sw_power_cap"]
    assert lib.shut


def test_nvml_sampler_no_reason_and_visible_devices(monkeypatch):
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "5,3")
    lib = FakeNvml(reasons=0)
    r = _sample(lib, idx=1)
    assert lib.handle_index == 3  # CUDA device 1 is NVML device 3
    assert r["reasons"] == []


def test_clock_sampler_falls_back_without_nvml_or_nvidia_smi(monkeypatch):
    monkeypatch.setenv("PATH", "/nonexistent")
    monkeypatch.setattr(bench, "NvmlSampler", lambda *a, **k: (_ for _ in ()).throw(OSError()))
    c = bench.ClockSampler()
    c.start(0)
    r = c.stop(0)
    assert r["sm_mhz"] is None and r["reasons"] == ["nvidia-smi unavailable"]


def test_nvidia_smi_csv_parsing(tmp_path):
    """The fallback keeps this GPU's rows and names the active slowdown reasons."""
    c = bench.ClockSampler()
    c.path = str(tmp_path / "clk.csv")
    with open(c.path, "w") as f:
        f.write("0, 2070, 2070, 580.1, 0x0, Not Active, Not Active, Not Active, Not Active\n")
        f.write("1, 900, 2070, 100.0, 0x8, Active, Not Active, Not Active, Not Active\n")
        f.write("0, 2055, 2070, 610.0, 0x4, Not Active, Not Active, Not Active, Active\n")
        f.write("garbage line\n")

    class Done:
        def terminate(self):
            pass

        def wait(self, timeout=None):
            return 0

    c.proc = Done()
    c.out = open(os.devnull, "w")
    r = c.stop(0)
    assert r["samples"] == 2 and r["sm_max_mhz"] == 2070.0
    assert r["sm_mhz"] == pytest.approx(2062.5)
    assert r["reasons"] == ["sw_power_cap"]  # GPU 1's hw_slowdown is not ours


def test_recorded_traffic_only_for_the_captured_sources(monkeypatch):
    """The roofline's DRAM traffic comes from the committed ncu record only while the kernel
    sources hash to the value it was taken at; otherwise the bench line reports null."""
    import json
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)["mesh3d"]["decode"]
    monkeypatch.setattr(bench, "kernel_source_hash", lambda: rec["source_hash"])
    value, how = bench.recorded_traffic("mesh3d", "decode", how=True)
    assert value == rec["dram_bytes_per_launch"] and "ncu" in how
    monkeypatch.setattr(bench, "kernel_source_hash", lambda: "0" * 16)
    assert bench.recorded_traffic("mesh3d", "decode", how=True) == (None, None)
    assert bench.recorded_traffic("no-such-workload", "decode") is None


def test_tensor_peak_follows_timed_region():
    """A kernel timed over a short region is compared with the burst GEMM peak; only a
    seconds-long timed region, which runs into the power cap as the sustained GEMM loop
    does, takes the sustained peak."""
    peaks = {"bf16_tflops": 1913.9, "bf16_tflops_sustained": 1717.3, "source": "measured"}
    v, kind = bench.tc_peak_for(peaks, 0.054)
    assert v == 1913.9 and kind == "bf16_tflops (measured)"
    v, kind = bench.tc_peak_for(peaks, bench.SUSTAINED_REGION_S - 1e-3)
    assert v == 1913.9
    v, kind = bench.tc_peak_for(peaks, bench.SUSTAINED_REGION_S)
    assert v == 1717.3 and kind == "bf16_tflops_sustained (measured)"
    assert bench.tc_peak_for(peaks, 10.0, bf16=False) == (None, None)


def test_l2_flush_choice_follows_input_size():
    """The chain is timed with the L2 flushed before each step exactly when its streamed
    tensors come near the L2's size (pde2d: 168 MB), and warm where they exceed it twice
    over (longseq, mesh3d); either can be forced, and the line's config says which ran."""
    from paper_2608_11519_gb300 import inputs
    pde, lng, mesh = inputs.get("pde2d"), inputs.get("longseq"), inputs.get("mesh3d")
    assert bench.l2_mode("auto", pde, "flarepp") == "flush"
    assert bench.l2_mode("auto", lng, "flarepp") == "warm"
    assert bench.l2_mode("auto", mesh, "flarepp") == "warm"
    assert bench.l2_mode("warm", pde, "flarepp") == "warm"
    assert bench.l2_mode("flush", mesh, "flarepp") == "flush"
    assert bench.FLUSH_BYTES > bench.L2_BYTES
    assert bench.arm_config(pde, "flarepp", 1)["l2"].startswith("flushed")
    assert bench.arm_config(pde, "flarepp", 1, "warm")["l2"].startswith("warm")
    assert bench.arm_config(mesh, "flarepp", 1)["l2"] == "inputs larger than L2 (no flush)"
