"""The clock sampler's reading of throttle reasons, checked without a GPU: NVML's reason bits
(the published nvmlClocksEventReason values) and the nvidia-smi CSV fallback are decoded into the
names the bench line reports.  The sampler only reads; nothing here touches a device."""
import os
import tempfile

from paper_2607_24981_gb300.clocks import ClockSampler


class _FakeNvml:
    max_mhz = 2070.0

    def __init__(self, samples):
        self.samples = list(samples)

    def sample(self):
        return self.samples.pop(0) if self.samples else None

    def close(self):
        pass


def test_nvml_reason_bits():
    clk = ClockSampler(0)
    clk.nvml = _FakeNvml([])
    clk.samples = [(2070.0, 0x0), (2070.0, 0x4), (1980.0, 0x4 | 0x8), (2070.0, 0x20 | 0x40)]
    s = clk.summary()
    assert s["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_power_cap", "sw_thermal_slowdown"]
    assert s["sm_mhz"] == 2070.0 and s["sm_min_mhz"] == 1980.0 and s["sm_max_mhz"] == 2070.0
    assert s["samples"] == 4


def test_nvml_clean_run():
    clk = ClockSampler(0)
    clk.nvml = _FakeNvml([])
    clk.samples = [(2070.0, 0x0)] * 5
    s = clk.summary()
    assert s["reasons"] == [] and s["sm_mhz"] == 2070.0


def test_nvidia_smi_csv_fallback():
    """Rows of `nvidia-smi --query-gpu=index,clocks.sm,clocks.max.sm,power.draw,
    clocks_event_reasons.active,hw_slowdown,hw_thermal_slowdown,sw_thermal_slowdown,sw_power_cap`."""
    f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
    f.write("0, 2070, 2070, 950.1, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n")
    f.write("0, 2055, 2070, 1398.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n")
    f.write("garbage line\n")
    f.write("0, 2070, 2070, 1400.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n")
    f.flush()
    clk = ClockSampler(0)
    clk.f = f
    s = clk.summary()
    assert s["reasons"] == ["sw_power_cap"] and s["samples"] == 3
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0
    assert not os.path.exists(f.name)
