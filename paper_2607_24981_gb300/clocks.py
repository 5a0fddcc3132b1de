"""SM clock and throttle-reason samples taken while a timed region runs.

    with ClockSampler(device_index) as clk:
        ...timed work...
    clk.summary()  -> {"sm_mhz": median, "sm_max_mhz": ..., "reasons": [...], "samples": n, "source": ...}

The samples come from NVML (the driver's management library, read through ctypes) every 2 ms on
a background thread, so even a timed region of a few milliseconds is covered; without NVML, from
`nvidia-smi -lms 200`.  A run that saw hw_slowdown, hw_thermal_slowdown or sw_thermal_slowdown, or SM
clocks stuck well below the maximum with no reason, is not a valid measurement; sw_power_cap is
reported and kept.  The sampler only reads clocks and reasons; it changes no setting of the GPU.
"""
from __future__ import annotations

import ctypes
import os
import statistics
import subprocess
import tempfile
import threading
import time

# clocks-event reason bits of NVML (nvmlClocksEventReason*)
_REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
            0x80: "hw_power_brake_slowdown"}
_NVML_CLOCK_SM = 1


class _Nvml:
    """The few NVML calls the sampler needs (read-only queries)."""

    def __init__(self, index: int):
        lib = None
        for name in ("libnvidia-ml.so.1", "libnvidia-ml.so"):
            try:
                lib = ctypes.CDLL(name)
                break
            except OSError:
                continue
        if lib is None or lib.nvmlInit_v2() != 0:
            raise OSError("NVML unavailable")
        self.lib = lib
        self.h = ctypes.c_void_p()
        if lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(index), ctypes.byref(self.h)) != 0:
            lib.nvmlShutdown()
            raise OSError("NVML device handle")
        get = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None)
        self.get_reasons = get or lib.nvmlDeviceGetCurrentClocksThrottleReasons
        v = ctypes.c_uint()
        self.max_mhz = float(v.value) if lib.nvmlDeviceGetMaxClockInfo(self.h, _NVML_CLOCK_SM, ctypes.byref(v)) == 0 else None

    def sample(self):
        mhz, r = ctypes.c_uint(), ctypes.c_ulonglong()
        if self.lib.nvmlDeviceGetClockInfo(self.h, _NVML_CLOCK_SM, ctypes.byref(mhz)) != 0:
            return None
        reasons = r.value if self.get_reasons(self.h, ctypes.byref(r)) == 0 else 0
        return float(mhz.value), reasons

    def close(self):
        self.lib.nvmlShutdown()


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int, period_s: float = 0.002):
        self.index, self.period = index, period_s
        self.samples: list = []
        self.nvml = None
        self.thread = None
        self.stop = threading.Event()
        self.p = None
        self.f = None

    def _loop(self):
        while not self.stop.is_set():
            s = self.nvml.sample()
            if s is not None:
                self.samples.append(s)
            time.sleep(self.period)

    def __enter__(self):
        try:
            self.nvml = _Nvml(self.index)
        except (OSError, AttributeError):
            self.nvml = None
        if self.nvml is not None:
            s = self.nvml.sample()  # one sample before the region starts, so none is ever empty
            if s is not None:
                self.samples.append(s)
            self.thread = threading.Thread(target=self._loop, daemon=True)
            self.thread.start()
            return self
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                       "--format=csv,noheader,nounits", "-lms", "200"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None
        return self

    def __exit__(self, *a):
        if self.thread is not None:
            s = self.nvml.sample()  # and one at its end
            if s is not None:
                self.samples.append(s)
            self.stop.set()
            self.thread.join(timeout=5)
        if self.p is not None:
            self.p.terminate()
            try:
                self.p.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.p.kill()

    def summary(self) -> dict:
        if self.nvml is not None:
            sm = [s[0] for s in self.samples]
            reasons = sorted({name for _, bits in self.samples for b, name in _REASONS.items() if bits & b})
            mx = self.nvml.max_mhz
            self.nvml.close()
            self.nvml = None
            if not sm:
                return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": ["unavailable"], "samples": 0, "source": "nvml"}
            return {"sm_mhz": statistics.median(sm), "sm_min_mhz": min(sm), "sm_max_mhz": mx, "reasons": reasons,
                    "samples": len(sm), "source": "nvml, every 2 ms"}
        if self.f is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        self.f.flush()
        self.f.seek(0)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.f.read().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.f.name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm), "source": "nvidia-smi, every 200 ms"}
