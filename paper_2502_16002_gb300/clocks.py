"""GPU clocks and throttle reasons sampled by nvidia-smi while a measurement runs.

Used by bench.py and the TTFT harness: a timed region is bracketed by start() / stop(), and
summary() reports the median SM clock under load, the maximum clock and every throttle
reason seen active in that window (a run that saw hw_slowdown, hw_thermal_slowdown or
sw_thermal_slowdown, or clocks stuck well below the maximum, is not a valid measurement;
sw_power_cap is kept and reported).  Reads only; it changes no GPU setting.
"""
from __future__ import annotations

import statistics
import subprocess
import time


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every interval_ms in a background reader.

    Each line is stamped when it arrives; summary() keeps the samples that fall inside
    the window marked with start() / stop()."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, interval_ms: int = 50):
        self.gpu = gpu_index
        self.interval_ms = int(interval_ms)
        self.proc = None
        self.lines = []
        self.t0 = self.t1 = None

    def __enter__(self):
        import threading
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", str(self.interval_ms)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None
            return self

        def reader():
            for line in self.proc.stdout:
                self.lines.append((time.time(), line))

        self.thread = threading.Thread(target=reader, daemon=True)
        self.thread.start()
        time.sleep(0.5)  # let the first samples arrive before the timed region
        return self

    def start(self):
        self.t0 = time.time()

    def stop(self):
        self.t1 = time.time()

    def __exit__(self, *a):
        if self.proc is None:
            return
        time.sleep(0.3)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, mx, reasons, n_all = [], None, set(), 0
        for t, line in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            n_all += 1
            pad = self.interval_ms / 1000.0
            if self.t0 is not None and not (self.t0 - pad <= t <= self.t1 + pad):
                continue
            try:
                sm.append(float(f[0]))
                mx = float(f[1])
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": 0,
                    "samples_total": n_all}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}
