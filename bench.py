#!/usr/bin/env python3
"""Throughput of the CoLA layer stack (forward + full backward) on GB300.

One step = one pass of the whole hot path over one batch: the forward of all
seven CoLA layers of a LLaMA-shaped block (q/k/v fused, o, gate, up, down;
h = B sigma(A x) each, Sec. 3.2 / Fig. 4) followed by their backward
(Sec. 3.4), every GEMM on the library's tcgen05 kernels through the C ABI.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 7b|1b|350m|60m|60m-q|...]
                    [--mode cola|cola_m|infer] [--impl cola|reference] [--graph on|off]

The default workload is the LLaMA-7B-shaped block in CoLA-M mode (32768
tokens); its line also carries the 1B block (65536 tokens) timed in the same
run.  Prints ONE JSON line (rank 0).  `value` is whole-job TFLOP/s
(algorithmic 6 n r (d_in + d_out) per layer), device-timed with CUDA events,
inputs resident in HBM; `e2e` is the same metric with each step's inputs
copied from pinned host memory and its results (weight and input gradients)
copied back inside the timed region.  The working set of every block
workload is larger than L2 (129 MB), so no L2 flush is needed between steps.

--impl reference times the fp64 CPU oracle (the only reference there is: the
paper publishes no implementation) on the host cores, on a bounded sample of
the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "CoLA layer fwd+bwd TFLOP/s and % of GB300 dense-BF16 peak; tokens/s per block"
METRIC_INFER = "CoLA block forward (inference) TFLOP/s and % of GB300 dense-BF16 peak; tokens/s"
L2_BYTES = 129 << 20


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                "source": "measured"}
    except Exception:  # noqa: BLE001 -- the file is driver-written; fall back to the recipe's figures
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# ---------------------------------------------------------------- the block
class Block:
    """All tensors of one CoLA block workload, resident on the device."""

    def __init__(self, wl, mode, device, seed=0, sigma="silu", gated_unfused=False):
        import torch

        from paper_2502_10940_gb300 import cola
        from paper_2502_10940_gb300 import inputs as I

        self.torch, self.cola = torch, cola
        self.wl, self.mode, self.sigma = wl, mode, sigma
        n = wl.n
        bf = torch.bfloat16
        self.X = {}
        for li, L in enumerate(wl.layers):
            if L.x not in self.X:
                self.X[L.x] = I.activation(n, L.d_in, seed, device, layer=100 + len(self.X))
        # projections that read one X with equal shapes (q/k/v, gate/up) run
        # through the shared-input entry points: one A-GEMM with N = count*r
        groups = {}
        for li, L in enumerate(wl.layers):
            groups.setdefault(L.x, []).append(li)
        self.layers = []
        self.train = mode != "infer"
        for li, L in enumerate(wl.layers):
            t = I.layer_inputs(n, L.d_in, L.d_out, L.r, seed=seed, device=device, layer=li, with_x=False,
                               with_dy=self.train)
            X = self.X[L.x]
            st = dict(L=L, X=X, A=t["A"], B=t["B"], dY=t.get("dY"))
            ldy = I.padded_ld(L.d_out)
            st["Y"] = torch.empty((n, ldy), dtype=bf, device=device)[:, :L.d_out]
            st["desc"] = cola.desc(n, L.d_in, L.d_out, L.r, ld_x=cola.ld_of(X), ld_y=ldy, ld_a=cola.ld_of(t["A"]),
                                   sigma=sigma, mode=mode)
            if self.train:
                st["dB"] = torch.empty((L.d_out, L.r), dtype=bf, device=device)
            self.layers.append(st)
        self.groups = []
        self.ws_bytes = 0
        for key, idx in groups.items():
            mem = [self.layers[i] for i in idx]
            L = mem[0]["L"]
            fuse = (wl.fused_qkv and 2 <= len(mem) <= 3
                    and all((m["L"].d_out, m["L"].r) == (L.d_out, L.r) for m in mem))
            parts = [mem] if fuse else [[m] for m in mem]
            for part in parts:
                c = len(part)
                ldx = cola.ld_of(part[0]["X"])
                g = dict(members=part, desc=part[0]["desc"], X=part[0]["X"])
                if c == 1:
                    g["A"] = part[0]["A"]
                else:
                    g["A"] = torch.empty((c * L.r, ldx), dtype=bf, device=device)[:, :L.d_in]
                    for j, m in enumerate(part):
                        g["A"][j * L.r:(j + 1) * L.r].copy_(m["A"])
                g["Z"] = torch.empty((n, c * L.r), dtype=bf, device=device) if self.train else None
                g["H"] = torch.empty((n, c * L.r), dtype=bf, device=device) if mode == "cola" else None
                if self.train:
                    g["dX"] = torch.empty((n, ldx), dtype=bf, device=device)[:, :L.d_in]
                    g["dA"] = torch.empty((c * L.r, ldx), dtype=bf, device=device)[:, :L.d_in]
                self.ws_bytes = max(self.ws_bytes, cola.cola_workspace_size(g["desc"], c))
                self.groups.append(g)
        # the gated MLP: the gate/up group's output GEMM forms M = Y_gate * Y_up
        # straight into the down layer's input, and the down layer's backward
        # forms dY_gate, dY_up straight into the gate/up upstream gradients
        self.gated = bool(getattr(wl, "gated", False))
        # gated_unfused (a comparison point, not the library's path): the same
        # gated MLP with the product and its backward as torch element-wise
        # ops between the library's calls (Y_gate, Y_up and dM stored)
        self.gated_unfused = self.gated and gated_unfused
        if self.gated:
            gu = [g for g in self.groups if [m["L"].name for m in g["members"]] == ["gate", "up"]]
            dn = [g for g in self.groups if [m["L"].name for m in g["members"]] == ["down"]]
            if len(gu) != 1 or len(dn) != 1:
                raise ValueError("a gated MLP needs one gate/up group and one down layer")
            gu, dn = gu[0], dn[0]
            gu["M_key"] = dn["members"][0]["L"].x
            dn["gate_up"] = gu
            if self.gated_unfused and self.train:
                dn["dM"] = dn["dX"]
            dn["dX"] = None
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device)
        cola.cola_workspace_init(self.ws)
        self.launches_per_step = None

    def _chained(self):
        """Tensors a gated step forms itself: the down layer's input M and the
        gate/up upstream gradients."""
        if not self.gated:
            return set()
        dn = [g for g in self.groups if "gate_up" in g][0]
        out = {id(self.X[dn["gate_up"]["M_key"]])}
        if self.train:
            out |= {id(m["dY"]) for m in dn["gate_up"]["members"]}
        return out

    # inputs a step consumes from outside (activations, and upstream gradients
    # when training)
    def step_inputs(self):
        ins = list(self.X.values()) + ([s["dY"] for s in self.layers] if self.train else [])
        chained = self._chained()
        return [t for t in ins if id(t) not in chained]

    def add_io_set(self):
        """A second set of the step's input and result buffers (same shapes
        and pitches), so that the next step's inputs can be copied in, and the
        last step's results copied out, while this step runs; bind(i) selects
        the set the next step reads and writes."""
        torch = self.torch

        def twin(t):
            full = torch.as_strided(t, (t.shape[0], t.stride(0)), (t.stride(0), 1))
            return full.clone()[:, :t.shape[1]]

        if not hasattr(self, "io_sets"):
            self.io_sets = [(dict(self.X), [s["dY"] for s in self.layers], self.step_results())]
        X0, dY0, R0 = self.io_sets[0]
        X2 = {k: twin(v) for k, v in X0.items()}
        dY2 = [twin(d) if d is not None else None for d in dY0]
        R2 = [twin(t) for t in R0]
        self.io_sets.append((X2, dY2, R2))

    def bind(self, i):
        X, dY, R = self.io_sets[i]
        self.X = dict(X)
        for s, d in zip(self.layers, dY):
            s["X"] = X[s["L"].x]
            s["dY"] = d
        for g in self.groups:
            g["X"] = X[g["members"][0]["L"].x]
        for (obj, key), t in zip(self._result_slots(), R):
            obj[key] = t

    # what a step hands back: the weight gradients and the block's input
    # gradients (training), or the outputs (inference)
    def _result_slots(self):
        if not self.train:
            # a gated MLP's gate and up outputs are consumed inside the kernel
            # that forms M = Y_gate * Y_up: not results
            inner = {id(m) for g in self.groups if "M_key" in g and not self.gated_unfused for m in g["members"]}
            return [(s, "Y") for s in self.layers if id(s) not in inner]
        return ([(g, "dA") for g in self.groups] + [(s, "dB") for s in self.layers] +
                [(g, "dX") for g in self.groups if g["dX"] is not None])

    def step_results(self):
        return [obj[key] for obj, key in self._result_slots()]

    def results_words(self):
        if not self.train:
            if self.gated and not self.gated_unfused:
                return "Y of every layer but gate and up (M = Y_gate * Y_up feeds the down layer on the device)"
            return "Y of every layer"
        if self.gated:
            return ("dA and dB of every layer and dX of the attention and gate/up input groups; Y, Z and H stay "
                    "on the device (they feed the block's attention / MLP ops and the backward)")
        return ("dA and dB of every layer and dX of every input group; Y, Z and H stay on the device "
                "(they feed the block's attention / MLP ops and the backward)")

    def forward(self):
        c = self.cola
        for g in self.groups:
            m = g["members"]
            if "M_key" in g and self.gated_unfused:
                c.cola_fwd_shared_x(g["desc"], g["X"], g["A"], [s["B"] for s in m], [s["Y"] for s in m], g["Z"],
                                    g["H"], self.ws)
                self.torch.mul(m[0]["Y"], m[1]["Y"], out=self.X[g["M_key"]])
            elif "M_key" in g:
                Yg, Yu = (m[0]["Y"], m[1]["Y"]) if self.train else (None, None)
                c.cola_fwd_gate_up(g["desc"], g["X"], g["A"], m[0]["B"], m[1]["B"], self.X[g["M_key"]], Yg, Yu,
                                   g["Z"], g["H"], self.ws)
            elif len(m) == 1:
                s = m[0]
                c.cola_fwd(g["desc"], g["X"], g["A"], s["B"], s["Y"], g["Z"], g["H"], self.ws)
            else:
                c.cola_fwd_shared_x(g["desc"], g["X"], g["A"], [s["B"] for s in m], [s["Y"] for s in m], g["Z"],
                                    g["H"], self.ws)

    def backward(self):
        c = self.cola
        for g in reversed(self.groups):
            m = g["members"]
            if "gate_up" in g and self.gated_unfused:
                s, gm = m[0], g["gate_up"]["members"]
                c.cola_bwd(g["desc"], g["X"], g["A"], s["B"], s["dY"], g["Z"], g["H"], g["dM"], g["dA"], s["dB"],
                           self.ws)
                self.torch.mul(g["dM"], gm[1]["Y"], out=gm[0]["dY"])
                self.torch.mul(g["dM"], gm[0]["Y"], out=gm[1]["dY"])
            elif "gate_up" in g:
                s, gm = m[0], g["gate_up"]["members"]
                c.cola_bwd_down_gated(g["desc"], g["X"], g["A"], s["B"], s["dY"], g["Z"], g["H"], gm[0]["Y"],
                                      gm[1]["Y"], gm[0]["dY"], gm[1]["dY"], g["dA"], s["dB"], self.ws)
            elif len(m) == 1:
                s = m[0]
                c.cola_bwd(g["desc"], g["X"], g["A"], s["B"], s["dY"], g["Z"], g["H"], g["dX"], g["dA"], s["dB"],
                           self.ws)
            else:
                c.cola_bwd_shared_x(g["desc"], g["X"], g["A"], [s["B"] for s in m], [s["dY"] for s in m], g["Z"],
                                    g["H"], g["dX"], g["dA"], [s["dB"] for s in m], self.ws)

    def step(self):
        self.forward()
        if self.train:
            self.backward()

    def check(self):
        st, code = self.cola.cola_check_status(self.ws)
        if st != 0:
            raise RuntimeError(f"device status {st} (code {code:#x})")

    def working_set_bytes(self):
        t = self.torch
        seen, total = set(), 0
        for obj in vars(self).values():
            items = obj if isinstance(obj, list) else [obj]
            for it in items:
                vals = it.values() if isinstance(it, dict) else [it]
                for v in vals:
                    if isinstance(v, t.Tensor) and v.is_cuda and v.data_ptr() not in seen:
                        seen.add(v.data_ptr())
                        total += v.untyped_storage().nbytes()
        return total


# ---------------------------------------------------------------- per-launch accounting
def launch_cost(kind, shapes, splits, flags):
    """(algorithmic bytes, flops) of one library launch, summed over the GEMMs
    it runs: each operand read once, each result written once, bf16 (2 B);
    the fp32 token-split partials of the weight gradients are implementation
    traffic and are not counted."""
    e = 2
    if kind == "fwd_fused":
        # X, A and B read, Z / H (as stored) and Y written; H stays on chip
        (m, r, k1), (_, n_out, _) = shapes
        nzh = (1 if flags & 1 else 0) + (1 if flags & 64 else 0)
        return e * (m * k1 + r * k1 + m * r * nzh + n_out * r + m * n_out), 2.0 * m * r * (k1 + n_out)
    if kind == "bwd_fused":
        # dY, B, the saved Z and A read; dZ (and, flag 1, H) and dX written; dZ stays on chip in between
        (m, r, k1), (_, n_out, _) = shapes
        nzh = 2 + (1 if flags & 1 else 0)
        return e * (m * k1 + k1 * r + m * r * nzh + r * n_out + m * n_out), 2.0 * m * r * (k1 + n_out)
    tb, tf = 0.0, 0.0
    for (m, n, k) in shapes:
        if kind in ("fwd_zh", "fwd_y") and flags & 2:
            b = e * (m * k + n * k)   # split-K partials; the reduce writes the output
        elif kind == "fwd_zh":
            b = e * (m * k + n * k + m * n * (2 if flags & 1 else 1))
        elif kind == "fwd_y":
            b = e * (m * k + n * k + m * n)
        elif kind == "bwd_dz":
            b = e * (m * k + n * k + m * n * (3 if flags & 1 else 2))
        elif kind == "wgrad":
            b = e * (k * m + k * n + m * n)
        elif kind == "bwd_dx":
            # flag 32: the gated epilogue read Y_gate, Y_up and wrote dY_gate, dY_up
            b = e * (m * k + n * k + m * n * (4 if flags & 32 else 1))
        elif kind == "fwd_glu":
            b = e * (m * k + n * k + m * n * (3 if flags & 1 else 1))   # M (+ Y_gate, Y_up)
        elif kind == "reduce":
            b = e * m * n * (2 if flags & 1 else 1)   # flag: the Z/H reduce writes Z and H
        elif kind == "sigma":
            b = e * 2 * m * n
        else:
            b = 0
        tb += b
        tf += 0.0 if kind in ("reduce", "sigma") else 2.0 * m * n * k
    return tb, tf


def summarize_trace(records, peaks, ridge):
    kinds = {}
    for kind, shapes, splits, flags, ms in records:
        b, f = launch_cost(kind, shapes, splits, flags)
        d = kinds.setdefault(kind, {"launches": 0, "ms": 0.0, "bytes": 0.0, "flops": 0.0})
        d["launches"] += 1
        d["ms"] += ms
        d["bytes"] += b
        d["flops"] += f
    total = sum(d["ms"] for d in kinds.values()) or 1.0
    for d in kinds.values():
        d["share"] = d["ms"] / total
    top = max(kinds, key=lambda x: kinds[x]["ms"])
    d = kinds[top]
    t = d["ms"] / 1e3
    intensity = d["flops"] / max(d["bytes"], 1.0)
    # every traced launch is bracketed by its own events: a kernel timed
    # alone, so the burst peak is its denominator (the sustained one beside it)
    if intensity >= ridge:
        achieved = d["flops"] / t / 1e12
        peak = peaks["bf16_tflops"]
        roof = {"bound": "tensor", "unit": "TFLOP/s",
                "frac_sustained": round(achieved / peaks["bf16_tflops_sustained"], 4),
                "peak_sustained": peaks["bf16_tflops_sustained"]}
    else:
        achieved = d["bytes"] / t / 1e9
        peak = peaks["hbm_gbs"]
        roof = {"bound": "hbm", "unit": "GB/s"}
    roof.update({"kernel": f"gemm {top}", "achieved": round(achieved, 1), "peak": peak,
                 "frac": round(achieved / peak, 4), "peak_source": peaks["source"],
                 "peak_kind": "burst (each launch timed alone)" if roof["bound"] == "tensor" else "copy",
                 "launches": d["launches"], "avg_launch_us": round(d["ms"] * 1e3 / d["launches"], 2),
                 "algorithmic_bytes_per_launch": int(d["bytes"] / d["launches"]),
                 "flop_per_launch": d["flops"] / d["launches"], "share": round(d["share"], 4)})
    return roof, {k: {"launches": v["launches"], "share": round(v["share"], 4),
                      "avg_us": round(v["ms"] * 1e3 / v["launches"], 2),
                      "gbs": round(v["bytes"] / (v["ms"] / 1e3) / 1e9, 1),
                      "tflops": round(v["flops"] / (v["ms"] / 1e3) / 1e12, 1)} for k, v in kinds.items()}


def kernel_source_hash():
    """sha256 of the GEMM kernel's code (gemm.cuh and ptx.cuh with comments
    and whitespace removed): a committed ncu figure stays valid while this
    hash, i.e. the code it was measured on, is unchanged."""
    import hashlib
    import re

    h = hashlib.sha256()
    for name in ("gemm.cuh", "ptx.cuh"):
        with open(os.path.join(ROOT, "paper_2502_10940_gb300", "csrc", name)) as g:
            src = g.read()
        src = re.sub(r"//[^\n]*", "", src)
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        h.update(re.sub(r"\s+", "", src).encode())
    return h.hexdigest()


def traffic_from_profile(kernel_key, workload, algorithmic_bytes):
    """dram bytes per launch from a committed ncu summary, valid only while the
    kernel code is unchanged (kernel_source_hash) and the launches it averaged
    carry the same algorithmic bytes as the ones timed now; else None."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(path):
        return None
    try:
        with open(path) as f:
            rec = json.load(f)
        entry = rec.get(workload, {}).get(kernel_key)
        if (entry and entry.get("src_sha256") == kernel_source_hash()
                and entry.get("algorithmic_bytes_per_launch") == algorithmic_bytes):
            return entry["dram_bytes_per_launch"]
    except Exception:  # noqa: BLE001 -- a missing or stale summary means "no traffic figure"
        return None
    return None


# ---------------------------------------------------------------- clocks
class ClockSampler:
    """SM clock, power and clock-event reasons sampled every 10 ms on a
    background thread while the timed region runs (NVML read-only queries
    through the driver's libnvidia-ml; falls back to nvidia-smi)."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, device_index):
        self.dev = device_index
        self.samples = []
        self.max_mhz = None
        self._stop = None
        self._thread = None
        self._nvml = None
        self._h = None
        self._smi = None
        self._opened = False

    def _open_nvml(self):
        import ctypes

        import torch
        lib = ctypes.CDLL("libnvidia-ml.so.1")
        if lib.nvmlInit_v2() != 0:
            raise RuntimeError("nvmlInit failed")
        h = ctypes.c_void_p()
        uuid = str(torch.cuda.get_device_properties(self.dev).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        if lib.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h)) != 0:
            if lib.nvmlDeviceGetHandleByIndex_v2(self.dev, ctypes.byref(h)) != 0:
                raise RuntimeError("no NVML handle")
        mx = ctypes.c_uint()
        if lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
            self.max_mhz = float(mx.value)
        self._reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            getattr(lib, "nvmlDeviceGetCurrentClocksThrottleReasons")
        self._nvml, self._h = lib, h

    def _sample_nvml(self):
        import ctypes
        c = ctypes.c_uint()
        r = ctypes.c_ulonglong()
        pw = ctypes.c_uint()
        if self._nvml.nvmlDeviceGetClockInfo(self._h, 1, ctypes.byref(c)) != 0:
            return
        self._reasons_fn(self._h, ctypes.byref(r))
        self._nvml.nvmlDeviceGetPowerUsage(self._h, ctypes.byref(pw))
        self.samples.append((float(c.value), int(r.value), pw.value / 1000.0))

    def open(self):
        """Load NVML (this can take a while on a cold start).  Called before
        the warm-up, so that the GPU does not idle between the warm-up and
        the timed region."""
        if self._opened:
            return
        self._opened = True
        try:
            self._open_nvml()
        except Exception:  # noqa: BLE001 -- no NVML: use nvidia-smi instead
            self._nvml = None

    def start(self):
        import threading
        self.open()
        if self._nvml is None:
            try:
                self._smi = subprocess.Popen(
                    ["nvidia-smi", "--query-gpu=clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active",
                     "--format=csv,noheader,nounits", "-lms", "100", "-i", str(self.dev)],
                    stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            except Exception:  # noqa: BLE001
                self._smi = None
            return
        self._stop = threading.Event()

        def loop():
            while not self._stop.is_set():
                self._sample_nvml()
                self._stop.wait(0.01)

        self._thread = threading.Thread(target=loop, daemon=True)
        self._thread.start()

    def stop(self):
        if self._thread is not None:
            self._stop.set()
            self._thread.join()
            self._sample_nvml()
        elif self._smi is not None:
            self._smi.terminate()
            out, _ = self._smi.communicate()
            for line in out.splitlines():
                parts = [p.strip() for p in line.split(",")]
                try:
                    self.samples.append((float(parts[0]), int(parts[3], 16), float(parts[2])))
                    self.max_mhz = float(parts[1])
                except (ValueError, IndexError):
                    continue
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": ["no clock samples"], "samples": 0}
        reasons = set()
        for _, bits, _ in self.samples:
            for b, nm in self.REASONS.items():
                if bits & b:
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(x[0] for x in self.samples), "sm_max_mhz": self.max_mhz,
                "reasons": sorted(reasons), "power_w_max": round(max(x[2] for x in self.samples), 1),
                "samples": len(self.samples), "source": "nvml" if self._nvml is not None else "nvidia-smi"}


# ---------------------------------------------------------------- CPU oracle
def oracle_block_sample(wl, n_s, seed=0):
    """The whole block (7 layers, fwd + bwd) through the fp64 oracle on n_s
    tokens of the same synthetic distribution.  Returns (seconds, flops)."""
    import oracle
    from paper_2502_10940_gb300 import inputs as I
    from paper_2502_10940_gb300.workloads import fwd_flops, layer_flops

    train = wl.phase != "infer"
    xs = {}
    for L in wl.layers:
        if L.x not in xs:
            xs[L.x] = I.activation(n_s, L.d_in, seed, "cpu", layer=100 + len(xs)).float().double().numpy()
    prepared = []
    for li, L in enumerate(wl.layers):
        t = I.layer_inputs(n_s, L.d_in, L.d_out, L.r, seed=seed, device="cpu", layer=li, with_x=False,
                           with_dy=train)
        prepared.append((xs[L.x], t["A"].float().double().numpy(), t["B"].float().double().numpy(),
                         t["dY"].float().double().numpy() if train else None))
    t0 = time.perf_counter()
    for X, A, B, dY in prepared:
        Z, H, Y = oracle.fwd(X, A, B, "silu")
        if train:
            oracle.bwd(X, A, B, dY, Z, H, "silu", "cola")
    dt = time.perf_counter() - t0
    f = layer_flops if train else fwd_flops
    return dt, float(sum(f(n_s, L.d_in, L.d_out, L.r) for L in wl.layers))


def phase_words(wl):
    return "fwd+bwd" if wl.phase != "infer" else "fwd only"


def calibrate_tokens(wl, target_s):
    n_s, dt = 64, 0.0
    while True:
        dt, _ = oracle_block_sample(wl, n_s)
        if dt >= 0.5 or n_s >= wl.n:
            break
        n_s *= 2
    return max(16, min(wl.n, int(n_s * target_s / max(dt, 1e-6)) // 16 * 16))


def cpu_baseline(wl, target_s=10.0):
    import oracle

    n_s = calibrate_tokens(wl, target_s)
    dt, fl = oracle_block_sample(wl, n_s)
    return {"value": round(fl / dt / 1e12, 6), "unit": "TFLOP/s", "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"{wl.name} block, all {len(wl.layers)} layers {phase_words(wl)} on {n_s} of {wl.n} tokens "
                      f"({dt:.1f} s, fp64 loops, OpenMP)",
            # every token costs the same, so the full step scales with the token count
            "full_step_s_extrapolated": round(dt * wl.n / n_s, 2)}


# ---------------------------------------------------------------- arms
def run_reference(args, wl):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import oracle

    budget = 150.0  # seconds for warmup + steps
    per_step = max(0.5, min(10.0, budget / max(1, args.steps + args.warmup)))
    n_s = calibrate_tokens(wl, per_step)
    for _ in range(args.warmup):
        oracle_block_sample(wl, n_s)
    tot_t, tot_f = 0.0, 0.0
    for _ in range(args.steps):
        dt, fl = oracle_block_sample(wl, n_s)
        tot_t += dt
        tot_f += fl
    value = tot_f / tot_t / 1e12
    sample = f"{wl.name} block, all {len(wl.layers)} layers {phase_words(wl)} on {n_s} of {wl.n} tokens per step"
    line = {"impl": "reference", "metric": METRIC if wl.phase != "infer" else METRIC_INFER, "value": round(value, 6), "unit": "TFLOP/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(tot_t / args.steps * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": wl.desc, "n_tokens_sampled": n_s,
                                            "mode": "cola" if wl.phase != "infer" else "infer"},
            "cpu_baseline": {"value": round(value, 6), "unit": "TFLOP/s", "cores": oracle.num_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# untimed steps after the warm-up until the GPU has run this long, so that the
# timed steps see the clocks and power state of sustained load (a GPU coming
# out of idle ramps its clocks up; a 1.4 kW part under a tensor-bound load
# reaches its power cap within a few hundred milliseconds)
SETTLE_S = 0.5


def settle_steps(fn, seconds, max_steps=20000):
    """Run fn() until `seconds` of wall time have passed with the device kept
    busy (synchronising after each batch of calls); returns the steps run and
    the seconds taken."""
    import torch

    torch.cuda.synchronize()
    t0 = time.perf_counter()
    n, batch = 0, 1
    while n < max_steps:
        for _ in range(batch):
            fn()
        n += batch
        torch.cuda.synchronize()
        dt = time.perf_counter() - t0
        if dt >= seconds:
            break
        batch = min(2 * batch, max(1, max_steps - n))
    return {"steps": n, "s": round(time.perf_counter() - t0, 3)}


def time_steps(fn, steps, stream, dist=None, flush=None):
    """Mean device time of one fn() over `steps` back-to-back calls.  With
    `flush` (a buffer larger than L2), each call is timed alone and the
    buffer is rewritten between calls, outside the timed intervals."""
    import torch

    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    if flush is None:
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        total = e0.elapsed_time(e1)
    else:
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for a, b in ev:
            flush.fill_(1)
            a.record(stream)
            fn()
            b.record(stream)
        torch.cuda.synchronize()
        total = sum(a.elapsed_time(b) for a, b in ev)
    if dist:
        dist.barrier()
    return max_over_ranks(total / steps, dist, "cuda")


def max_over_ranks(value, dist=None, device="cpu"):
    """The largest of the ranks' values (the job's step time is its slowest
    rank's); the value itself without a process group."""
    if not dist:
        return value
    import torch

    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_tflops(flops_per_rank_step, world, ms_per_step):
    """Weak scaling: every rank runs the whole workload on its own batch, so
    the job processes world x the per-rank work in the (max-over-ranks) step
    time."""
    return flops_per_rank_step * world / (ms_per_step / 1e3) / 1e12


def full_rank_baseline(wl, device, steps, warmup, seed=0, flush=None, settle=0.0, graph=False):
    """Same-shape full-rank layers (fwd Y = X W^T, bwd dX = dY W, dW = dY^T X;
    forward only for an inference workload) with torch.matmul (cuBLAS);
    layers reading one input (q/k/v, gate/up) are fused into one GEMM with
    their output widths concatenated.  With `graph`, the step is captured
    once as a CUDA graph and replayed, as the CoLA step is, so that both
    sides pay the same launch costs (which set the time of the small
    workloads)."""
    import torch

    n = wl.n
    bf = torch.bfloat16
    train = wl.phase != "infer"
    g = torch.Generator(device=device).manual_seed(seed + 77)
    groups = {}
    for L in wl.layers:
        key = L.x if wl.fused_qkv else L.name
        groups.setdefault(key, []).append(L)
    bufs = []
    flops = 0.0
    for key, Ls in groups.items():
        d_in = Ls[0].d_in
        d_out = sum(L.d_out for L in Ls)
        # flops count the logical widths; the GEMMs run on widths rounded up
        # to a multiple of 8 so that cuBLAS gets 16-byte aligned rows (as the
        # CoLA path gets through its padded pitches)
        flops += (6.0 if train else 2.0) * n * d_in * d_out
        d_in, d_out = -(-d_in // 8) * 8, -(-d_out // 8) * 8
        X = torch.randn((n, d_in), generator=g, device=device, dtype=torch.float32).to(bf)
        W = (torch.randn((d_out, d_in), generator=g, device=device, dtype=torch.float32) * d_in ** -0.5).to(bf)
        b = dict(X=X, W=W, Y=torch.empty((n, d_out), dtype=bf, device=device))
        if train:
            b["dY"] = torch.randn((n, d_out), generator=g, device=device, dtype=torch.float32).to(bf)
            b["dX"] = torch.empty((n, d_in), dtype=bf, device=device)
            b["dW"] = torch.empty((d_out, d_in), dtype=bf, device=device)
        bufs.append(b)

    def step():
        for b in bufs:
            torch.matmul(b["X"], b["W"].t(), out=b["Y"])
        if not train:
            return
        for b in reversed(bufs):
            torch.matmul(b["dY"], b["W"], out=b["dX"])
            torch.matmul(b["dY"].t(), b["X"], out=b["dW"])

    for _ in range(warmup):
        step()
    run = step
    if graph:
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            step()
        run = g.replay
        for _ in range(warmup):
            run()
    st = settle_steps(run, settle)
    ms = time_steps(run, steps, torch.cuda.current_stream(), flush=flush)
    del bufs
    return {"ms_per_step": round(ms, 4), "tflops": round(flops / (ms / 1e3) / 1e12, 1), "flops": flops,
            "impl": "torch.matmul (cuBLAS) bf16", "cuda_graph": bool(graph), "settle": st}


def timed_block(wl, mode, args, device, stream, dist=None, seed=0, **block_kw):
    """Build the block, count its launches with the library trace, warm it
    up, capture its step as a CUDA graph (unless --graph off) and time K
    steps (clocks sampled meanwhile).  Returns a dict of what it built and
    measured."""
    import torch

    from paper_2502_10940_gb300 import cola

    sampler = ClockSampler(torch.cuda.current_device())
    sampler.open()
    blk = Block(wl, mode, device, seed=seed, **block_kw)
    # launches per step, counted by the library's trace
    with cola.Trace(512) as tr:
        blk.step()
    blk.launches_per_step = tr.count.value
    blk.check()

    for _ in range(args.warmup):
        blk.step()
    torch.cuda.synchronize()
    # each step replays as one CUDA graph: its launches are recorded once
    # (after the eager warm-up, which set every kernel's attributes) and
    # replayed with no host work per launch and less launch overhead on the
    # GPU (measured: -2 % step time on the 60M and 1B blocks)
    use_graph = args.graph != "off"
    step_fn, graph = blk.step, None
    if use_graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            blk.step()
        step_fn = graph.replay
        for _ in range(args.warmup):
            step_fn()
        torch.cuda.synchronize()
        blk.check()
    # a working set that fits in L2 is timed step by step with L2 rewritten
    # between steps
    ws_bytes = blk.working_set_bytes()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device) if ws_bytes < L2_BYTES else None
    settle = settle_steps(step_fn, args.settle)
    sampler.start()
    ms = time_steps(step_fn, args.steps, stream, dist, flush=flush)
    clocks = sampler.stop()
    blk.check()
    return dict(blk=blk, graph=graph, step_fn=step_fn, use_graph=use_graph, ms=ms, clocks=clocks,
                flush=flush, ws_bytes=ws_bytes, settle=settle)


def modes_ratio(wl, mode, blk, args, device, stream, seed=0):
    """The same workload in its other mode: CoLA-M's time over CoLA's, the two
    modes timed alternately (3 rounds each, medians) so that both see the
    same clocks.  None if the workload has one mode."""
    other = [m for m in wl.modes if m != mode]
    if not other:
        return None
    ob = Block(wl, other[0], device, seed=seed)
    for _ in range(args.warmup):
        ob.step()
    t_this, t_other = [], []
    for _ in range(3):
        t_this.append(time_steps(blk.step, args.steps, stream))
        t_other.append(time_steps(ob.step, args.steps, stream))
    ob.check()
    blk.check()
    ms_a, ms_o = statistics.median(t_this), statistics.median(t_other)
    ms_m, ms_c = (ms_a, ms_o) if mode == "cola_m" else (ms_o, ms_a)
    return {mode: round(ms_a, 4), other[0]: round(ms_o, 4), "cola_m_over_cola": round(ms_m / ms_c, 4),
            "how": "alternating, 3 rounds each, medians (eager launches)"}


def run_cola(args, wl):
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist_mod
        dist_mod.init_process_group("nccl")
        dist = dist_mod
    torch.cuda.set_device(local)
    device = f"cuda:{local}"

    from paper_2502_10940_gb300 import build
    from paper_2502_10940_gb300 import cola
    from paper_2502_10940_gb300.workloads import WORKLOADS

    build.build()
    cola.cola_set_fused_forward(args.fused_forward == "on")
    peaks = _peaks()
    ridge = peaks["bf16_tflops"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    mode = args.mode or wl.modes[0]
    if (mode == "infer") != (wl.phase == "infer"):
        raise SystemExit(f"mode {mode} does not fit the {wl.phase} workload {wl.name}")
    stream = torch.cuda.current_stream()
    tb = timed_block(wl, mode, args, device, stream, dist, seed=args.seed + rank,
                     **({"gated_unfused": True} if args.gated_unfused else {}))
    blk, graph, use_graph, ms, clocks, flush = (tb[k] for k in ("blk", "graph", "use_graph", "ms", "clocks",
                                                                  "flush"))

    # the same steps again with every launch bracketed by events: per-kernel times
    cap = blk.launches_per_step * args.steps
    with cola.Trace(cap) as tr:
        time_steps(blk.step, args.steps, stream)
    records = tr.records()
    roofline, kinds = summarize_trace(records, peaks, ridge)
    roofline["traffic"] = traffic_from_profile(roofline["kernel"], wl.name,
                                               roofline["algorithmic_bytes_per_launch"])
    trace_ms = sum(r[-1] for r in records) / args.steps

    flops = wl.flops
    value = whole_job_tflops(flops, world, ms)
    line = {"metric": METRIC if blk.train else METRIC_INFER, "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": wl.desc, "n_tokens": wl.n, "mode": mode, "sigma": "silu",
                       "layers": [f"{L.name}:{L.d_in}->{L.d_out},r={L.r}" for L in wl.layers],
                       "shared_x_groups": ["+".join(m["L"].name for m in g["members"]) for g in blk.groups],
                       "parallelism": "replicas" if world > 1 else "single-gpu",
                       "phase": "fwd+bwd" if blk.train else "fwd only (inference)",
                       "saved_activation_elems": sum(g[k].numel() for g in blk.groups for k in ("Z", "H")
                                                     if g.get(k) is not None),
                       "cuda_graph": use_graph,
                       "fused_forward": args.fused_forward == "on",
                       "l2": (f"flushed between steps (256 MB write): working set {tb['ws_bytes'] / 1e6:.1f} MB < L2"
                              if flush is not None else
                              f"no flush: working set {tb['ws_bytes'] / 1e9:.2f} GB > 129 MB L2")},
            "tokens_per_s": round(wl.n * world / (ms / 1e3), 1),
            "pct_dense_bf16_peak": round(100.0 * value / world / peaks["bf16_tflops"], 2),
            "pct_dense_bf16_peak_sustained": round(100.0 * value / world / peaks["bf16_tflops_sustained"], 2),
            "roofline": roofline, "kernels": kinds,
            # the per-kernel figures come from eager steps with events around
            # every launch; their sum per step, beside the graph-timed step
            "trace_ms_per_step": round(trace_ms, 4),
            "kernels_how": "eager steps, CUDA events around each launch; shares are of trace_ms_per_step",
            "gpu_launches": blk.launches_per_step * args.steps, "clocks": clocks,
            "settle": {**tb["settle"], "how": "untimed steps after the warm-up, device kept busy, "
                                              "before the timed region and the clock samples"}}

    if not args.no_extras:
        # end to end: each step's activations (and, training, upstream
        # gradients) come from pinned host memory; the step's results (see
        # results_words) go back to pinned host memory
        def full_rows(t):   # the whole padded row-major buffer behind a view
            return torch.as_strided(t, (t.shape[0], t.stride(0)), (t.stride(0), 1))

        # The inputs and results are double-buffered: step k+1's inputs are
        # copied in on one stream and step k-1's results copied out on another
        # while step k runs.  A step waits for its inputs and for the copy-out
        # of the results its buffer set last held; a copy into an input buffer
        # waits for the step that last read it.  With graphs, one graph per
        # buffer set.
        blk.add_io_set()
        sets_in, sets_out = [], []
        for i in range(2):
            blk.bind(i)
            sets_in.append([full_rows(t) for t in blk.step_inputs()])
            sets_out.append([full_rows(t) for t in blk.step_results()])
        run_set = [blk.step, blk.step]
        if use_graph:
            g1 = torch.cuda.CUDAGraph()
            blk.bind(1)
            with torch.cuda.graph(g1):
                blk.step()
            run_set = [graph.replay, g1.replay]
        blk.bind(0)
        h_in = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in sets_in[0]]
        h_out = [[torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in sets_out[0]] for _ in range(2)]
        for h, t in zip(h_in, sets_in[0]):
            h.copy_(t)
        copy_stream, out_stream = torch.cuda.Stream(), torch.cuda.Stream()

        def copy_in(dst):
            for h, t in zip(h_in, dst):
                t.copy_(h, non_blocking=True)

        def e2e_run(K):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            ev_in = [torch.cuda.Event(), torch.cuda.Event()]
            ev_done = [torch.cuda.Event(), torch.cuda.Event()]
            ev_out = [torch.cuda.Event(), torch.cuda.Event()]
            if dist:
                dist.barrier()
            torch.cuda.synchronize()
            e0.record(stream)
            copy_stream.wait_event(e0)
            out_stream.wait_event(e0)
            with torch.cuda.stream(copy_stream):
                copy_in(sets_in[0])
            ev_in[0].record(copy_stream)
            for k in range(K):
                cur, nxt = k % 2, (k + 1) % 2
                if k + 1 < K:
                    if k >= 1:
                        copy_stream.wait_event(ev_done[nxt])
                    with torch.cuda.stream(copy_stream):
                        copy_in(sets_in[nxt])
                    ev_in[nxt].record(copy_stream)
                stream.wait_event(ev_in[cur])
                if k >= 2:
                    stream.wait_event(ev_out[cur])
                if not use_graph:
                    blk.bind(cur)
                run_set[cur]()
                ev_done[cur].record(stream)
                out_stream.wait_event(ev_done[cur])
                with torch.cuda.stream(out_stream):
                    for h, t in zip(h_out[cur], sets_out[cur]):
                        h.copy_(t, non_blocking=True)
                ev_out[cur].record(out_stream)
            stream.wait_stream(out_stream)
            e1.record(stream)
            torch.cuda.synchronize()
            if dist:
                dist.barrier()
            return max_over_ranks(e0.elapsed_time(e1) / K, dist, "cuda")

        e2e_run(2)
        e2e_steps = max(3, args.steps // 2)
        ms_e2e = e2e_run(e2e_steps)
        blk.bind(0)
        blk.check()
        bi = sum(t.numel() * t.element_size() for t in sets_in[0])
        bo = sum(t.numel() * t.element_size() for t in sets_out[0])
        line["e2e"] = {"value": round(whole_job_tflops(flops, world, ms_e2e), 2), "unit": "TFLOP/s",
                       "ms_per_step": round(ms_e2e, 4), "steps": e2e_steps, "h2d_bytes_per_step": bi,
                       "d2h_bytes_per_step": bo,
                       "inputs": "double-buffered, next step's copies overlap this step",
                       "results": "double-buffered, last step's copies overlap this step",
                       "results_to_host": blk.results_words()}
        del h_in, h_out, sets_in, sets_out, run_set
        if use_graph:
            del g1
        if rank == 0 and world == 1:
            fr = full_rank_baseline(wl, device, max(3, args.steps // 2), 3, seed=args.seed, flush=flush,
                                    settle=args.settle, graph=use_graph)
            fr["speedup_cola_vs_full_rank"] = round(fr["ms_per_step"] / ms, 3)
            line["full_rank"] = fr
            mr = modes_ratio(wl, mode, blk, args, device, stream, seed=args.seed + rank)
            if mr:
                line["modes"] = mr
            # the 1B block in the same run (its value and CoLA-M / CoLA ratio),
            # after the main workload's tensors are released
            if wl.name == "7b":
                del blk, graph, tb
                torch.cuda.synchronize()
                torch.cuda.empty_cache()
                w1 = WORKLOADS["1b"]
                t1 = timed_block(w1, w1.modes[0], args, device, stream, None, seed=args.seed)
                v1 = whole_job_tflops(w1.flops, 1, t1["ms"])
                line["also"] = {"1b": {"workload": w1.desc, "mode": w1.modes[0], "value": round(v1, 2),
                                       "unit": "TFLOP/s", "ms_per_step": round(t1["ms"], 4),
                                       "pct_dense_bf16_peak": round(100.0 * v1 / peaks["bf16_tflops"], 2),
                                       "cuda_graph": t1["use_graph"], "clocks": t1["clocks"],
                                       "settle": t1["settle"],
                                       "modes": modes_ratio(w1, w1.modes[0], t1["blk"], args, device, stream,
                                                            seed=args.seed)}}
                del t1
                # the same 7B block with the gated MLP chained through the library
                torch.cuda.synchronize()
                torch.cuda.empty_cache()
                wg = WORKLOADS["7b-gated"]
                tg = timed_block(wg, mode, args, device, stream, None, seed=args.seed)
                vg = whole_job_tflops(wg.flops, 1, tg["ms"])
                del tg["blk"], tg["graph"]
                tu = timed_block(wg, mode, args, device, stream, None, seed=args.seed, gated_unfused=True)
                line["also"]["7b_gated"] = {"workload": wg.desc, "mode": mode, "value": round(vg, 2),
                                            "unit": "TFLOP/s", "ms_per_step": round(tg["ms"], 4),
                                            "pct_dense_bf16_peak": round(100.0 * vg / peaks["bf16_tflops"], 2),
                                            "cuda_graph": tg["use_graph"], "clocks": tg["clocks"],
                                            "settle": tg["settle"],
                                            "unfused_ms_per_step": round(tu["ms"], 4),
                                            "unfused_how": "the library's GEMMs with the product and its "
                                                           "backward as torch element-wise ops between them"}
                del tg, tu
            line["cpu_baseline"] = cpu_baseline(wl)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


def main(argv=None):
    from paper_2502_10940_gb300.workloads import WORKLOADS

    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="cola", choices=["cola", "reference"])
    ap.add_argument("--workload", default="7b", choices=sorted(WORKLOADS))
    ap.add_argument("--mode", default=None, choices=["cola", "cola_m", "infer"])
    ap.add_argument("--graph", default="on", choices=["on", "off"],
                    help="replay each step as one CUDA graph (off: launch every kernel from the host)")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--settle", type=float, default=SETTLE_S,
                    help="seconds of untimed steps after the warm-up, before the timed region")
    ap.add_argument("--no-extras", action="store_true", help="skip e2e, full-rank and CPU baselines")
    ap.add_argument("--fused-forward", default="on", choices=["on", "off"],
                    help="single-layer forwards with r <= 128: one fused kernel (on) or two GEMMs (off)")
    ap.add_argument("--gated-unfused", action="store_true",
                    help="gated workloads: the product and its backward as torch element-wise ops (comparison)")
    args = ap.parse_args(argv)
    args.warmup = max(3, args.warmup)   # at least 3 untimed warm-up steps, always
    args.steps = max(1, args.steps)
    wl = WORKLOADS[args.workload]
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_cola(args, wl)


if __name__ == "__main__":
    sys.exit(main())
