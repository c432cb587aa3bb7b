#!/usr/bin/env python3
"""Benchmark of the NVFP4 ScaleSweep hot path on GB300.

A step is one pass of the hot path over the largest single-GPU workload: two
Qwen2.5-72B-shaped weights, 8192x29568 and 29568x8192 (484.4M bf16 elements,
synthetic Laplace(0, 0.015) with 0.05% outlier input channels x30): the
global scale S = amax/(6*256) of each matrix, then ScaleSweep with the WMSE
objective (per-input-channel lognormal(0,1) weights), block 16, writing packed
FP4 codes plus linear and swizzled E4M3 scales -- one grouped launch that
reduces the scales while it sweeps.  The metric is Gelem/s of the whole step;
the kernel is also reported against its FP32 and HBM rooflines.  Every other
configuration (the 2048x2048 weight, the Llama-3-8B layer, the 8192x4096
activation, K/V/Q, and the Qwen shapes at blocks 16/32/64 with MSE and WMSE) is
timed as a leg in its own step's launch shape, beside AbsMax in the same shape.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl {gb300,reference}]

With N > 1 the script runs under torch.distributed.run: every rank quantises its
own copy of the workload (weak scaling, no collective on the data path); the
timed region is bracketed by barriers and the slowest rank's time is reported.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import statistics
import sys
import threading
import time

import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "qwen72b-b16-wmse"
# every other configuration is timed as a leg in its own step's launch shape
LEG_CONFIGS = ["qwen72b-b16-mse", "qwen72b-b32-mse", "qwen72b-b32-wmse", "qwen72b-b64-mse", "qwen72b-b64-wmse",
               "weight-2048", "llama8b", "act-8192", "kvq"]
METRIC = "NVFP4 ScaleSweep Gelem/s and % of GB300 HBM roofline; overhead vs AbsMax kernel"
L2_BYTES = 129 * 1024 * 1024


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """Samples SM clock and clock-event reasons through NVML (read-only) in a
    background thread while the timed region runs."""

    REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap", 0x8: "hw_slowdown",
               0x10: "sync_boost", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
               0x80: "hw_power_brake_slowdown", 0x100: "display_clock_setting"}

    def __init__(self, device_index: int = 0, period_s: float = 0.01):
        self.period = period_s
        self.samples: list[tuple[int, int]] = []
        self.max_mhz = None
        self.ok = False
        self._stop = threading.Event()
        try:
            self.nvml = ctypes.CDLL("libnvidia-ml.so.1")
            if self.nvml.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            props = torch.cuda.get_device_properties(device_index)
            found = False
            try:
                bus = f"{props.pci_domain_id:08x}:{props.pci_bus_id:02x}:{props.pci_device_id:02x}.0".encode()
                found = self.nvml.nvmlDeviceGetHandleByPciBusId_v2(ctypes.c_char_p(bus), ctypes.byref(self.h)) == 0
            except AttributeError:
                found = False
            if not found:
                try:
                    uuid = ("GPU-" + str(props.uuid)).encode()
                    found = self.nvml.nvmlDeviceGetHandleByUUID(ctypes.c_char_p(uuid), ctypes.byref(self.h)) == 0
                except AttributeError:
                    found = False
            if not found and self.nvml.nvmlDeviceGetHandleByIndex_v2(0, ctypes.byref(self.h)) != 0:
                return
            mx = ctypes.c_uint()
            if self.nvml.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = int(mx.value)
            self.ok = True
        except OSError:
            self.ok = False

    def _read(self):
        c = ctypes.c_uint()
        r = ctypes.c_ulonglong()
        if self.nvml.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(c)) != 0:
            return None
        if self.nvml.nvmlDeviceGetCurrentClocksEventReasons(self.h, ctypes.byref(r)) != 0:
            if self.nvml.nvmlDeviceGetCurrentClocksThrottleReasons(self.h, ctypes.byref(r)) != 0:
                r.value = 0
        return int(c.value), int(r.value)

    def _run(self):
        while not self._stop.is_set():
            s = self._read()
            if s:
                self.samples.append(s)
            time.sleep(self.period)

    def __enter__(self):
        if self.ok:
            self._t = threading.Thread(target=self._run, daemon=True)
            self._t.start()
        return self

    def __exit__(self, *a):
        if self.ok:
            self._stop.set()
            self._t.join()
            s = self._read()
            if s:
                self.samples.append(s)

    def summary(self) -> dict:
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [], "samples": 0,
                    "source": "nvml" if self.ok else "unavailable"}
        mhz = [m for m, _ in self.samples]
        bits = 0
        for _, r in self.samples:
            bits |= r
        reasons = [n for b, n in self.REASONS.items() if bits & b and n != "gpu_idle"]
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": self.max_mhz, "reasons": reasons,
                "samples": len(mhz), "source": "nvml"}


# ----------------------------------------------------------------------------- workload
_inputs_cache: dict = {}


def load_workload(name: str, device: str):
    """Device copies of a workload's tensors and WMSE weights (drawn once per
    distinct tensor set: the six Qwen2.5-72B-shaped configurations share it)."""
    from paper_2606_07618_gb300 import workloads as W
    wl = W.workload(name)
    key = tuple((t.seed, t.rows, t.cols) for t in wl.tensors)
    if key not in _inputs_cache:
        _inputs_cache.clear()
        torch.cuda.empty_cache()
        _inputs_cache[key] = ([W.draw(t).to(device) for t in wl.tensors],
                              [W.draw_weights(t).to(device) for t in wl.tensors])
    xs, ws = _inputs_cache[key]
    return wl, xs, ws


def make_inputs(device: str, name: str = "llama8b"):
    wl, xs, ws = load_workload(name, device)
    return wl, xs, ws


def candidates(wl) -> int:
    """Candidates per block of the default window (Sec. 4.2.2)."""
    return 11 if (wl.objective == "mse" and wl.block == 16) else 16


def alu_ops_per_elem(wl) -> int:
    """Algorithmic FP32 work of the sweep per element: per candidate one
    multiply (t = y r), one fma (e = y - q v), one fma accumulating e^2, and
    for WMSE one more multiply (w e)."""
    return (4 if wl.objective == "wmse" else 3) * candidates(wl)


def hbm_bytes(wl, xs, both_layouts=True):
    """Algorithmic HBM bytes of one step: the global-scale reduction reads each
    input once, the sweep reads it again and writes the packed codes and the
    scales (both layouts for block 16), plus the WMSE channel weights."""
    inb = xs[0].element_size()
    layouts = 2 if (both_layouts and wl.block == 16) else 1
    per_elem = inb + inb + 0.5 + layouts / wl.block
    wbytes = sum(4 * x.shape[1] for x in xs) if wl.objective == "wmse" else 0
    return sum(x.numel() for x in xs) * per_elem + wbytes


def traffic_per_launch(record, elems_per_launch):
    """DRAM bytes per launch from a committed ncu capture (profiles/<record>),
    scaled by elements; None if the kernel sources changed since the capture."""
    import hashlib
    path = os.path.join(ROOT, "profiles", record)
    try:
        with open(path) as f:
            rec = json.load(f)
        h = hashlib.sha256()
        for fn in rec["source_files"]:
            with open(os.path.join(ROOT, fn), "rb") as f:
                h.update(f.read())
        if h.hexdigest() != rec["source_sha256"]:
            return None
        return round(rec["dram_bytes_per_element"] * elems_per_launch)
    except (OSError, KeyError, ValueError):
        return None


def reduce_max_ms(ms: float, world: int, device) -> float:
    """Slowest rank's time (the whole-job time under weak scaling)."""
    if world <= 1:
        return ms
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def alg_bytes_per_elem(block=16, in_bytes=2, both_layouts=True):
    return in_bytes + 0.5 + (1.0 / block) * (2 if both_layouts else 1)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


class L2Flush:
    """Rewrites a buffer of twice the L2 size (on the timing stream) so that a
    timed call that follows starts with nothing of its inputs in L2."""

    def __init__(self, device):
        self.buf = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device)

    def __call__(self):
        self.buf.fill_(1.0)


def time_calls(fn, reps, stream, flush=None, warm=3):
    """Mean device time of one call (CUDA events on `stream`), optionally with
    L2 flushed before each call (then only the call is inside the events)."""
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    if flush is None:
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            fn()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    for a, b in ev:
        flush()
        a.record(stream)
        fn()
        b.record(stream)
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in ev) / reps


# ----------------------------------------------------------------------------- GPU arm
def run_gpu(args, rank, world):
    from paper_2606_07618_gb300 import binding as B
    from paper_2606_07618_gb300 import step as ST
    dev = f"cuda:{torch.cuda.current_device()}"
    stream = torch.cuda.current_stream()
    wl, xs, ws = load_workload(WORKLOAD, dev)
    total = sum(x.numel() for x in xs)
    st = ST.for_workload(wl, xs, ws)
    nsm = torch.cuda.get_device_properties(dev).multi_processor_count
    hbm_peak, peak_kind = peaks()

    # The step: one grouped call over both matrices that reduces each one's
    # global scale on the device and sweeps every block.  At this size the
    # library runs its pipelined schedule: the larger matrix's reduction, its
    # sweep with the other matrix's reduction running beside it on the
    # registers the sweep leaves free, then the other matrix's sweep.
    def step(events=None):
        if events is not None:
            events[0].record(stream)
        st(stream=stream)
        if events is not None:
            events[1].record(stream)

    # two reductions and two sweeps (the workspace reset is a memset; these
    # shapes need no swizzle pad kernel)
    launches_per_step = 4 if st.pipelined else 1

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device()) as clk:
        t0.record(stream)
        for k in range(args.steps):
            step(ev[k])
        t1.record(stream)
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    ms = t0.elapsed_time(t1)
    kern_ms = sum(ev[k][0].elapsed_time(ev[k][1]) for k in range(args.steps)) / args.steps
    ms = reduce_max_ms(ms, world, dev)
    ms_step = ms / args.steps
    value = world * total / (ms_step * 1e-3) / 1e9
    assert int(st.status.item()) == 0, "non-finite input detected"

    # ---- roofline of the step's kernels as one unit, from the per-step events
    # (the two reductions run beside the sweeps, so the call is the unit a
    # CUDA event can bracket without breaking the overlap)
    clk_sum = clk.summary()
    sm_mhz = clk_sum["sm_mhz"] or clk_sum["sm_max_mhz"] or 2070
    alu_peak = nsm * 128 * sm_mhz * 1e6

    def fracs(wl_, xs_, t_ms):
        n = sum(x.numel() for x in xs_)
        gbs = hbm_bytes(wl_, xs_) / (t_ms * 1e-3) / 1e9
        ops = alu_ops_per_elem(wl_) * n / (t_ms * 1e-3)
        return round(gbs, 1), round(gbs / hbm_peak, 4), round(ops / 1e12, 3), round(ops / alu_peak, 4)

    gbs, hfrac, tops, afrac = fracs(wl, xs, kern_ms)
    roofline = {"bound": "alu", "achieved": tops, "peak": round(alu_peak / 1e12, 3), "unit": "Tops/s",
                "frac": afrac, "traffic": None,
                "kernel": (f"quantize_group_kernel<bf16,ScaleSweep,WMSE,block {wl.block},pipelined S> x2 with "
                           f"group_reduce_kernel x2 beside them ({len(xs)} tensors, one call per step)")
                if st.pipelined else
                f"quantize_group_kernel<bf16,ScaleSweep,WMSE,block {wl.block},dynamic S> "
                f"({len(xs)} tensors, one launch per step)",
                "peak_note": f"{nsm} SMs x 128 FP32 lanes x median SM clock {sm_mhz} MHz "
                             f"(of measured clock; the work is {alu_ops_per_elem(wl)} FP32 ops per element: "
                             f"{candidates(wl)} candidates x 4, counted for every window candidate, including "
                             f"those the sweep's exact offset bound rules out without evaluating them)",
                "hbm": {"achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": hfrac, "peak_kind": peak_kind,
                        "bytes": round(hbm_bytes(wl, xs)), "bytes_per_elem": round(hbm_bytes(wl, xs) / total, 4)},
                "launch_ms": round(kern_ms, 4),
                "launch_note": "events around the call: the 256-byte workspace memset and the "
                               + ("four launches" if st.pipelined else "kernel")}
    # DRAM bytes of the step's launches from one ncu capture (null for the
    # two-phase schedule, which has no current record)
    roofline["traffic"] = traffic_per_launch("quantize_group_pipelined_qwen72b_traffic.json", total) \
        if st.pipelined else None

    reps = max(3, min(20, args.steps))
    flush = L2Flush(dev)
    legs = {}

    # ---- every configuration in its step's launch shape, and AbsMax in the same shape
    for name in ([] if args.no_legs else LEG_CONFIGS):
        wl_c, xs_c, ws_c = load_workload(name, dev)
        sc = ST.for_workload(wl_c, xs_c, ws_c)
        small = sum(x.numel() * x.element_size() for x in xs_c) < 2 * L2_BYTES
        fl = flush if small else None
        t_ss = time_calls(lambda: sc(stream=stream), reps, stream, fl)
        t_ab = time_calls(lambda: sc.absmax(stream=stream), reps, stream, fl)
        assert int(sc.status.item()) == 0
        n = sc.numel
        g, hf, tp, af = fracs(wl_c, xs_c, t_ss)
        legs[name] = {"elements": n, "launch": "fused dynamic" if sc.fused else f"grouped dynamic x{len(xs_c)}",
                      "block": wl_c.block, "objective": wl_c.objective, "D": wl_c.fp8_div, "ms": round(t_ss, 4),
                      "gelem_s": round(n / (t_ss * 1e-3) / 1e9, 2), "hbm_gbs": g, "hbm_frac": hf,
                      "fp32_tops": tp, "fp32_frac": af, "absmax_ms": round(t_ab, 4),
                      "overhead_vs_absmax": round(t_ss / t_ab, 3), "l2": "flushed before each call" if small
                      else "inputs > L2"}
        if small:                               # the same calls back to back, inputs left in L2
            t_hot = time_calls(lambda: sc(stream=stream), reps, stream)
            t_hot_ab = time_calls(lambda: sc.absmax(stream=stream), reps, stream)
            legs[name]["hot_l2"] = {"ms": round(t_hot, 4), "gelem_s": round(n / (t_hot * 1e-3) / 1e9, 2),
                                    "absmax_ms": round(t_hot_ab, 4),
                                    "overhead_vs_absmax": round(t_hot / t_hot_ab, 3)}
        del sc
    _inputs_cache.clear()                       # the headline's tensors stay referenced by xs / ws

    # ---- the headline workload's other legs
    def gel(t):
        return round(total / (t * 1e-3) / 1e9, 2)

    st_static = ST.QuantizeStep(xs, ws, block=wl.block, objective=B.NVFP4_OBJ_WMSE, fp8_div=wl.fp8_div)
    st_static(stream=stream)
    S_fixed = st_static.S.clone()

    def static_sweep():
        B.scalesweep_quantize_group(st_static.desc, st_static.dtype, B.NVFP4_OBJ_WMSE, 0.0, S_fixed, None, None,
                                    stream=stream, block=wl.block)

    def two_phase():
        B.scalesweep_quantize_group(st.desc, st.dtype, B.NVFP4_OBJ_WMSE, wl.fp8_div, st.S, st.status, st.workspace,
                                    stream=stream, block=wl.block, schedule=B.NVFP4_GROUP_SCHEDULE_TWO_PHASE)

    def absmax_static():
        B.absmax_quantize_group(st_static.desc, st_static.dtype, 0.0, S_fixed, None, None, stream=stream,
                                block=wl.block)

    gsw = [torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=dev) for x in xs]
    Sg = torch.empty(len(xs), device=dev)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)

    def per_tensor_launches():
        for i, x in enumerate(xs):
            o = st_static.outs[i]
            B.nvfp4_global_scale(x, wl.fp8_div, Sg[i:i + 1], None, gsw[i], stream=stream)
            B.scalesweep_quantize(x, wl.block, Sg[i:i + 1], B.NVFP4_OBJ_WMSE, ws[i], 0, *win, o["codes"],
                                  o["sf_linear"], o["sf_swizzled"], None, stream=stream)

    def four_six():
        for i, x in enumerate(xs):
            o = st_static.outs[i]
            B.four_over_six_quantize(x, wl.block, S_fixed[i:i + 1], B.NVFP4_OBJ_WMSE, ws[i], 0, o["codes"],
                                     o["sf_linear"], o["sf_swizzled"], None, stream=stream)

    dq = torch.empty(max(x.numel() for x in xs), dtype=torch.bfloat16, device=dev)

    def dequant():
        for i, x in enumerate(xs):
            o = st_static.outs[i]
            B.nvfp4_dequantize(o["codes"], o["sf_swizzled"], B.NVFP4_SF_SWIZZLED, S_fixed[i:i + 1], x.shape[0],
                               x.shape[1], wl.block, dq[:x.numel()], stream=stream)

    def global_scales():
        for i, x in enumerate(xs):
            B.nvfp4_global_scale(x, wl.fp8_div, Sg[i:i + 1], None, gsw[i], stream=stream)

    if args.no_legs:
        return dict(value=value, ms_step=ms_step, total=total, roofline=roofline, clocks=clk_sum, legs=None,
                    overhead=None, e2e=None, cpu=None, launches=launches_per_step * args.steps, wl=wl)
    t_gs = time_calls(static_sweep, reps, stream)
    t_2p = time_calls(two_phase, reps, stream)
    t_as = time_calls(absmax_static, reps, stream)
    t_pt = time_calls(per_tensor_launches, reps, stream)
    t_46 = time_calls(four_six, reps, stream)
    t_dq = time_calls(dequant, reps, stream)
    t_am = time_calls(global_scales, reps, stream)
    t_ab = legs[WORKLOAD]["absmax_ms"] if WORKLOAD in legs else time_calls(lambda: st.absmax(stream=stream), reps,
                                                                             stream)
    legs[WORKLOAD + " (headline) static scales"] = {
        "scalesweep_grouped_static": {"ms": round(t_gs, 4), "gelem_s": gel(t_gs)},
        "scalesweep_grouped_dynamic_two_phase_schedule": {"ms": round(t_2p, 4), "gelem_s": gel(t_2p)},
        "absmax_grouped_static": {"ms": round(t_as, 4), "gelem_s": gel(t_as)},
        "per_tensor_global_scale_then_sweep": {"ms": round(t_pt, 4), "gelem_s": gel(t_pt)},
        "four_over_six_wmse_per_tensor": {"ms": round(t_46, 4), "gelem_s": gel(t_46)},
        "dequant_bf16_swizzled": {"ms": round(t_dq, 4), "gelem_s": gel(t_dq)},
        "global_scale_per_tensor": {"ms": round(t_am, 4), "gelem_s": gel(t_am)}}
    overhead = {"scalesweep_wmse_vs_absmax_grouped_dynamic": round(kern_ms / t_ab, 3),
                "scalesweep_wmse_vs_absmax_grouped_static": round(t_gs / t_as, 3),
                "per_config": {k: v["overhead_vs_absmax"] for k, v in legs.items() if "overhead_vs_absmax" in v}}

    # ---- end to end through the public API (QuantizeStep) with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(wl, xs, ws, dev, stream, world, args)

    # ---- CPU baseline: the oracle on a bounded sample, rank 0 at N = 1 only
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu = cpu_baseline(wl, [x.cpu() for x in xs], [w.cpu() for w in ws], st.S.cpu(), budget_s=args.cpu_seconds)

    return dict(value=value, ms_step=ms_step, total=total, roofline=roofline, clocks=clk_sum, legs=legs,
                overhead=overhead, e2e=e2e, cpu=cpu, launches=launches_per_step * args.steps, wl=wl)


def run_e2e(wl, xs, ws, dev, stream, world, args):
    """The step through the public API with pinned host buffers: every step
    uploads its inputs, quantises them (one QuantizeStep call) and downloads
    codes and both scale layouts.  H2D, compute and D2H run on three streams,
    event-ordered per step, with two device buffer sets alternating so the
    upload of step k+1 only waits for the kernels of step k-1."""
    from paper_2606_07618_gb300 import step as ST
    hx = [x.cpu().pin_memory() for x in xs]
    sets = []
    for _ in range(2):
        dx = [torch.empty_like(x) for x in xs]
        sets.append((dx, ST.for_workload(wl, dx, ws)))
    hout = [{k: torch.empty_like(v, device="cpu").pin_memory() for k, v in o.items() if v is not None}
            for o in sets[0][1].outs]
    up, down = torch.cuda.Stream(), torch.cuda.Stream()
    comp_done = [torch.cuda.Event(), torch.cuda.Event()]
    d2h_done = [torch.cuda.Event(), torch.cuda.Event()]
    state = {"k": 0}

    def e2e_step():
        pb = state["k"] & 1
        first_use = state["k"] < 2
        state["k"] += 1
        dx, sc = sets[pb]
        if not first_use:
            up.wait_event(comp_done[pb])            # step k-2's kernels are done with this input set
        with torch.cuda.stream(up):
            for i in range(len(xs)):
                dx[i].copy_(hx[i], non_blocking=True)
        loaded = torch.cuda.Event()
        loaded.record(up)
        if not first_use:
            stream.wait_event(d2h_done[pb])         # step k-2's downloads are done with these outputs
        stream.wait_event(loaded)
        sc(stream=stream)
        comp_done[pb].record(stream)
        with torch.cuda.stream(down):
            down.wait_event(comp_done[pb])
            for i, o in enumerate(sc.outs):
                for k, h in hout[i].items():
                    h.copy_(o[k], non_blocking=True)
        d2h_done[pb].record(down)

    def e2e_time(reps):
        for _ in range(3):
            e2e_step()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        up.wait_stream(stream)
        for _ in range(reps):
            e2e_step()
        stream.wait_stream(up)
        stream.wait_stream(down)                    # the last step's results are on the host
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps

    # 30 steps per trial: the pipeline's fill and drain (one step's compute and
    # download) then cost ~1/30 of a step each, not 1/10
    e_reps = max(3, min(30, args.steps))
    total = sum(x.numel() for x in xs)
    h2d = sum(x.numel() * x.element_size() for x in xs)
    d2h = sum(h.numel() * h.element_size() for d in hout for h in d.values())
    dx0 = sets[0][0]

    def h2d_only():
        for i in range(len(xs)):
            dx0[i].copy_(hx[i], non_blocking=True)

    # The host link is shared with the rest of the machine (another GPU's
    # traffic through the same CPU has been seen to halve it for a while), so
    # the pipeline is timed in three trials, the median reported, and the link
    # is measured alone before and after them.
    t_h2d_before = time_calls(h2d_only, e_reps, stream)
    trials = sorted(e2e_time(e_reps) for _ in range(3))
    t_e2e = trials[1]
    t_h2d = time_calls(h2d_only, e_reps, stream)

    # zero-copy variant: the same call with inputs and outputs in pinned host
    # memory, so the kernels' loads and stores cross the host link themselves
    # (the in-launch global-scale phase reads the inputs a second time)
    zc_outs = [{k: torch.empty_like(v, device="cpu").pin_memory() if v is not None else None for k, v in o.items()}
               for o in sets[0][1].outs]
    zc = ST.QuantizeStep(hx, ws, block=wl.block, objective=sets[0][1].objective, fp8_div=wl.fp8_div, outs=zc_outs,
                         device=dev)
    t_zc = time_calls(lambda: zc(stream=stream), max(3, min(5, args.steps)), stream)
    assert int(zc.status.item()) == 0
    same = all(torch.equal(zc_outs[i][k], sets[0][1].outs[i][k].cpu()) for i in range(len(xs))
               for k in ("codes", "sf_linear"))
    return {"value": round(world * total / (t_e2e * 1e-3) / 1e9, 3), "unit": "Gelem/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": round(t_e2e, 4),
            "trials_ms_per_step": [round(t, 4) for t in trials],
            "h2d_gb_s_alone": round(h2d / (t_h2d * 1e-3) / 1e9, 1),
            "h2d_gb_s_alone_before": round(h2d / (t_h2d_before * 1e-3) / 1e9, 1),
            "link_bound_gelem_s": round(total / (t_h2d * 1e-3) / 1e9, 2),
            "streams": "H2D, compute and D2H on three streams, event-ordered per step, two buffer sets",
            "zero_copy": {"value": round(world * total / (t_zc * 1e-3) / 1e9, 3), "unit": "Gelem/s",
                          "ms_per_step": round(t_zc, 4), "same_outputs_as_copy_path": bool(same),
                          "path": "one QuantizeStep call on pinned host inputs and outputs: the kernels load "
                                  "the inputs over the host link twice (amax phase, sweep) and store the outputs "
                                  "over it"},
            "link_note": "the host link moves ~211 GB/s H2D and ~193 GB/s D2H whether copy engines (1-8 "
                         "streams) or SM loads drive it, so the copy pipeline is bound by the H2D of the "
                         "inputs (2 B/element)"}


def cpu_baseline(wl, xs_cpu, ws_cpu, S_cpu, budget_s=12.0, probe_rows=64):
    """Time the CPU oracle, as it stands, on leading rows of every tensor of the
    workload, sized to about `budget_s` seconds of wall time."""
    import oracle
    oracle.build()
    threads = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    obj = oracle.WMSE if wl.objective == "wmse" else oracle.MSE

    def run(rows, nthreads=threads):
        t = time.perf_counter()
        n = 0
        for i, x in enumerate(xs_cpu):
            r = min(rows, x.shape[0])
            xs = x[:r].float().numpy()
            S = float(S_cpu[i]) if S_cpu is not None else oracle.global_scale(xs, wl.fp8_div)[0]
            oracle.quantize(0, xs, wl.block, S, obj, w=ws_cpu[i].numpy() if obj == oracle.WMSE else None,
                            w_row_stride=0, nthreads=nthreads)
            n += xs.size
        return n, time.perf_counter() - t

    n, dt = run(probe_rows)
    rate = n / max(dt, 1e-6)
    per_row = sum(x.shape[1] for x in xs_cpu)
    rows = int(max(probe_rows, min(max(x.shape[0] for x in xs_cpu), budget_s * rate / per_row)))
    n, dt = run(rows)
    # the same oracle on one thread, on a sample of about a tenth of the time
    rows1 = int(max(8, min(rows, 0.1 * budget_s * (n / dt) / threads / per_row)))
    n1, dt1 = run(rows1, nthreads=1)
    return {"value": round(n / dt / 1e9, 6), "unit": "Gelem/s", "cores": threads, "kind": "oracle",
            "sample": f"first {rows} rows of each of the {len(xs_cpu)} {wl.name} tensors ({n} elements, "
                      f"{dt:.1f} s), same S, {wl.objective.upper()}, block {wl.block}",
            "one_thread": {"value": round(n1 / dt1 / 1e9, 6), "unit": "Gelem/s", "cores": 1,
                           "sample": f"first {rows1} rows of each tensor ({n1} elements, {dt1:.1f} s)"}}


# ----------------------------------------------------------------------------- reference arm
def run_reference(args, rank, world):
    if rank != 0:
        return None
    from paper_2606_07618_gb300 import workloads as W
    import oracle
    oracle.build()
    wl = W.workload(WORKLOAD)
    rows = args.ref_rows
    xs = [W.draw(t, rows=slice(0, rows)) for t in wl.tensors]
    ws = [W.draw_weights(t) for t in wl.tensors]
    threads = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    xf = [x.float().numpy() for x in xs]
    obj = oracle.WMSE if wl.objective == "wmse" else oracle.MSE

    def step():
        for x, w in zip(xf, ws):
            # the per-call global scale of the sample, then the sweep
            S = oracle.global_scale(x, wl.fp8_div)[0]
            oracle.quantize(0, x, wl.block, S, obj, w=w.numpy(), w_row_stride=0, nthreads=threads)

    for _ in range(args.warmup):
        step()
    t = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = (time.perf_counter() - t) / args.steps
    n = sum(x.size for x in xf)
    value = n / dt / 1e9
    return {"impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "Gelem/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": config_dict(wl, world),
            "cpu_baseline": {"value": round(value, 6), "unit": "Gelem/s", "cores": threads, "kind": "oracle",
                             "sample": f"first {rows} rows of each of the {len(xf)} {wl.name} tensors per step ({n} "
                                       f"elements): global scale of the sample, then the sweep, "
                                       f"{wl.objective.upper()}, block {wl.block}"},
            "e2e": {"value": round(value, 6), "unit": "Gelem/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def config_dict(wl, world):
    return {"workload": "qwen2.5-72b-shaped-weights-wmse-block16",
            "tensors": {t.name: [t.rows, t.cols] for t in wl.tensors},
            "elements": wl.numel, "input": "bf16", "block": wl.block, "objective": wl.objective,
            "global_scale": f"amax/(6*{int(wl.fp8_div)}) computed on the device every step, in the call",
            "scale_layouts": "linear+swizzled",
            "parallelism": f"replicas{world}" if world > 1 else "single-gpu",
            "l2": "no flush: each step streams the 968 MB of inputs (> 129 MB L2) twice, once for the global scales "
                  "and once for the sweep (the pipelined schedule: the larger matrix's reduction, then its sweep "
                  "with the other matrix's reduction beside it, then the other matrix's sweep)"}


def run_kernel_case(args):
    """One kernel on one synthetic [rows, cols] tensor (larger than L2 by
    default), timed with CUDA events; used for ncu captures and sweeps."""
    from paper_2606_07618_gb300 import binding as B
    from paper_2606_07618_gb300 import workloads as W
    dev = "cuda"
    x = W.small_tensor(args.rows, args.cols, 7, dist="normal", std=0.02, outliers=max(1, args.cols // 1000),
                       mult=20.0).to(dev)
    w = torch.exp(torch.randn(args.cols, generator=torch.Generator().manual_seed(3))).to(dev)
    S = torch.empty(1, device=dev)
    ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=dev)
    B.nvfp4_global_scale(x, 256.0, S, None, ws)
    o = B.empty_outputs(args.rows, args.cols, args.block, device=dev, linear=True, swizzled=args.block == 16)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    dq = torch.empty(args.rows, args.cols, dtype=torch.bfloat16, device=dev)
    dws = torch.empty(B.nvfp4_dynamic_workspace(), dtype=torch.uint8, device=dev)
    fns = {
        "sweep_wmse": lambda: B.scalesweep_quantize(x, args.block, S, 1, w, 0, *win, o["codes"], o["sf_linear"],
                                                    o["sf_swizzled"]),
        "sweep_mse": lambda: B.scalesweep_quantize(x, args.block, S, 0, None, 0, *win, o["codes"], o["sf_linear"],
                                                   o["sf_swizzled"]),
        "sweep_wmse_tight": lambda: B.scalesweep_quantize(x, args.block, S, 1, w, 0, B.NVFP4_WINDOW_TIGHT,
                                                          B.NVFP4_WINDOW_TIGHT, o["codes"], o["sf_linear"],
                                                          o["sf_swizzled"]),
        "sweep_mse_tight": lambda: B.scalesweep_quantize(x, args.block, S, 0, None, 0, B.NVFP4_WINDOW_TIGHT,
                                                         B.NVFP4_WINDOW_TIGHT, o["codes"], o["sf_linear"],
                                                         o["sf_swizzled"]),
        "absmax": lambda: B.absmax_quantize(x, args.block, S, o["codes"], o["sf_linear"], o["sf_swizzled"]),
        "four_six": lambda: B.four_over_six_quantize(x, args.block, S, 1, w, 0, o["codes"], o["sf_linear"],
                                                     o["sf_swizzled"]),
        "dequant": lambda: B.nvfp4_dequantize(o["codes"], o["sf_linear"], 1, S, args.rows, args.cols, args.block, dq),
        "dequant_swizzled": lambda: B.nvfp4_dequantize(o["codes"], o["sf_swizzled"], B.NVFP4_SF_SWIZZLED, S, args.rows,
                                                       args.cols, args.block, dq),
        "amax": lambda: B.nvfp4_global_scale(x, 256.0, S, None, ws),
        "mse_two_launch": lambda: (B.nvfp4_global_scale(x, 256.0, S, None, ws),
                                   B.scalesweep_quantize(x, args.block, S, 0, None, 0, *win, o["codes"],
                                                         o["sf_linear"], o["sf_swizzled"])),
        "mse_fused": lambda: B.scalesweep_quantize_dynamic(x, args.block, 256.0, 0, None, 0, *win, S, None, dws,
                                                           o["codes"], o["sf_linear"], o["sf_swizzled"]),
        "wmse_fused": lambda: B.scalesweep_quantize_dynamic(x, args.block, 256.0, 1, w, 0, *win, S, None, dws,
                                                            o["codes"], o["sf_linear"], o["sf_swizzled"]),
    }
    S1 = torch.empty(1, device=dev)
    gws = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=dev)
    d1 = B.group_descriptors([x], [w], [0], [o["codes"]], [o["sf_linear"]], [o["sf_swizzled"]])
    fns["sweep_wmse_group"] = lambda: B.scalesweep_quantize_group(d1, B.NVFP4_IN_BF16, 1, 0.0, S, None, None)
    fns["wmse_group_dynamic"] = lambda: B.scalesweep_quantize_group(d1, B.NVFP4_IN_BF16, 1, 256.0, S1, None, gws)
    if args.kernel_case.startswith("qwen"):
        # the headline step (both Qwen2.5-72B-shaped matrices, WMSE, in-launch
        # scales), or a slice of each (2048 and 7392 leading rows: 242 MB of
        # inputs, still above L2) for profiler captures
        from paper_2606_07618_gb300 import step as ST
        if args.kernel_case.startswith("qwen_slice"):
            from paper_2606_07618_gb300 import workloads as W
            wlq = W.workload(WORKLOAD)
            qx = [W.draw(t, rows=slice(0, r)).to(dev) for t, r in zip(wlq.tensors, (2048, 7392))]
            qw = [W.draw_weights(t).to(dev) for t in wlq.tensors]
        else:
            wlq, qx, qw = load_workload(WORKLOAD, dev)
        sq = ST.for_workload(wlq, qx, qw)
        fns["qwen_group"] = fns["qwen_slice_group"] = lambda: sq()
        fns["qwen_absmax_group"] = fns["qwen_slice_absmax_group"] = lambda: sq.absmax()
        sq()
        Sq = sq.S.clone()
        fns["qwen_group_static"] = fns["qwen_slice_group_static"] = lambda: B.scalesweep_quantize_group(
            sq.desc, B.NVFP4_IN_BF16, 1, 0.0, Sq, None, None, block=wlq.block)
        n = sq.numel
    elif args.kernel_case.startswith(("group_layer", "layer_")):
        # the Llama-3-8B layer in one grouped launch (dynamic scales), as the bench step
        _, xs, wl_ws = make_inputs(dev)
        lo = [B.empty_outputs(t.shape[0], t.shape[1], 16, device=dev, linear=True, swizzled=True) for t in xs]
        dl = B.group_descriptors(xs, wl_ws, [0] * len(xs), [q["codes"] for q in lo], [q["sf_linear"] for q in lo],
                                 [q["sf_swizzled"] for q in lo])
        SL = torch.empty(len(xs), device=dev)
        fns["group_layer"] = lambda: B.scalesweep_quantize_group(dl, B.NVFP4_IN_BF16, 1, 256.0, SL, None, gws)
        SS = torch.empty(len(xs), device=dev)
        B.scalesweep_quantize_group(dl, B.NVFP4_IN_BF16, 1, 256.0, SS, None, gws)
        fns["group_layer_static"] = lambda: B.scalesweep_quantize_group(dl, B.NVFP4_IN_BF16, 1, 0.0, SS, None, None)
        dlin = B.group_descriptors(xs, wl_ws, [0] * len(xs), [q["codes"] for q in lo], [q["sf_linear"] for q in lo],
                                   [None] * len(xs))
        fns["group_layer_linear"] = lambda: B.scalesweep_quantize_group(dlin, B.NVFP4_IN_BF16, 1, 256.0, SL, None, gws)
        fns["group_layer_static_linear"] = lambda: B.scalesweep_quantize_group(dlin, B.NVFP4_IN_BF16, 1, 0.0, SS, None,
                                                                               None)
        fns["layer_per_tensor_static"] = lambda: [
            B.scalesweep_quantize(t, 16, SS[i:i + 1], 1, wl_ws[i], 0, *win, lo[i]["codes"], lo[i]["sf_linear"],
                                  lo[i]["sf_swizzled"]) for i, t in enumerate(xs)]
        n = sum(t.numel() for t in xs)
    else:
        n = x.numel()
    fn = fns[args.kernel_case]
    fns["sweep_mse"]()
    for _ in range(2):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.reps):
        fn()
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.reps
    print(json.dumps({"kernel_case": args.kernel_case, "rows": args.rows, "cols": args.cols, "block": args.block,
                      "ms": round(ms, 4), "gelem_s": round(n / ms / 1e6, 2)}), flush=True)


def run_table7(args):
    """Latency of the NVFP4 quantisation operator at hidden 8192 for the batch
    sizes of the paper's latency table (Appendix E, Table 7), on this GPU:
    per-call global scale + ScaleSweep (MSE and WMSE) or AbsMax, both scale
    layouts, timed with CUDA events (context for the paper's RTX PRO 6000
    figures, not a like-for-like comparison)."""
    from paper_2606_07618_gb300 import binding as B
    from paper_2606_07618_gb300 import workloads as W
    dev = "cuda"
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    l2 = torch.cuda.get_device_properties(torch.cuda.current_device()).L2_cache_size
    flush = torch.empty(2 * l2 // 4, dtype=torch.float32, device=dev)
    rows = []
    for b in (128, 256, 512, 1024, 2048, 4096, 8192, 16384, 32768):
        t = W.workload(f"table7-{b}").tensors[0]
        x = W.draw(t).to(dev)
        w = torch.exp(torch.randn(t.cols, generator=torch.Generator().manual_seed(b))).to(dev)
        S = torch.empty(1, device=dev)
        ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=dev)
        o = B.empty_outputs(b, t.cols, 16, device=dev, linear=True, swizzled=True)

        B.nvfp4_global_scale(x, 256.0, S, None, ws)     # static scale: computed once, as in the paper
        dws = torch.empty(B.nvfp4_dynamic_workspace(), dtype=torch.uint8, device=dev)
        S2 = torch.empty(1, device=dev)

        def op(kind):
            def f():
                if kind.endswith("_fused"):
                    if kind.startswith("absmax"):
                        B.absmax_quantize_dynamic(x, 16, 256.0, S2, None, dws, o["codes"], o["sf_linear"],
                                                  o["sf_swizzled"])
                    else:
                        obj = B.NVFP4_OBJ_WMSE if kind.startswith("wmse") else B.NVFP4_OBJ_MSE
                        B.scalesweep_quantize_dynamic(x, 16, 256.0, obj, w if obj else None, 0, *win, S2, None,
                                                      dws, o["codes"], o["sf_linear"], o["sf_swizzled"])
                    return
                if kind.endswith("_dyn"):
                    B.nvfp4_global_scale(x, 256.0, S, None, ws)
                    kind_ = kind[:-4]
                else:
                    kind_ = kind
                if kind_ == "absmax":
                    B.absmax_quantize(x, 16, S, o["codes"], o["sf_linear"], o["sf_swizzled"])
                else:
                    obj = B.NVFP4_OBJ_WMSE if kind_ == "wmse" else B.NVFP4_OBJ_MSE
                    B.scalesweep_quantize(x, 16, S, obj, w if kind_ == "wmse" else None, 0, *win, o["codes"],
                                          o["sf_linear"], o["sf_swizzled"])
            return f

        res = {"batch": b}
        reps = 50
        for kind in ("absmax", "mse", "wmse", "absmax_dyn", "mse_dyn", "wmse_dyn", "absmax_fused", "mse_fused",
                     "wmse_fused"):
            f = op(kind)
            for _ in range(5):
                f()
            torch.cuda.synchronize()
            a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for _ in range(reps):
                f()
            e.record()
            torch.cuda.synchronize()
            res[kind + "_ms"] = round(a.elapsed_time(e) / reps, 4)
        # Cold L2: before every timed call a buffer of twice the L2 size is
        # rewritten (the call's own launch is already queued when the flush ends,
        # so the events see the device time of the call with its inputs in HBM).
        for kind in ("absmax", "mse", "wmse"):
            f = op(kind)
            tot = 0.0
            for _ in range(20):
                flush.add_(1.0)
                a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                f()
                e.record()
                torch.cuda.synchronize()
                tot += a.elapsed_time(e)
            res[kind + "_l2flush_ms"] = round(tot / 20, 4)
        # The same calls captured once in a CUDA graph and replayed: the library
        # never allocates or synchronises, so a caller can remove the per-call
        # host cost this way; what remains is the device time per call.
        for kind in ("absmax", "mse", "wmse", "mse_dyn", "wmse_dyn"):
            f = op(kind)
            try:
                side = torch.cuda.Stream()
                side.wait_stream(torch.cuda.current_stream())
                with torch.cuda.stream(side):
                    for _ in range(3):
                        f()
                torch.cuda.current_stream().wait_stream(side)
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    for _ in range(reps):
                        f()
                g.replay()
                torch.cuda.synchronize()
                a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                for _ in range(4):
                    g.replay()
                e.record()
                torch.cuda.synchronize()
                res[kind + "_graph_ms"] = round(a.elapsed_time(e) / (4 * reps), 4)
            except RuntimeError as exc:          # capture refused: report, keep the eager numbers
                res[kind + "_graph_ms"] = None
                res[kind + "_graph_error"] = str(exc)[:120]
        res["mse_rel"] = round(res["mse_ms"] / res["absmax_ms"], 3)
        res["wmse_rel"] = round(res["wmse_ms"] / res["absmax_ms"], 3)
        rows.append(res)
        print(json.dumps(res), flush=True)


def run_quality(args):
    """Quantisation error of AbsMax, 4/6, ScaleSweep, the FP8-quantised optimal
    scale and the optimal FP32 scale (Appendix C) on synthetic 72B-shaped Laplace
    weights -- the analogue of the paper's Fig. 1 (block sizes 16/32/64, MSE and
    WMSE) and Fig. 2 (global scale divisor D).  NMSE = sum w (x - x_hat)^2 /
    sum w x^2 over the sampled rows; gap = NMSE / NMSE(optimal FP32) - 1."""
    from paper_2606_07618_gb300 import binding as B
    from paper_2606_07618_gb300 import workloads as W
    dev = "cuda"
    wl = W.workload("qwen72b-b16-mse")
    xs = [W.draw(t, rows=slice(0, args.quality_rows)).to(dev) for t in wl.tensors]
    ws_ = [W.draw_weights(t).to(dev) for t in wl.tensors]
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)

    def study(block, obj, D):
        num = {k: 0.0 for k in ("absmax", "four_six", "scalesweep", "fp8_opt", "fp32_opt")}
        den = 0.0
        for x, w in zip(xs, ws_):
            rows, cols = x.shape
            S = torch.empty(1, device=dev)
            wsp = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=dev)
            B.nvfp4_global_scale(x, D, S, None, wsp)
            wt = w if obj else None
            wf = (w.double() if obj else torch.ones(cols, dtype=torch.float64, device=dev))
            xd = x.double()
            den += float((xd * xd * wf).sum())
            o = B.empty_outputs(rows, cols, block, device=dev, linear=True)
            deq = torch.empty(rows, cols, device=dev)
            for name in ("absmax", "four_six", "scalesweep"):
                if name == "absmax":
                    B.absmax_quantize(x, block, S, o["codes"], o["sf_linear"])
                elif name == "four_six":
                    B.four_over_six_quantize(x, block, S, obj, wt, 0, o["codes"], o["sf_linear"])
                else:
                    B.scalesweep_quantize(x, block, S, obj, wt, 0, *win, o["codes"], o["sf_linear"])
                B.nvfp4_dequantize(o["codes"], o["sf_linear"], B.NVFP4_SF_LINEAR, S, rows, cols, block, deq)
                num[name] += float(((xd - deq.double()) ** 2 * wf).sum())
            nb = rows * cols // block
            so, lo = torch.empty(nb, device=dev), torch.empty(nb, device=dev)
            code, lf = torch.empty(nb, dtype=torch.uint8, device=dev), torch.empty(nb, device=dev)
            B.nvfp4_optimal_scale(x, block, S, obj, wt, 0, so, lo, code, lf)
            s2 = float(S.item()) ** 2
            num["fp32_opt"] += float(lo.double().sum()) * s2
            num["fp8_opt"] += float(lf.double().sum()) * s2
        nm = {k: v / den for k, v in num.items()}
        gap = {k: round(nm[k] / nm["fp32_opt"] - 1.0, 5) for k in nm if k != "fp32_opt"}
        return {"block": block, "objective": "wmse" if obj else "mse", "D": D,
                "nmse": {k: float(f"{v:.6g}") for k, v in nm.items()}, "gap_vs_fp32_opt": gap}

    out = []
    for block in (16, 32, 64):
        for obj in (0, 1):
            out.append(study(block, obj, 256.0))
            print(json.dumps(out[-1]), flush=True)
    for D in (448.0, 384.0, 192.0, 128.0, 64.0):
        out.append(study(16, 0, D))
        print(json.dumps(out[-1]), flush=True)
    return out


def run_ldlq(args):
    """LDLQ (GPTQ with ScaleSweep scales, static reordering; Appendix A.2) on the
    Llama-3-8B layer shapes: the Hessian factorization per input width and the
    error-feedback pass per weight, CUDA-event timed, with the proxy loss
    tr(E H E^T) of LDLQ vs rounding at the same scales on sampled rows.
    Synthetic Hessians: low-rank (256) plus diagonal with lognormal channel
    scales (sigma 0.8), built with torch matmul outside the timed region."""
    from paper_2606_07618_gb300 import binding as B
    dev = "cuda"
    g = torch.Generator().manual_seed(23)
    hess = {}
    rows_out = []
    shapes = (("q", (4096, 4096)), ("k", (1024, 4096)), ("gate", (14336, 4096)), ("down", (4096, 14336)))
    if args.ldlq_shape:
        r_, c_ = (int(v) for v in args.ldlq_shape.split("x"))
        shapes = (("custom", (r_, c_)),)
    for n in sorted({c for _, (_, c) in shapes}):
        scale = torch.exp(torch.randn(n, generator=g) * 0.8).to(dev)
        A = torch.randn(n, 256, generator=g).to(dev) * scale[:, None]
        H = (A @ A.T) / 256 + torch.diag(scale * scale * 0.05)
        perm = torch.empty(n, dtype=torch.int32, device=dev)
        U = torch.empty(n, n, device=dev)
        D = torch.empty(n, device=dev)
        st = torch.zeros(1, dtype=torch.int32, device=dev)
        ws = torch.empty(B.nvfp4_ldlq_prepare_workspace(n), dtype=torch.uint8, device=dev)
        B.nvfp4_ldlq_prepare(H, 0.01, perm, U, D, st, ws)
        torch.cuda.synchronize()
        a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = max(1, args.reps // 2)
        a.record()
        for _ in range(reps):
            B.nvfp4_ldlq_prepare(H, 0.01, perm, U, D, st, ws)
        e.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(e) / reps
        hess[n] = (H, perm, U)
        rows_out.append({"ldlq_prepare": n, "ms": round(ms, 3), "status": int(st.item()),
                         "tflops_fp32": round(2 * n ** 3 / 3 / (ms * 1e-3) / 1e12, 2)})
        print(json.dumps(rows_out[-1]), flush=True)
    for name, (rows, cols) in shapes:
        H, perm, U = hess[cols]
        W = (torch.randn(rows, cols, generator=g) * 0.02).to(torch.bfloat16).to(dev)
        S = torch.empty(1, device=dev)
        gws = torch.empty(B.nvfp4_global_scale_workspace(W.numel()), dtype=torch.uint8, device=dev)
        B.nvfp4_global_scale(W, 256.0, S, None, gws)
        sf = torch.empty(rows, cols // 16, dtype=torch.uint8, device=dev)
        rtn = torch.empty(rows, cols // 2, dtype=torch.uint8, device=dev)
        imp = torch.diagonal(H).contiguous()
        B.scalesweep_quantize(W, 16, S, B.NVFP4_OBJ_WMSE, imp, 0, B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT,
                              rtn, sf)
        codes = torch.empty_like(rtn)
        st = torch.zeros(1, dtype=torch.int32, device=dev)
        ws = torch.empty(B.nvfp4_ldlq_workspace(rows, cols), dtype=torch.uint8, device=dev)
        B.ldlq_quantize(W, 16, S, sf, perm, U, codes, st, ws)
        torch.cuda.synchronize()
        a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = max(1, args.reps // 2)
        a.record()
        for _ in range(reps):
            B.ldlq_quantize(W, 16, S, sf, perm, U, codes, st, ws)
        e.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(e) / reps
        # proxy loss on 256 sampled rows (evaluation only)
        idx = torch.linspace(0, rows - 1, 256, device=dev).long()
        losses = []
        for c in (codes, rtn):
            xh = torch.empty(256, cols, device=dev)
            B.nvfp4_dequantize(c[idx].contiguous(), sf[idx].contiguous(), B.NVFP4_SF_LINEAR, S, 256, cols, 16, xh)
            E = W[idx].float() - xh
            losses.append(float(((E @ H) * E).sum()))
        rows_out.append({"ldlq_quantize": name, "rows": rows, "cols": cols, "ms": round(ms, 3),
                         "status": int(st.item()), "gemm_tflops_fp32": round(rows * cols * cols / (ms * 1e-3) / 1e12, 2),
                         "proxy_loss_ldlq_over_rtn": round(losses[0] / losses[1], 4)})
        print(json.dumps(rows_out[-1]), flush=True)
    return rows_out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-legs", action="store_true", help="time the headline step only (profiler launch lists)")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--ref-rows", type=int, default=64)
    ap.add_argument("--kernel-case", default=None,
                    choices=["sweep_wmse", "sweep_mse", "absmax", "four_six", "dequant", "dequant_swizzled", "amax",
                             "mse_two_launch",
                             "sweep_wmse_group", "wmse_group_dynamic", "group_layer", "group_layer_static",
                             "sweep_wmse_tight", "sweep_mse_tight",
                             "layer_per_tensor_static", "group_layer_linear", "group_layer_static_linear",
                             "mse_fused", "wmse_fused", "qwen_group", "qwen_group_static", "qwen_absmax_group",
                             "qwen_slice_group", "qwen_slice_group_static", "qwen_slice_absmax_group"])
    ap.add_argument("--rows", type=int, default=16384)
    ap.add_argument("--cols", type=int, default=8192)
    ap.add_argument("--block", type=int, default=16)
    ap.add_argument("--reps", type=int, default=5)
    ap.add_argument("--table7", action="store_true")
    ap.add_argument("--quality", action="store_true")
    ap.add_argument("--quality-rows", type=int, default=2048)
    ap.add_argument("--ldlq", action="store_true")
    ap.add_argument("--ldlq-shape", default=None, help="one ROWSxCOLS weight instead of the Llama-3-8B shapes")
    args = ap.parse_args()
    if args.ldlq:
        run_ldlq(args)
        return
    if args.quality:
        run_quality(args)
        return
    if args.table7:
        run_table7(args)
        return
    if args.kernel_case:
        run_kernel_case(args)
        return
    if args.warmup < 3:
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        res = run_reference(args, rank, world)
        if res is not None:
            print(json.dumps(res), flush=True)
        return
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (the library has no CPU path)")
    torch.cuda.set_device(local)
    if world > 1:
        torch.distributed.init_process_group("nccl")
    r = run_gpu(args, rank, world)
    if rank == 0:
        wl = r["wl"]
        out = {"metric": METRIC, "value": round(r["value"], 3), "unit": "Gelem/s", "n_gpus": world,
               "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(r["ms_step"], 4),
               "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
               "data": "synthetic (seeded Laplace(0,0.015) Qwen2.5-72B-shaped weights with x30 outlier channels, "
                       "lognormal channel weights)",
               "config": config_dict(wl, world), "roofline": r["roofline"], "clocks": r["clocks"],
               "gpu_launches": r["launches"], "legs": r["legs"], "overhead_vs_absmax": r["overhead"],
               "e2e": r["e2e"], "cpu_baseline": r["cpu"]}
        print(json.dumps(out), flush=True)
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
