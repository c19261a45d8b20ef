#!/usr/bin/env python
"""Throughput of the W4A4 quantized linear hot path on the backbone-shaped gated-MLP block.

One step = one pass of the whole online path over one batch: for 816 prefix tokens of hidden
size 2048 (bf16), rotate + quantise the input (Hadamard 2048, per-token int4), the gate/up
projection 2048 -> 2 x 16384 as one int4 GEMM whose epilogue dequantises and applies the GELU
gate (h = gelu(gate) * up), rotate + quantise h (Hadamard 8 x 2048, per-token int4) and the
down projection 16384 -> 2048.  Algorithmic work: 2 * 816 * (2048 * 32768 + 16384 * 2048)
= 164.3 G integer ops per step.  Inputs are synthetic (seeded Gaussian activations with 1%
Student-t channels, Gaussian weights) in the shapes of the Pi-0.5 backbone MLP.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints one JSON line (rank 0).  Under torchrun each rank runs its own replica of the block
(weak scaling, no collective on the data path); the time is the maximum over ranks.

The line also carries the two layer stacks (skipped with --no-stacks):
  "dit": the DiT action head, 18 blocks (qkv 1024 -> 3072, o 1024 -> 1024, up 1024 -> 4096,
         down 4096 -> 1024) at M = 50 tokens with per-step scale tables, one CUDA graph per
         denoising step: microseconds per step (L2 flushed before each) and per 10-step rollout;
  "backbone": 18 layers of hidden 2048 with the gated 16384 MLP, per-token scales, one forward
         pass at M = 816 (TOPS) and at M = 1 (HBM-bound: GB/s of packed weights; one kernel
         per linear);
  "dit"."w4a8" and "w4a8_gate_up": the W4A8 variant (8-bit activation codes) on the DiT stack
         and on the backbone's gate/up projection;
  "dit"."grouped": the DiT stack with Hadamard blocks of 64 and per-step, per-group tables.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

M, K_IN, HIDDEN = 816, 2048, 16384
HAD_IN, HAD_HIDDEN = 2048, 2048
OPS_GATEUP = 2 * M * K_IN * 2 * HIDDEN
OPS_DOWN = 2 * M * HIDDEN * K_IN
OPS_STEP = OPS_GATEUP + OPS_DOWN
METRIC = "W4A4 linear TOPS"
WORKLOAD = ("backbone gated-MLP block: 816 tokens x 2048 -> gate/up 2x16384 (GELU-gated) -> down 2048, "
            "bf16 activations, per-token int4 activations, per-channel int4 weights, Hadamard 2048")
FP8_OVER_BF16 = 4.5 / 2.25  # nominal dense tensor-rate ratio (E4M3 operands vs bf16)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--sets", type=int, default=3, help="rotating weight+activation sets (working set > L2)")
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="CPU-baseline sample budget")
    ap.add_argument("--no-stacks", action="store_true", help="skip the DiT and backbone stack legs")
    ap.add_argument("--no-sweep", action="store_true", help="skip the single-layer and sweep legs")
    ap.add_argument("--sweep-points", default=None,
                    help="only time these sweep points, 'M,K,N;M,K,N' (a short run for profiling); prints their line")
    return ap.parse_args()


# --------------------------------------------------------------------------------------
# distributed plumbing (timing only; the data path has no collective)
# --------------------------------------------------------------------------------------

def dist_init():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist

        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def job_value(world: int, ops_per_step: float, steps: int, ms: float) -> float:
    """Whole-job TOPS: every rank runs `steps` steps of its own replica (weak scaling); `ms` is
    the slowest rank's time."""
    return world * ops_per_step * steps / (ms * 1e-3) / 1e12


def max_over_ranks(world, value: float, device) -> float:
    if world == 1:
        return value
    import torch.distributed as dist

    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --------------------------------------------------------------------------------------
# measured peaks, clocks, ncu traffic
# --------------------------------------------------------------------------------------

def peaks():
    """Measured roofline denominators: E4M3 tensor rate as the measured bf16 GEMM rate times the
    nominal E4M3/bf16 ratio, burst (a kernel timed alone) and sustained (inside a long loop),
    and the HBM copy bandwidth."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"tflops": d["bf16_tflops"] * FP8_OVER_BF16, "tflops_sustained": d["bf16_tflops_sustained"] * FP8_OVER_BF16,
                "gbs": d["hbm_gbs"], "src": "measured"}
    return {"tflops": 1900.0 * FP8_OVER_BF16, "tflops_sustained": 1700.0 * FP8_OVER_BF16, "gbs": 6800.0, "src": "fallback"}


class _Nvml:
    """The few NVML queries the clock record needs, through ctypes (reading only)."""
    SM = 1  # NVML_CLOCK_SM
    REASONS = {0x8: "hw_slowdown", 0x40: "hw_thermal_slowdown", 0x20: "sw_thermal_slowdown", 0x4: "sw_power_cap"}

    def __init__(self, device_index: int):
        import ctypes

        self.c = ctypes
        lib = ctypes.CDLL("libnvidia-ml.so.1")
        if lib.nvmlInit_v2() != 0:
            raise OSError("nvmlInit failed")
        self.lib = lib
        self.h = ctypes.c_void_p()
        props = torch.cuda.get_device_properties(device_index)
        bus = None
        if all(hasattr(props, a) for a in ("pci_domain_id", "pci_bus_id", "pci_device_id")):
            bus = f"{props.pci_domain_id:08x}:{props.pci_bus_id:02x}:{props.pci_device_id:02x}.0".encode()
        if bus is None or lib.nvmlDeviceGetHandleByPciBusId_v2(bus, ctypes.byref(self.h)) != 0:
            if lib.nvmlDeviceGetHandleByIndex_v2(device_index, ctypes.byref(self.h)) != 0:
                raise OSError("no NVML handle")
        self.reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            lib.nvmlDeviceGetCurrentClocksThrottleReasons

    def sample(self):
        c = self.c
        mhz, mx, mw, rs = c.c_uint(), c.c_uint(), c.c_uint(), c.c_ulonglong()
        if self.lib.nvmlDeviceGetClockInfo(self.h, self.SM, c.byref(mhz)) != 0:
            return None
        self.lib.nvmlDeviceGetMaxClockInfo(self.h, self.SM, c.byref(mx))
        self.lib.nvmlDeviceGetPowerUsage(self.h, c.byref(mw))
        self.reasons_fn(self.h, c.byref(rs))
        reasons = [name for bit, name in self.REASONS.items() if rs.value & bit]
        return float(mhz.value), float(mx.value), mw.value / 1000.0, reasons


class ClockSampler:
    """SM clocks, power and slowdown reasons sampled every few milliseconds from a host thread
    while the GPU runs; each sample is tagged with whether the timed region was running (its
    start event had completed and its end event had not).  NVML through ctypes; nvidia-smi at
    200 ms when NVML cannot be opened."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, period_s: float = 0.002):
        self.gpu = gpu_index
        self.period = period_s
        self.samples = []
        self.region = None  # (start event, end event) of the timed region
        self.proc = self.thread = self.nvml = None
        self.stop_flag = False

    def start(self, region=None):
        import threading

        self.region = region
        try:
            self.nvml = _Nvml(self.gpu)
        except (OSError, AttributeError):
            self.nvml = None
        if self.nvml is not None:
            self.thread = threading.Thread(target=self._poll, daemon=True)
            self.thread.start()
            return
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None

    def _in_region(self):
        if self.region is None:
            return False
        a, b = self.region
        try:
            return a.query() and not b.query()
        except RuntimeError:
            return False

    def _poll(self):
        while not self.stop_flag:
            r = self.nvml.sample()
            if r is not None:
                self.samples.append(r + (self._in_region(),))
            time.sleep(self.period)

    def _smi_rows(self):
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        rows = []
        for r in (r.split(", ") for r in out.strip().splitlines() if r.strip()):
            try:
                rows.append((float(r[1]), float(r[2]), float(r[3]),
                             [n for n, v in zip(names, r[5:9]) if v.strip().lower() == "active"], False))
            except (ValueError, IndexError):
                continue
        return rows

    def stop(self):
        if self.thread is not None:
            self.stop_flag = True
            self.thread.join(timeout=5)
            rows, how = self.samples, "NVML every 2 ms"
        elif self.proc is not None:
            rows, how = self._smi_rows(), "nvidia-smi every 200 ms"
        else:
            return None
        return self.summarize(rows, how)

    @staticmethod
    def summarize(rows, how):
        """rows: (sm MHz, max SM MHz, watts, [slowdown reasons], inside the timed region)."""
        if not rows:
            return None
        inside = [r for r in rows if r[4]]
        use = inside if len(inside) >= 3 else rows
        reasons = sorted({n for r in use for n in r[3]})
        return {"sm_mhz": statistics.median(r[0] for r in use), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "power_w_max": round(max(r[2] for r in use), 1), "samples": len(use),
                "samples_in_timed_region": len(inside),
                "window": ("the timed region" if use is inside else
                           "back-to-back steps bracketing the timed region (too short to sample alone)"),
                "how": how}


def gemm_source_hash():
    """sha256 over the GEMM kernel's sources (the kernel template and its dispatch)."""
    h = hashlib.sha256()
    for f in ("gemm_kernel.cuh", "gemm.cu", "ptx.cuh"):
        h.update(open(os.path.join(ROOT, "paper_2605_28803_gb300", "csrc", f), "rb").read())
    return h.hexdigest()


def gemm_traffic():
    """dram bytes per launch of the GEMM kernel from the committed ncu summary, or None if the
    kernel source changed since the counters were taken."""
    p = os.path.join(ROOT, "profiles", "gemm_w4a4_traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p))
    if gemm_source_hash() != d.get("gemm_source_sha256"):
        return None
    return d.get("dram_bytes_per_step")


# --------------------------------------------------------------------------------------
# the workload
# --------------------------------------------------------------------------------------

def pack_workload():
    from paper_2605_28803_gb300 import qvla as Q
    from paper_2605_28803_gb300 import workloads as W

    mlp = W.gated_mlp(seed=1, m=M, k=K_IN, hidden=HIDDEN, had_in=HAD_IN, had_hidden=HAD_HIDDEN)
    packed = {}
    for name, w, had in (("gate", mlp.w_gate, HAD_IN), ("up", mlp.w_up, HAD_IN), ("down", mlp.w_down, HAD_HIDDEN)):
        n, k = w.shape
        wq = np.zeros((n, k // 2), np.uint8)
        ws = np.zeros(n, np.float32)
        Q.qvla_pack_weights_host(np.ascontiguousarray(w), Q.F32, n, k, had_block=had, wq=wq, wscale=ws)
        packed[name] = (wq, ws)
    return mlp, packed


def run_ours(args):
    from paper_2605_28803_gb300 import qvla as Q

    world, rank, local = dist_init()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream()
    mlp, packed = pack_workload()

    sets = []
    for _ in range(args.sets):
        gu = Q.qvla_layer_create_gated(HIDDEN, K_IN, HAD_IN, Q.BF16, Q.BF16, packed["gate"][0], packed["gate"][1],
                                       packed["up"][0], packed["up"][1])
        dn = Q.qvla_layer_create(K_IN, HIDDEN, HAD_HIDDEN, Q.BF16, Q.BF16, packed["down"][0], packed["down"][1])
        s = {
            "gu": gu, "dn": dn,
            "x": mlp.x.to(dev),
            "h": torch.empty(M, HIDDEN, dtype=torch.bfloat16, device=dev),
            "y": torch.empty(M, K_IN, dtype=torch.bfloat16, device=dev),
        }
        s["ws_gu"] = torch.empty(Q.qvla_linear_workspace_bytes(gu, M), dtype=torch.uint8, device=dev)
        s["ws_dn"] = torch.empty(Q.qvla_linear_workspace_bytes(dn, M), dtype=torch.uint8, device=dev)
        sets.append(s)

    def step(s, ev=None):
        # four launches, the two halves of qvla_w4a4_linear for each layer: rotate+quantise x,
        # gated gate/up GEMM, rotate+quantise h, down GEMM; ev[i] is recorded on the launching
        # stream before launch i (ev[4] after the last)
        if ev is not None:
            ev[0].record(stream)
        Q.qvla_linear_quantize(s["gu"], s["x"], M, -1, s["ws_gu"], s["ws_gu"].numel(), stream)
        if ev is not None:
            ev[1].record(stream)
        Q.qvla_linear_gemm(s["gu"], s["ws_gu"], s["ws_gu"].numel(), M, s["h"], stream)
        if ev is not None:
            ev[2].record(stream)
        Q.qvla_linear_quantize(s["dn"], s["h"], M, -1, s["ws_dn"], s["ws_dn"].numel(), stream)
        if ev is not None:
            ev[3].record(stream)
        Q.qvla_linear_gemm(s["dn"], s["ws_dn"], s["ws_dn"].numel(), M, s["y"], stream)
        if ev is not None:
            ev[4].record(stream)

    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    w0.record(stream)
    for i in range(args.warmup):
        step(sets[i % args.sets])
    w1.record(stream)
    torch.cuda.synchronize()
    Q.qvla_check_device(stream)
    warm_ms = w0.elapsed_time(w1) / max(1, args.warmup)

    # ---- device-timed region: inputs resident in HBM ----
    K = args.steps
    # per-kernel events on every EVERY-th step only: between events the kernels of the other
    # steps keep overlapping their launch with the previous kernel's tail
    EVERY = 8
    evs = {i: [torch.cuda.Event(enable_timing=True) for _ in range(5)] for i in range(0, K, EVERY)}
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    # Untimed steps before and after the timed region (about 0.3 s each) keep the GPU under the
    # same load while the clock sampler runs, so that a short timed region still has a clock
    # record around it; samples taken inside the region are reported when there are enough.
    roll = int(min(20000, max(1, 300.0 / max(warm_ms, 1e-3))))
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start((t0, t1))
    for i in range(roll):
        step(sets[i % args.sets])
    t0.record(stream)
    for i in range(K):
        step(sets[i % args.sets], evs.get(i))
    t1.record(stream)
    for i in range(roll):
        step(sets[i % args.sets])
    torch.cuda.synchronize()
    barrier(world)
    clk = clocks.stop()
    Q.qvla_check_device(stream)
    ms = max_over_ranks(world, t0.elapsed_time(t1), dev)
    ne = len(evs)
    rqx_ms = sum(e[0].elapsed_time(e[1]) for e in evs.values()) / ne
    gemm_gu_ms = sum(e[1].elapsed_time(e[2]) for e in evs.values()) / ne
    rqh_ms = sum(e[2].elapsed_time(e[3]) for e in evs.values()) / ne
    gemm_dn_ms = sum(e[3].elapsed_time(e[4]) for e in evs.values()) / ne
    value = job_value(world, OPS_STEP, K, ms)

    # ---- end to end through the public API with host buffers ----
    # Each step copies its input from pinned host memory, runs both linears through
    # qvla_w4a4_linear and reads its output back to pinned host memory.  The copies run on their
    # own streams so that step i + 1's input upload and step i - 1's read-back overlap step i's
    # kernels (the rotating sets keep the buffers of steps in flight apart): the pipelining a
    # serving loop does.  The timed region spans the first upload to the last read-back.
    x_host = mlp.x.pin_memory()
    y_host = torch.empty(M, K_IN, dtype=torch.bfloat16).pin_memory()
    K2 = max(1, min(K, 2000))
    h2d, d2h = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    nset = args.sets
    in_ready = [torch.cuda.Event() for _ in range(K2)]
    x_free = [torch.cuda.Event() for _ in range(K2)]   # the set's input has been read
    y_ready = [torch.cuda.Event() for _ in range(K2)]
    y_free = [torch.cuda.Event() for _ in range(K2)]   # the set's output has been read back
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(h2d)
    for i in range(K2):
        s = sets[i % nset]
        with torch.cuda.stream(h2d):
            if i >= nset:
                h2d.wait_event(x_free[i - nset])
            s["x"].copy_(x_host, non_blocking=True)
            in_ready[i].record(h2d)
        stream.wait_event(in_ready[i])
        if i >= nset:
            stream.wait_event(y_free[i - nset])
        Q.qvla_w4a4_linear(s["gu"], s["x"], M, -1, s["h"], s["ws_gu"], s["ws_gu"].numel(), stream)
        x_free[i].record(stream)
        Q.qvla_w4a4_linear(s["dn"], s["h"], M, -1, s["y"], s["ws_dn"], s["ws_dn"].numel(), stream)
        y_ready[i].record(stream)
        with torch.cuda.stream(d2h):
            d2h.wait_event(y_ready[i])
            y_host.copy_(s["y"], non_blocking=True)
            y_free[i].record(d2h)
    e1.record(d2h)
    torch.cuda.synchronize()
    barrier(world)
    Q.qvla_check_device(stream)
    ms2 = max_over_ranks(world, e0.elapsed_time(e1), dev)
    e2e = job_value(world, OPS_STEP, K2, ms2)

    pk = peaks()
    extra = {}
    if not args.no_stacks:
        extra.update(run_stacks(dev, stream, pk))
    if not args.no_sweep:
        extra["single_layer"] = run_single_layer(dev, stream, pk)
        extra["sweep"] = run_sweep(dev, stream, pk, oracle_point=(rank == 0 and world == 1))
    achieved = (OPS_GATEUP + OPS_DOWN) / ((gemm_gu_ms + gemm_dn_ms) * 1e-3) / 1e12
    cpu = cpu_baseline(mlp, packed, args.cpu_seconds) if (rank == 0 and world == 1) else None
    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "TOPS", "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": round(ms / K, 5), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int4", "data": "synthetic",
            "config": {"workload": WORKLOAD, "tokens": M, "hidden": K_IN, "mlp_hidden": HIDDEN,
                       "l2": f"{args.sets} rotating weight+activation sets (~{args.sets * 117} MB) > 129 MB L2",
                       "parallelism": f"replica per GPU x{world}"},
            "roofline": {"bound": "tensor", "achieved": round(achieved, 1), "peak": round(pk["tflops"], 1),
                         "unit": "TFLOP/s", "frac": round(achieved / pk["tflops"], 4), "traffic": gemm_traffic(),
                         "kernel": "gemm_w4a4 (gate/up + down launches)",
                         "peak_note": f"{pk['src']} burst bf16 x {FP8_OVER_BF16:g} (nominal E4M3/bf16 ratio); each "
                                      "GEMM launch is timed alone by its own events",
                         "peak_sustained": round(pk["tflops_sustained"], 1),
                         "frac_of_sustained": round(achieved / pk["tflops_sustained"], 4)},
            "kernels_us_note": f"CUDA events around each launch on every {EVERY}th timed step",
            "kernels_us": {"rotate_quantize_x": round(rqx_ms * 1e3, 2), "gemm_gate_up": round(gemm_gu_ms * 1e3, 2),
                           "rotate_quantize_h": round(rqh_ms * 1e3, 2), "gemm_down": round(gemm_dn_ms * 1e3, 2)},
            "e2e": {"value": round(e2e, 2), "unit": "TOPS", "h2d_bytes_per_step": M * K_IN * 2,
                    "d2h_bytes_per_step": M * K_IN * 2, "steps": K2,
                    "note": "qvla_w4a4_linear with pinned host input and output copies every step, the copies "
                            "on their own streams overlapping the neighbouring steps' kernels"},
            "gpu_launches": 4 * K,
            "clocks": clk,
            "cpu_baseline": cpu,
        }
        line.update(extra)
        print(json.dumps(line), flush=True)
    for s in sets:
        s["gu"].close()
        s["dn"].close()


# --------------------------------------------------------------------------------------
# the layer stacks
# --------------------------------------------------------------------------------------

DIT_SEED, DIT_M, DIT_T, DIT_CAL_ROWS = 2, 50, 10, 16


def _algorithmic_bytes(weights, m, xb=2, yb=2):
    """Bytes a fused linear must move: activations in, packed weights, scales and bias, outputs."""
    return sum(xb * m * w.k + w.packed.nbytes + 8 * w.packed.shape[0] + yb * m * w.n for w in weights)


def _time_replays(fn, reps, flush=None, stream=None):
    """Mean milliseconds of fn() over reps runs, each bracketed by CUDA events on the launching
    stream; flush() (outside the events) runs first when given."""
    evs = []
    for _ in range(reps):
        if flush is not None:
            flush()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        evs.append((a, b))
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in evs) / reps


def _dit_stack(S, Q, W, weights, peaks, act_bits, dev, stream, flush, peak_gbs, peak_src, profile=False):
    """One DiT stack (18 blocks, M = 50, T = 10) with int4 or 8-bit activation codes: per-step
    microseconds with L2 flushed, per rollout, and back to back.  peaks[layer] is [T] (one scale
    per step) or [T, G] (per-group scales)."""
    qmax = np.float32(7 if act_bits == 4 else 127)
    st = S.LinearStack(weights, DIT_M, "f16", "f16", dev, input_sets=DIT_T, act_bits=act_bits)
    for i, w in enumerate(weights):
        for t in range(DIT_T):
            st.set_input(i, torch.from_numpy(W.dit_layer_input(DIT_SEED, i, t, DIT_M, w.k, DIT_T, profile)), t)
    st.set_step_tables([p / qmax for p in peaks])
    graphs = [st.capture(t) for t in range(DIT_T)]
    for _ in range(3):
        for g in graphs:
            g.replay()
    torch.cuda.synchronize()
    Q.qvla_check_device(stream)
    reps = 20
    step_ms = sum(_time_replays(g.replay, reps, flush, stream) for g in graphs) / DIT_T
    roll_ms = _time_replays(lambda: [g.replay() for g in graphs], reps, flush, stream)
    warm_ms = _time_replays(lambda: [g.replay() for g in graphs], reps, None, stream) / DIT_T
    Q.qvla_check_device(stream)
    dit_bytes = _algorithmic_bytes(weights, DIT_M)
    dit_gbs = dit_bytes / (step_ms * 1e-3) / 1e9
    out = {
        "us_per_step": round(step_ms * 1e3, 2), "us_per_rollout": round(roll_ms * 1e3, 2),
        "us_per_step_warm": round(warm_ms * 1e3, 2), "steps": DIT_T, "tokens": DIT_M,
        "linears_per_step": len(weights), "gpu_launches_per_step": 2 * len(weights),
        "weight_bytes": st.weight_bytes, "ops_per_step": st.ops,
        "roofline": {"bound": "hbm", "achieved": round(dit_gbs, 1), "peak": round(peak_gbs, 1), "unit": "GB/s",
                     "frac": round(dit_gbs / peak_gbs, 4), "bytes_per_step": dit_bytes,
                     "peak_note": f"{peak_src} HBM copy bandwidth"},
        "timing": "CUDA-graph replay per step, L2 flushed (256 MB write) before each timed step or rollout; "
                  "'warm' = 10 steps back to back without a flush",
    }
    st.close()
    del graphs, st
    torch.cuda.empty_cache()
    return out


def _w4a8_gate_up(Q, W, dev, stream, flush, peak_tflops):
    """The backbone's gate/up projection (816 x 2048 -> 2 x 16384, GELU-gated) with 8-bit
    activation codes: rotate + quantise and the GEMM, TOPS of the integer product.  The tensor
    cores run two E4M3 passes per product (high and low nibble planes), so the E4M3 rate the
    hardware sustains is twice the reported TOPS."""
    rng = np.random.default_rng(7)
    codes = rng.integers(-7, 8, (2 * HIDDEN, K_IN)).astype(np.int8)
    packed = W.pack_nibbles(codes)
    ws = np.full(2 * HIDDEN, 2 ** -9, np.float32)
    layer = Q.qvla_layer_create_gated(HIDDEN, K_IN, HAD_IN, Q.BF16, Q.BF16, packed[:HIDDEN], ws[:HIDDEN],
                                      packed[HIDDEN:], ws[HIDDEN:])
    x = torch.from_numpy(rng.standard_normal((M, K_IN), dtype=np.float32)).to(dev, torch.bfloat16)
    h = torch.empty(M, HIDDEN, dtype=torch.bfloat16, device=dev)
    nb = Q.qvla_w4a8_workspace_bytes(layer, M)
    work = torch.empty(nb, dtype=torch.uint8, device=dev)

    def run():
        Q.qvla_w4a8_linear(layer, x, M, -1, h, work, nb, stream)

    for _ in range(3):
        run()
    torch.cuda.synchronize()
    Q.qvla_check_device(stream)
    ms = _time_replays(run, 20, flush, stream)
    Q.qvla_check_device(stream)
    layer.close()
    tops = OPS_GATEUP / (ms * 1e-3) / 1e12
    return {"us": round(ms * 1e3, 1), "tops": round(tops, 1), "e4m3_tflops_issued": round(2 * tops, 1),
            "frac_of_e4m3_peak": round(2 * tops / peak_tflops, 4),
            "timing": "rotate+quantise (8-bit codes) and GEMM launches, L2 flushed before each of 20 runs"}


def run_stacks(dev, stream, pk):
    from paper_2605_28803_gb300 import qvla as Q
    from paper_2605_28803_gb300 import stack as S
    from paper_2605_28803_gb300 import workloads as W

    scratch = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # 256 MB > 129 MB L2

    def flush():
        scratch.zero_()

    # ---- DiT action head: per-step tables calibrated with the library's rotated-absmax pass ----
    weights = W.dit_stack(DIT_SEED)
    peak = torch.zeros(1, dtype=torch.float32, device=dev)
    peaks = []  # [layer][step] rotated absmax of the calibration draw
    for i, w in enumerate(weights):
        row = []
        for t in range(DIT_T):
            xc = torch.from_numpy(W.dit_layer_input(DIT_SEED + 1000, i, t, DIT_CAL_ROWS, w.k, DIT_T)).to(dev, torch.float16)
            peak.zero_()
            Q.qvla_rotated_absmax(xc, Q.F16, DIT_CAL_ROWS, w.k, w.had_block, peak, stream)
            row.append(np.float32(peak.item()))
        peaks.append(np.asarray(row, dtype=np.float32))
    dit = _dit_stack(S, Q, W, weights, peaks, 4, dev, stream, flush, pk["gbs"], pk["src"])
    dit["w4a8"] = _dit_stack(S, Q, W, weights, peaks, 8, dev, stream, flush, pk["gbs"], pk["src"])
    # the paper's rotation configuration: Hadamard blocks of 64, per-step tables per 128-channel
    # group, inputs with uneven channel magnitudes
    wb = W.dit_stack_blocks(weights, 64)
    gpeaks = []
    for i, w in enumerate(wb):
        row = []
        for t in range(DIT_T):
            xc = torch.from_numpy(W.dit_layer_input(DIT_SEED + 1000, i, t, DIT_CAL_ROWS, w.k, DIT_T, True)).to(
                dev, torch.float16)
            gp = torch.zeros(w.k // 128, dtype=torch.float32, device=dev)
            Q.qvla_rotated_absmax_groups(xc, Q.F16, DIT_CAL_ROWS, w.k, w.had_block, gp, stream)
            row.append(gp.cpu().numpy())
        gpeaks.append(np.asarray(row, dtype=np.float32))
    dit["grouped"] = _dit_stack(S, Q, W, wb, gpeaks, 4, dev, stream, flush, pk["gbs"], pk["src"], profile=True)
    dit["tables"] = ("per-step, per-layer, calibrated with qvla_rotated_absmax on a separate 16-token draw "
                     "(absmax / 7; absmax / 127 for the W4A8 variant); 'grouped': Hadamard blocks of 64 and "
                     "per-step tables per 128-channel group (qvla_rotated_absmax_groups)")
    w4a8_gu = _w4a8_gate_up(Q, W, dev, stream, flush, pk["tflops"])

    # ---- backbone forward at M = 816 and M = 1 (per-token scales) ----
    weights = W.backbone_stack(seed=3)
    bb = {"layers": 18, "linears": len(weights), "weight_bytes": int(sum(w.packed.nbytes for w in weights))}
    for m in (816, 1):
        st = S.LinearStack(weights, m, "bf16", "bf16", dev)
        for i, w in enumerate(weights):
            st.set_input(i, torch.from_numpy(W.backbone_layer_input(3, i, m, w.k)))
        g = st.capture(-1)
        g.replay()
        torch.cuda.synchronize()
        Q.qvla_check_device(stream)
        ms = _time_replays(g.replay, 10, flush, stream)
        Q.qvla_check_device(stream)
        if m > 1:
            tops = st.ops / (ms * 1e-3) / 1e12
            bb["m816"] = {"us_per_forward": round(ms * 1e3, 1), "tops": round(tops, 1),
                          "roofline": {"bound": "tensor", "achieved": round(tops, 1), "peak": round(pk["tflops"], 1),
                                       "unit": "TFLOP/s", "frac": round(tops / pk["tflops"], 4)}}
        else:
            nbytes = _algorithmic_bytes(weights, m)
            gbs = nbytes / (ms * 1e-3) / 1e9
            bb["m1"] = {"us_per_forward": round(ms * 1e3, 1),
                        "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": round(pk["gbs"], 1),
                                     "unit": "GB/s", "frac": round(gbs / pk["gbs"], 4), "bytes": nbytes}}
        st.close()
        del g, st
        torch.cuda.empty_cache()
    bb["timing"] = ("CUDA-graph replay of one forward, L2 flushed before each; M = 816: the rotate-quantise "
                    "kernel and the GEMM per linear; M = 1: one kernel per linear (the decode GEMV that "
                    "rotates and quantises its token itself)")
    del scratch
    torch.cuda.empty_cache()
    return {"dit": dit, "backbone": bb, "w4a8_gate_up": w4a8_gu}


# --------------------------------------------------------------------------------------
# config 1 (one per-step layer) and the config-5 sweep of single linears
# --------------------------------------------------------------------------------------

def _linear_bytes(m, k, n, xb=2, yb=2):
    """Algorithmic bytes of one fused linear: activations in, packed int4 weights, the weight
    scales, outputs."""
    return xb * m * k + n * k // 2 + 4 * n + yb * m * n


def _roofline_point(ops, nbytes, sec, pk):
    """Whichever roofline bounds a linear of this arithmetic intensity, and the fraction of it
    reached: HBM left of the ridge (peak tensor rate / HBM bandwidth), the tensor rate right."""
    ridge = pk["tflops"] * 1e12 / (pk["gbs"] * 1e9)
    if ops / nbytes < ridge:
        ach = nbytes / sec / 1e9
        return {"bound": "hbm", "achieved": round(ach, 1), "unit": "GB/s", "frac": round(ach / pk["gbs"], 4)}
    ach = ops / sec / 1e12
    return {"bound": "tensor", "achieved": round(ach, 1), "unit": "TFLOP/s", "frac": round(ach / pk["tflops"], 4)}


def run_single_layer(dev, stream, pk):
    """The 64 x 512 x 512 per-step layer (random orthogonal SVD stand-in folded into the weights,
    Hadamard 512, a T = 10 step table from each step's rotated absmax): one qvla_w4a4_linear
    timed cold (L2 flushed before each call) and as one CUDA graph of the 10 steps replayed back
    to back."""
    from paper_2605_28803_gb300 import qvla as Q
    from paper_2605_28803_gb300 import workloads as W

    case = W.single_layer_steps(seed=0)
    n, k = case.w.shape
    m, steps = case.x_steps[0].shape[0], len(case.x_steps)
    wq, ws = np.zeros((n, k // 2), np.uint8), np.zeros(n, np.float32)
    Q.qvla_pack_weights_host(np.ascontiguousarray(case.w), Q.F32, n, k, rot=np.ascontiguousarray(case.rot),
                             rot_block=case.rot_block, had_block=case.had_block, wq=wq, wscale=ws)
    layer = Q.qvla_layer_create(n, k, case.had_block, Q.F16, Q.F16, wq, ws, None)
    xs = [x.to(dev) for x in case.x_steps]
    peak = torch.zeros(1, dtype=torch.float32, device=dev)
    table = []
    for t in range(steps):
        peak.zero_()
        Q.qvla_rotated_absmax(xs[t], Q.F16, m, k, case.had_block, peak, stream)
        table.append(np.float32(peak.item()) / np.float32(7))
    Q.qvla_set_step_scales(layer, np.asarray(table, np.float32))
    y = torch.empty(m, n, dtype=torch.float16, device=dev)
    nb = Q.qvla_linear_workspace_bytes(layer, m)
    work = torch.empty(nb, dtype=torch.uint8, device=dev)
    scratch = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def one(t):
        Q.qvla_w4a4_linear(layer, xs[t], m, t, y, work, nb, stream)

    for t in range(steps):
        one(t)
    torch.cuda.synchronize()
    Q.qvla_check_device(stream)
    reps = 20
    cold_ms = sum(_time_replays(lambda t=t: one(t), reps, scratch.zero_, stream) for t in range(steps)) / steps
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for t in range(steps):
            Q.qvla_w4a4_linear(layer, xs[t], m, t, y, work, nb, torch.cuda.current_stream())
    g.replay()
    torch.cuda.synchronize()
    graph_ms = _time_replays(g.replay, reps, None, stream) / steps
    Q.qvla_check_device(stream)
    layer.close()
    del g, scratch
    torch.cuda.empty_cache()
    nbytes, ops = _linear_bytes(m, k, n), 2 * m * n * k
    return {"shape": f"M={m} K={k} N={n}, f16 in/out, Hadamard {case.had_block}, T={steps} step table",
            "us_cold": round(cold_ms * 1e3, 2), "us_graph": round(graph_ms * 1e3, 2),
            "gbs_cold": round(nbytes / (cold_ms * 1e-3) / 1e9, 1), "gbs_graph": round(nbytes / (graph_ms * 1e-3) / 1e9, 1),
            "tops_graph": round(ops / (graph_ms * 1e-3) / 1e12, 2), "bytes": nbytes, "ops": ops,
            "frac_hbm_graph": round(nbytes / (graph_ms * 1e-3) / 1e9 / pk["gbs"], 4),
            "timing": "qvla_w4a4_linear (2 launches); cold: L2 flushed before each of 20 calls per step; "
                      "graph: the 10 steps captured once, replayed back to back, time / 10"}


SWEEP_M = (1, 16, 50, 256, 816, 3200, 8192)
SWEEP_KN = ((1024, 1024), (1024, 4096), (2048, 2048), (2048, 16384), (16384, 2048))


def run_sweep(dev, stream, pk, oracle_point=True, points_only=None):
    """The single-linear sweep: qvla_w4a4_linear at M in SWEEP_M x (K, N) in SWEEP_KN, f16 in and
    out, per-token scales, Hadamard K (2048 blocks at K = 16384).  Each point: 10 calls of the
    linear, L2 flushed before each, CUDA events around it; then 10 calls of its two halves
    (qvla_linear_quantize, qvla_linear_gemm) with events around each.  The
    weights are uniform random code bytes (the time of a linear does not depend on its values);
    the activations are drawn on the device (N(0,1), 0.5% channels x20)."""
    from paper_2605_28803_gb300 import qvla as Q
    from paper_2605_28803_gb300 import workloads as W

    scratch = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    mmax = max(SWEEP_M)
    points = []
    kn_list = SWEEP_KN if points_only is None else sorted({(k, n) for _, k, n in points_only})
    for kn_i, (k, n) in enumerate(kn_list):
        had = k if k <= 4096 else 2048
        rng = np.random.default_rng(500 + kn_i)
        packed = rng.integers(0, 256, (n, k // 2), dtype=np.uint8)
        ws = (rng.uniform(0.8, 1.2, n) * 0.5 / np.sqrt(k)).astype(np.float32)
        layer = Q.qvla_layer_create(n, k, had, Q.F16, Q.F16, packed, ws, None)
        x = W.sweep_input_device(mmax if points_only is None else max(m for m, _, _ in points_only), k,
                                 seed=600 + kn_i, device=dev, dtype="f16")
        y = torch.empty(x.shape[0], n, dtype=torch.float16, device=dev)
        nb = Q.qvla_linear_workspace_bytes(layer, x.shape[0])
        work = torch.empty(nb, dtype=torch.uint8, device=dev)
        ms = SWEEP_M if points_only is None else sorted({m for m, kk, nn in points_only if (kk, nn) == (k, n)})
        for m in ms:
            xm, ym = x[:m], y[:m]

            def halves(ev=None):
                if ev:
                    ev[0].record(stream)
                Q.qvla_linear_quantize(layer, xm, m, -1, work, nb, stream)
                if ev:
                    ev[1].record(stream)
                Q.qvla_linear_gemm(layer, work, nb, m, ym, stream)
                if ev:
                    ev[2].record(stream)

            def linear(ev=None):
                if ev:
                    ev[0].record(stream)
                Q.qvla_w4a4_linear(layer, xm, m, -1, ym, work, nb, stream)
                if ev:
                    ev[1].record(stream)

            def timed(fn, nev):
                for _ in range(3):
                    fn()
                torch.cuda.synchronize()
                evs = []
                for _ in range(10):
                    scratch.zero_()
                    e = [torch.cuda.Event(enable_timing=True) for _ in range(nev)]
                    fn(e)
                    evs.append(e)
                torch.cuda.synchronize()
                return evs

            # launches of the whole linear: one where the decode GEMV rotates and quantises
            # itself (the workspace then stays untouched), else the two halves
            work.fill_(0xA5)
            linear()
            torch.cuda.synchronize()
            launches = 1 if bool(torch.all(work == 0xA5).item()) else 2
            ev_l = timed(linear, 2)
            ev_h = timed(halves, 3)
            t_all = statistics.median(e[0].elapsed_time(e[1]) for e in ev_l) * 1e-3
            t_rq = statistics.median(e[0].elapsed_time(e[1]) for e in ev_h) * 1e-3
            t_gemm = statistics.median(e[1].elapsed_time(e[2]) for e in ev_h) * 1e-3
            ops, nbytes = 2 * m * n * k, _linear_bytes(m, k, n)
            pt = {"M": m, "K": k, "N": n, "us": round(t_all * 1e6, 2), "launches": launches,
                  "us_rotate_quantize": round(t_rq * 1e6, 2), "us_gemm": round(t_gemm * 1e6, 2),
                  "tops": round(ops / t_all / 1e12, 2), "gbs": round(nbytes / t_all / 1e9, 1)}
            pt["roofline"] = _roofline_point(ops, nbytes, t_all, pk)
            points.append(pt)
        Q.qvla_check_device(stream)
        layer.close()
        del x, y, work
        torch.cuda.empty_cache()
    del scratch
    torch.cuda.empty_cache()
    out = {"points": points,
           "timing": "us: median of 10 calls of qvla_w4a4_linear (launches: 1 where the decode GEMV takes the "
                     "token, else 2), L2 flushed (256 MB write) before each; us_rotate_quantize / us_gemm: the "
                     "two halves called separately, likewise; bytes = 2MK + NK/2 + 4N + 2MN; roofline = HBM left "
                     "of the ridge, burst E4M3 right of it",
           "ridge_ops_per_byte": round(pk["tflops"] * 1e12 / (pk["gbs"] * 1e9), 1)}
    if oracle_point:
        out["oracle_point"] = _oracle_sweep_point()
    return out


def _oracle_sweep_point(m=256, k=2048, n=2048):
    """The oracle's host time for one sweep point (K, N) = (2048, 2048), M = 256: rotate,
    quantise, integer GEMM and dequantise in numpy float64 (the offline weight pack not timed)."""
    from oracle import qvla_oracle as O
    from paper_2605_28803_gb300 import workloads as W

    case = W.sweep_linear(m, k, n, seed=4, xdtype="f16", ydtype="f16")
    _, ws, codes = O.pack_weights(case.w.astype(np.float64), case.had_block)
    x64 = case.x.double().numpy()
    t0 = time.perf_counter()
    O.w4a4_linear(x64, codes, ws, case.had_block, out_fmt="f16")
    el = time.perf_counter() - t0
    return {"M": m, "K": k, "N": n, "seconds": round(el, 3), "tops": round(2 * m * n * k / el / 1e12, 6),
            "cores": cpu_cores(), "kind": "oracle"}


# --------------------------------------------------------------------------------------
# the CPU oracle (baseline leg and --impl reference)
# --------------------------------------------------------------------------------------

def oracle_block(x64, oc):
    from oracle import qvla_oracle as O

    gate = O.w4a4_linear(x64, oc["gate"][0], oc["gate"][1], HAD_IN, out_fmt="bf16")["y"]
    up = O.w4a4_linear(x64, oc["up"][0], oc["up"][1], HAD_IN, out_fmt="bf16")["y"]
    h = O.round_to_format(O.gated_glue(gate, up), "bf16")
    return O.w4a4_linear(h, oc["down"][0], oc["down"][1], HAD_HIDDEN, out_fmt="bf16")["y"]


def oracle_weights(mlp):
    from oracle import qvla_oracle as O

    out = {}
    for name, w, had in (("gate", mlp.w_gate, HAD_IN), ("up", mlp.w_up, HAD_IN), ("down", mlp.w_down, HAD_HIDDEN)):
        _, ws, codes = O.pack_weights(w.astype(np.float64), had)
        out[name] = (codes, ws)
    return out


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def cpu_baseline(mlp, packed, seconds, tokens=16):
    """The oracle as it stands on a bounded sample: 16-token slices of the same block, repeated
    for about `seconds` of host time.  The oracle's offline weight pack is not timed."""
    oc = oracle_weights(mlp)
    x64 = mlp.x.double().numpy()
    done, t0 = 0, time.perf_counter()
    i = 0
    while True:
        rows = slice((i * tokens) % M, (i * tokens) % M + tokens)
        oracle_block(x64[rows], oc)
        done += tokens
        i += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    ops = 2 * done * (K_IN * 2 * HIDDEN + HIDDEN * K_IN)
    return {"value": round(ops / el / 1e12, 6), "unit": "TOPS", "cores": cpu_cores(), "kind": "oracle",
            "sample": f"{done} tokens ({i} slices of {tokens}) of the same block, {el:.1f} s, numpy float64"}


def run_reference(args, budget_s: float = 90.0):
    """The oracle timed on the host, rank 0 only.  Each step is a bounded sample (4 tokens of the
    block); the run times up to --steps steps but stops after about budget_s seconds, and
    reports the number of steps it actually timed."""
    world, rank, _ = dist_init()
    if rank != 0:
        return
    from paper_2605_28803_gb300 import workloads as W

    mlp = W.gated_mlp(seed=1, m=M, k=K_IN, hidden=HIDDEN, had_in=HAD_IN, had_hidden=HAD_HIDDEN)
    oc = oracle_weights(mlp)
    x64 = mlp.x.double().numpy()
    tokens = 4
    # the requested warm-up steps, stopping after about 20 s but never before min(W, 3)
    warm = 0
    w0 = time.perf_counter()
    while warm < args.warmup and (warm < 3 or time.perf_counter() - w0 < 20.0):
        oracle_block(x64[:tokens], oc)
        warm += 1
    t0 = time.perf_counter()
    done = 0
    while done < args.steps:
        r0 = (done * tokens) % M
        oracle_block(x64[r0:r0 + tokens], oc)
        done += 1
        if time.perf_counter() - t0 > budget_s:
            break
    el = time.perf_counter() - t0
    ops = 2 * tokens * done * (K_IN * 2 * HIDDEN + HIDDEN * K_IN)
    value = ops / el / 1e12
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "TOPS", "n_gpus": world,
        "steps": done, "warmup": warm, "ms_per_step": round(el / done * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int4", "data": "synthetic",
        "config": {"workload": WORKLOAD, "tokens": M, "hidden": K_IN, "mlp_hidden": HIDDEN},
        "cpu_baseline": {"value": round(value, 6), "unit": "TOPS", "cores": cpu_cores(), "kind": "oracle",
                         "sample": f"{tokens} tokens of the block per step, {done} steps in {el:.1f} s "
                                   f"(numpy float64 oracle; {args.steps} requested)"},
        "e2e": {"value": round(value, 6), "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_points(args):
    """Only the named sweep points (3 untimed and 10 timed calls each): a short run whose kernel
    launches a profiler can pick out."""
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    pts = [tuple(int(v) for v in p.split(",")) for p in args.sweep_points.split(";") if p.strip()]
    out = run_sweep(dev, torch.cuda.current_stream(), peaks(), oracle_point=False, points_only=pts)
    print(json.dumps({"sweep_points": out["points"]}), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif args.sweep_points:
        run_points(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
