#!/usr/bin/env python
"""Benchmark: circuit evaluations/s of the batched statevector engine on GB300.

One step = one pass of the whole hot path over one batch: the forward sweep to
per-qubit <Z> (saving the final states) plus the adjoint backward to dL/dx and
dL/dw.  The timed workload (``value``) is the 16-qubit / 8-layer / batch-512
complex64 circuit (RY(x) encoding, RX RY RZ per qubit per layer, CX ring): the
largest configuration of the path that fits one GPU.  Sub-records (``configs``)
time every other workload the same way: the 4-, 8- and 12-qubit circuits, the
32 random circuits (forward only) and the 16-qubit circuit in complex128 and in
double-float complex128.  Inputs are seeded and synthetic.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With --gpus N > 1 and no torchrun environment, the script starts itself under
torch.distributed.run with N ranks.  Each rank runs the same per-rank batch
(weak scaling); the shared-weight gradient is summed across ranks with one
all-reduce per step.  Rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
import socket
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "circuit evals/sec (fwd; fwd+adjoint bwd) at 4-16 qubits; % of roofline"
FP32_LANES_PER_SM = 128
SM_MAX_MHZ = 2070.0
# double-float complex128: each component of a 2x2 update (4 products, 3 sums:
# 7 of the 14 algorithmic flops per amplitude) is one compensated dot product
# of 43 FP32 instructions, so 14 flops cost 86 FP32 instructions
DF_FP32_OPS_PER_14_FLOPS = 86.0


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "sm_max_mhz": SM_MAX_MHZ}, "fallback"


def num_sms():
    try:
        import torch
        return torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    except Exception:
        return 152


def fp32_peak_tflops(sm_mhz, sms=None):
    # FP32 CUDA-core peak: SMs x 128 lanes x 2 flop (FFMA) x clock
    return (sms or num_sms()) * FP32_LANES_PER_SM * 2 * sm_mhz * 1e6 / 1e12


def flops_per_eval(info):
    """Algorithmic flops of one evaluation by the counting rule of the hot-path
    scope (per amplitude: 14 per fused single-qubit run, 6 per RZZ, 3 per CRZ,
    0 for permutations; <Z> (3 + n)):
      forward  F = sum_f 2^n + (3 + n) 2^n
      backward   = 2 sum_f 2^n + 4 2^n (parametrised angle slots) + (n + 2) 2^n
    sum_f 2^n is the plan's forward count without the <Z> term."""
    n = info["num_qubits"]
    dim = float(1 << n)
    gates = info["fwd_flops_per_eval"] - (3 + n) * dim
    return info["fwd_flops_per_eval"], 2 * gates + 4 * dim * info["num_terms"] + (n + 2) * dim


def rooflines(parts, dtype, fma, pk, pk_kind):
    """Roofline fractions of the forward and backward calls of a workload, from
    parts = [(plan info, batch, forward seconds, backward seconds or None)] (one
    per circuit; their work and times are summed).  Arithmetic ceiling by state
    type: complex64 FP32 (SMs x 128 lanes x 2 x sm_max_mhz), complex128 the
    measured FP64 FMA rate, double-float the measured FP32 instruction rate x 14
    / 86 (its 2x2 updates' instruction mix).  HBM-tiled calls are also held
    against the copy bandwidth with the state bytes their passes move; the bound
    reported is the ceiling the call comes closest to."""
    if dtype == "c64":
        alu = fp32_peak_tflops(pk.get("sm_max_mhz", SM_MAX_MHZ))
        alu_basis = ("FP32 FFMA: %d SMs x 128 lanes x 2 x %.0f MHz (%s sm_max_mhz)"
                     % (num_sms(), pk.get("sm_max_mhz", SM_MAX_MHZ), pk_kind))
    elif dtype == "c128":
        alu = fma["fp64_tflops"]
        alu_basis = "measured FP64 FMA rate (vqc_fma_peak); GB300's FP64 rate is ~1/75 of FP32"
    else:
        alu = fma["fp32_tflops"] / 2.0 * 14.0 / DF_FP32_OPS_PER_14_FLOPS
        alu_basis = ("double-float: measured FP32 instruction rate (vqc_fma_peak / 2) x 14 flops "
                     "per 86 FP32 instructions of a 2x2 update")
    out = {}
    for idx, name in ((2, "fwd"), (3, "bwd")):
        if any(p[idx] is None for p in parts):
            continue
        secs = sum(p[idx] for p in parts)
        flops = sum(flops_per_eval(p[0])[idx - 2] * p[1] for p in parts)
        r = {"alu": {"achieved": flops / secs / 1e12, "peak": alu, "unit": "TFLOP/s",
                     "flops": flops, "basis": alu_basis}}
        r["alu"]["frac"] = r["alu"]["achieved"] / alu
        if all(p[0][name + "_path"] == 1 for p in parts):
            hbm = pk.get("hbm_gbs", 6800.0)
            nbytes = sum(p[0][name + "_hbm_bytes_per_eval"] * p[1] for p in parts)
            ach = nbytes / secs / 1e9
            r["hbm"] = {"achieved": ach, "peak": hbm, "unit": "GB/s", "bytes": nbytes,
                        "frac": ach / hbm, "basis": "copy bandwidth, %s hbm_gbs" % pk_kind}
        r["bound"] = max(("alu", "hbm") if "hbm" in r else ("alu",), key=lambda k: r[k]["frac"])
        r["frac"] = r[r["bound"]]["frac"]
        r["call_ms"] = secs * 1e3
        out[name] = r
    return out


class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index, self.proc, self.lines = index, None, []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# state type -> (torch real, torch complex, numpy real, arithmetic label, state label)
DTYPES = {"c64": ("float32", "complex64", np.float32, "f32", "complex64"),
          "c128": ("float64", "complex128", np.float64, "f64", "complex128"),
          "c128df": ("float64", "complex128", np.float64, "f32x2 (double-float)", "complex128")}


# ------------------------------------------------------------------ data-parallel step
def dp_shard(cfg, dtype, rank, world, batch=None):
    """This rank's workload: rows [rank B, (rank + 1) B) of a global batch of
    world x B rows (B = the configuration's batch unless given).  Samples are
    independent, so the shards need no exchange in the forward."""
    from paper_2607_11985_gb300 import workloads as wl
    return wl.config(cfg, dtype=dtype, batch=batch, rank=rank, world=world)


def dp_sum(t, world):
    """The data-parallel step's one exchange: the shared-weight gradient dw
    summed over the ranks, in place (a torch tensor on the rank's device)."""
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t)
    return t


# ------------------------------------------------------------------ CPU oracle baseline
def oracle_rate(w_, seconds=10.0, chunk=None, backward=True):
    """Oracle fwd(+bwd) evaluations/s on one host core, on a bounded sample of
    the workload's rows (cycled; at least one chunk)."""
    from oracle import oracle as orc
    if chunk is None:
        chunk = max(1, min(16, int(2e7 / ((1 << w_.spec.n) * max(1, len(w_.spec.gates))))))
    done, t0, row = 0, time.perf_counter(), 0
    while done == 0 or time.perf_counter() - t0 < seconds:
        rows = [(row + i) % w_.batch for i in range(chunk)]
        x = w_.x[rows]
        orc.forward(w_.spec, x, w_.w)
        if backward:
            orc.backward(w_.spec, x, w_.w, w_.gE[rows])
        done += chunk
        row += chunk
    dt = time.perf_counter() - t0
    return done / dt, done, dt


def oracle_rate_parallel(w_, seconds=10.0, workers=None, backward=True):
    """The same oracle on all host cores: one thread per core, each cycling its
    own rows (the oracle runs in C; ctypes releases the GIL during each call)."""
    import concurrent.futures as cf
    from oracle import oracle as orc
    workers = workers or os.cpu_count() or 1
    orc.forward(w_.spec, w_.x[:1], w_.w)    # load the library before the threads start
    t0 = time.perf_counter()

    def work(k):
        done, row = 0, k
        while done == 0 or time.perf_counter() - t0 < seconds:
            rows = [row % w_.batch]
            orc.forward(w_.spec, w_.x[rows], w_.w)
            if backward:
                orc.backward(w_.spec, w_.x[rows], w_.w, w_.gE[rows])
            done += 1
            row += workers
        return done

    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        done = sum(ex.map(work, range(workers)))
    dt = time.perf_counter() - t0
    return done / dt, done, dt, workers


# ------------------------------------------------------------------ our engine
class CircuitBench:
    """One compiled circuit with its device inputs, outputs and workspaces, and
    the calls a step makes through the C ABI (forward with the final state
    saved, backward from it; or the one-call forward+backward)."""

    def __init__(self, torch, w_, stream):
        from paper_2607_11985_gb300 import binding as B
        from paper_2607_11985_gb300.circuit import Circuit
        self.B, self.w_ = B, w_
        t_real, t_cplx = getattr(torch, DTYPES[w_.dtype][0]), getattr(torch, DTYPES[w_.dtype][1])
        self.c = c = Circuit(w_.spec, w_.dtype)
        self.Bt = Bt = w_.batch
        self.info = c.info(Bt)
        self.sp = stream.cuda_stream
        dev = lambda a: torch.tensor(np.asarray(a), dtype=t_real, device="cuda")   # noqa: E731
        self.x = dev(w_.x) if w_.spec.num_x else None
        self.w = dev(w_.w) if w_.spec.num_w else None
        self.gE = dev(w_.gE)
        self.E = torch.empty(Bt, w_.spec.n, dtype=t_real, device="cuda")
        self.st = torch.empty(Bt, 1 << w_.spec.n, dtype=t_cplx, device="cuda")
        self.dx = torch.empty_like(self.x) if self.x is not None else None
        self.dw = torch.empty_like(self.w) if self.w is not None else None
        self.ws = [c.workspace(Bt, m, stream) for m in (0, 1, 3)]

    @staticmethod
    def _p(t):
        return None if t is None else t.data_ptr()

    def fwd(self):
        p, (ws, wsb) = self._p, self.ws[0]
        self.B.vqc_forward(self.c.plan, self.Bt, p(self.x), p(self.w), None, p(self.E), p(self.st),
                           p(ws), wsb, self.sp)

    def bwd(self):
        p, (ws, wsb) = self._p, self.ws[1]
        self.B.vqc_backward(self.c.plan, self.Bt, p(self.x), p(self.w), None, p(self.st), p(self.gE),
                            p(self.dx), p(self.dw), p(ws), wsb, self.sp)

    def step(self):
        self.fwd()
        if self.w_.backward:
            self.bwd()

    def fused(self):
        p, (ws, wsb) = self._p, self.ws[2]
        self.B.vqc_forward_backward(self.c.plan, self.Bt, p(self.x), p(self.w), None, p(self.gE),
                                    p(self.E), p(self.dx), p(self.dw), p(ws), wsb, self.sp)

    def launches(self):
        """Library kernels per step: resident forward 1, resident backward 2
        (sweep + fixed-order dw sum); HBM-tiled: one launch per pass plus the
        per-sample tables (circuits with x; the complex64 backward from a saved
        state evaluates its own) and the partial sums (E; the per-sample
        gradient terms, dx and dw); cluster forward 1, cluster backward 2."""
        inf, nx, nw = self.info, self.w_.spec.num_x > 0, self.w_.spec.num_w > 0
        f = inf["fwd_passes"] + 1 + int(nx) if inf["fwd_path"] == 1 else 1
        if not self.w_.backward:
            return f
        if inf["bwd_path"] == 1:
            b = inf["bwd_passes"] + int(nx or nw) + int(nx) + int(nw) + int(nx and self.w_.dtype != "c64")
        else:
            b = 1 + int(nw)
        return f + b

    def host_step(self, stream_ptr):
        """The end-to-end call on host numpy arrays (vqc_evaluate_host)."""
        w_, rdt = self.w_, DTYPES[self.w_.dtype][2]
        xh = np.ascontiguousarray(w_.x, dtype=rdt) if w_.spec.num_x else None
        wh = np.ascontiguousarray(w_.w, dtype=rdt) if w_.spec.num_w else None
        gh = np.ascontiguousarray(w_.gE, dtype=rdt) if w_.backward else None
        Eh = np.empty((self.Bt, w_.spec.n), rdt)
        dxh = np.empty_like(xh) if (gh is not None and xh is not None) else None
        dwh = np.empty_like(wh) if (gh is not None and wh is not None) else None
        h2d = sum(a.nbytes for a in (xh, wh, gh) if a is not None)
        d2h = sum(a.nbytes for a in (Eh, dxh, dwh) if a is not None)
        step = self.c.prepare_host(xh, wh, gh, out=(Eh, dxh, dwh), stream=stream_ptr)
        return step, h2d, d2h, (Eh, dxh, dwh)


def time_calls(torch, fn, n, flush, stream):
    """Device time (ms) of n calls, one CUDA-event pair per call on the launch
    stream, L2 flushed before each (outside the events)."""
    pairs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
             for _ in range(n)]
    for a, b in pairs:
        flush.zero_()
        a.record(stream)
        fn()
        b.record(stream)
    torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in pairs]


def stats(v):
    return {"median": statistics.median(v), "mean": statistics.mean(v),
            "std": statistics.pstdev(v), "n": len(v)}


def measure_workload(torch, ws_list, steps, warmup, flush, stream, fma, pk, pk_kind,
                     e2e_steps=10, cpu_seconds=0.0, rank=0, world=1):
    """Time one workload (one or more circuits, same dtype) through the C ABI:
    K steps (forward + backward from the saved state; forward only for
    forward-only workloads), each call type on its own, the one-call
    forward+backward, and end to end from host arrays; plus rooflines and the
    oracle on a bounded sample.  Device times are per-rank; rates are whole-job
    (world x per-rank batch)."""
    benches = [CircuitBench(torch, w_, stream) for w_ in ws_list]
    has_bwd = ws_list[0].backward
    for b in benches:
        for _ in range(warmup):
            b.step()
            if has_bwd and world > 1:
                dp_sum(b.dw, world)
    torch.cuda.synchronize()
    evals = sum(b.Bt for b in benches)
    step_ms = [0.0] * steps
    for b in benches:
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps)]
        for i in range(steps):
            flush.zero_()                               # L2 flush, outside the step events
            ev[i][0].record(stream)
            b.step()
            if has_bwd and world > 1:
                dp_sum(b.dw, world)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        for i in range(steps):
            step_ms[i] += ev[i][0].elapsed_time(ev[i][1])
    n_calls = max(5, min(steps, 200))
    fwd_ms = [time_calls(torch, b.fwd, n_calls, flush, stream) for b in benches]
    bwd_ms = [time_calls(torch, b.bwd, n_calls, flush, stream) for b in benches] if has_bwd else None
    fused_ms = [time_calls(torch, b.fused, n_calls, flush, stream) for b in benches] if has_bwd else None
    sum_mean = lambda per: sum(statistics.mean(v) for v in per)   # noqa: E731
    total = torch.tensor([sum(step_ms)], dtype=torch.float64, device="cuda")
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(total, op=dist.ReduceOp.MAX)
    total_ms = float(total.item())
    rec = {
        "circuits": len(benches), "batch_per_gpu": benches[0].Bt,
        "qubits": sorted({w_.spec.n for w_ in ws_list}), "dtype": ws_list[0].dtype,
        "path": {0: "resident", 1: "hbm-tiled", 2: "cluster"}[benches[0].info["fwd_path"]] +
                ("" if not has_bwd or benches[0].info["bwd_path"] == benches[0].info["fwd_path"] else
                 " fwd / %s bwd" % {0: "resident", 1: "hbm-tiled", 2: "cluster"}[benches[0].info["bwd_path"]]),
        "value": world * evals * steps / (total_ms / 1e3),
        "unit": "circuit evals/s (%s)" % ("fwd+adjoint bwd" if has_bwd else "fwd"),
        "ms_per_step": total_ms / steps,
        "fwd": {"value": world * evals / (sum_mean(fwd_ms) / 1e3), "unit": "circuit evals/s (fwd)",
                "ms": sum_mean(fwd_ms)},
        "time_stats_ms": {"step": stats(step_ms), "fwd": stats([sum(t) for t in zip(*fwd_ms)])},
        "gpu_launches": sum(b.launches() for b in benches) * steps,
    }
    if has_bwd:
        rec["bwd"] = {"value": world * evals / (sum_mean(bwd_ms) / 1e3), "ms": sum_mean(bwd_ms)}
        rec["fwd_bwd_two_calls"] = {"value": world * evals / ((sum_mean(fwd_ms) + sum_mean(bwd_ms)) / 1e3),
                                    "unit": "circuit evals/s (fwd+adjoint bwd)",
                                    "basis": "sum of the separately timed forward and backward calls"}
        rec["fused"] = {"value": world * evals / (sum_mean(fused_ms) / 1e3),
                        "unit": "circuit evals/s (fwd+adjoint bwd)", "ms_per_step": sum_mean(fused_ms),
                        "call": "vqc_forward_backward (gE known before the call)"}
        rec["time_stats_ms"]["bwd"] = stats([sum(t) for t in zip(*bwd_ms)])
        rec["time_stats_ms"]["fused"] = stats([sum(t) for t in zip(*fused_ms)])
    if len(benches) > 1:
        rec["concurrent"] = concurrent_steps(torch, benches, steps, flush, stream, world, evals)
    parts = [(b.info, b.Bt, statistics.mean(f) / 1e3,
              statistics.mean(bw) / 1e3 if has_bwd else None)
             for b, f, bw in zip(benches, fwd_ms, bwd_ms if has_bwd else [None] * len(benches))]
    rec["roofline"] = rooflines(parts, ws_list[0].dtype, fma, pk, pk_kind)
    if e2e_steps:
        rec["e2e"] = e2e_rate(torch, benches, e2e_steps, stream, world)
    if cpu_seconds > 0 and rank == 0:
        rec["cpu_baseline"] = cpu_baseline(ws_list, cpu_seconds, has_bwd)
    rec["_benches"] = benches
    return rec


def concurrent_steps(torch, benches, steps, flush, stream, world, evals, nstreams=8):
    """A workload of several independent circuits with their steps issued on
    `nstreams` streams at once (each circuit on its own buffers; fork and join
    through events on the launch stream), so that small launches share the
    GPU: device time per step, L2 flushed before each."""
    streams = [torch.cuda.Stream() for _ in range(nstreams)]
    saved = [b.sp for b in benches]
    ms = []
    try:
        for j, b in enumerate(benches):
            b.sp = streams[j % nstreams].cuda_stream
        for i in range(steps + 2):
            flush.zero_()
            a = torch.cuda.Event(enable_timing=True)
            e = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for st in streams:
                st.wait_event(a)
            for b in benches:
                b.step()
            for st in streams:
                j = torch.cuda.Event()
                j.record(st)
                stream.wait_event(j)
            e.record(stream)
            torch.cuda.synchronize()
            if i >= 2:
                ms.append(a.elapsed_time(e))
    finally:
        for b, sp in zip(benches, saved):
            b.sp = sp
    t = statistics.mean(ms)
    return {"value": world * evals / (t / 1e3), "ms_per_step": t, "streams": nstreams,
            "unit": "circuit evals/s (%s)" % ("fwd+adjoint bwd" if benches[0].w_.backward else "fwd"),
            "basis": "every circuit's step issued on %d streams at once (2 untimed rounds first)" % nstreams}


def e2e_rate(torch, benches, steps, stream, world):
    """End to end through vqc_evaluate_host: host numpy inputs in, outputs out,
    every step (host wall clock, including the Python call)."""
    hs = [b.host_step(stream.cuda_stream) for b in benches]
    for step, *_ in hs:
        step()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        for step, _, _, outs in hs:
            step()
            if world > 1 and outs[2] is not None:     # the data-parallel dw sum of the step
                t = torch.from_numpy(outs[2]).to("cuda")
                dp_sum(t, world)
                outs[2][:] = t.cpu().numpy()
    dt = time.perf_counter() - t0
    t = torch.tensor([dt], dtype=torch.float64, device="cuda")
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    evals = sum(b.Bt for b in benches)
    for _, _, _, outs in hs:
        assert all(np.all(np.isfinite(a)) for a in outs if a is not None)
    from paper_2607_11985_gb300 import binding as B
    direct = B.vqc_host_direct(torch.cuda.current_device())
    return {"value": world * evals * steps / float(t.item()),
            "unit": "circuit evals/s (%s, host buffers)" % ("fwd+adjoint bwd" if benches[0].w_.backward else "fwd"),
            "call": "Circuit.prepare_host -> vqc_evaluate_host (pageable numpy in/out; %s)" % (
                "kernels access the host arrays in place over NVLink-C2C" if direct
                else "one packed copy each way"),
            "h2d_bytes_per_step": sum(h[1] for h in hs), "d2h_bytes_per_step": sum(h[2] for h in hs),
            "steps": steps}


def cpu_baseline(ws_list, seconds, backward):
    """The oracle on one host core, on a bounded sample: rows cycled through the
    workload's circuits (seconds split evenly)."""
    per = seconds / len(ws_list)
    done, dt = 0, 0.0
    for w_ in ws_list:
        _, d, t = oracle_rate(w_, seconds=per, backward=backward)
        done += d
        dt += t
    return {"value": done / dt, "unit": "circuit evals/s (%s)" % ("fwd+adjoint bwd" if backward else "fwd"),
            "cores": 1, "kind": "oracle",
            "sample": "%d rows of the workload (cycled%s), %.1f s" % (
                done, ", over its %d circuits" % len(ws_list) if len(ws_list) > 1 else "", dt)}


SUB_RECORDS = [("cfg1", 1, "c64"), ("cfg2", 2, "c64"), ("cfg3", 3, "c64"), ("cfg4", 4, "c64"),
               ("cfg5_c64", 5, "c64"), ("cfg5_c128", 5, "c128"), ("cfg5_c128df", 5, "c128df")]


def kernel_name(info, dtype, mode):
    rname = {"c64": "float", "c128": "double", "c128df": "dd"}[dtype]
    k, path = info[mode + "_k"], info[mode + "_path"]
    if path == 1:
        return "pass_kernel<%s,K=%d,%s> x %d passes" % (rname, k, mode, info[mode + "_passes"])
    if path == 2:
        return "cluster_fwd_kernel<%s,K=%d>" % (rname, k)
    return "sweep_kernel<%s,K=%d,%s>" % (rname, k, mode)


def traffic_of(workload, mode):
    """DRAM bytes per call from the committed ncu capture of this kernel build
    (profiles/traffic.txt: workload, mode, source digest, bytes), else None."""
    tpath = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(tpath):
        return None
    with open(tpath) as f:
        for line in f:
            parts = line.split()
            if len(parts) >= 4 and not line.startswith("#") and parts[0] == workload \
                    and parts[1] == mode and parts[2] == info_digest():
                return float(parts[3])
    return None


def run_ours(args, rank, world, local_rank):
    import torch
    import __graft_entry__
    from paper_2607_11985_gb300 import binding as B

    __graft_entry__.build()
    torch.cuda.set_device(local_rank)
    stream = torch.cuda.current_stream()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")   # > 129 MB L2
    pk, pk_kind = peaks()
    # measured FMA rates (outside the timed region): packed FP32 for complex64
    # sweeps, FP64 for complex128 ones
    fma = {"fp32_tflops": B.vqc_fma_peak(0), "fp64_tflops": B.vqc_fma_peak(1),
           "kernel": "independent FMA chains over every SM (vqc_fma_peak), best of 5 launches"}
    head = dp_shard(args.config, args.dtype, rank, world)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    sampler = ClockSampler(local_rank)
    if rank == 0:
        sampler.start()
    torch.cuda._sleep(int(50e-3 * SM_MAX_MHZ * 1e6))   # queue work ahead of the GPU
    t_wall = time.perf_counter()
    rec = measure_workload(torch, head, args.steps, args.warmup, flush, stream, fma, pk, pk_kind,
                           e2e_steps=max(10, min(args.steps, 200)),
                           cpu_seconds=0.0 if args.no_cpu_baseline else args.cpu_seconds,
                           rank=rank, world=world)
    t_wall = time.perf_counter() - t_wall
    clocks = sampler.stop() if rank == 0 else None
    benches = rec.pop("_benches")
    info, w0 = benches[0].info, head[0]
    subs = {}
    if not args.no_subrecords:
        for key, cfg, dt in SUB_RECORDS:
            if cfg == args.config and dt == args.dtype:
                continue
            try:
                r = measure_workload(torch, dp_shard(cfg, dt, rank, world), min(args.steps, 10),
                                     min(args.warmup, 3), flush, stream, fma, pk, pk_kind, e2e_steps=5,
                                     cpu_seconds=0.0 if args.no_cpu_baseline else args.sub_cpu_seconds,
                                     rank=rank, world=world)
                bs = r.pop("_benches")
                r["workload"] = bs[0].w_.name.split("_rank")[0] if len(bs) == 1 else \
                    "cfg4_" + "random32_n10-14_B256_c64_fwd"
                del bs
                subs[key] = r
            except Exception as e:   # report, do not hide
                subs[key] = {"error": str(e)[:300]}
            torch.cuda.empty_cache()
    if rank != 0:
        return None
    has_bwd = w0.backward
    dom = "bwd" if has_bwd else "fwd"
    rl = rec["roofline"][dom]
    main = rl[rl["bound"]]
    alt = {k: rl[k] for k in ("alu", "hbm") if k in rl and k != rl["bound"]}
    wname = w0.name.split("_rank")[0]
    out = {
        "metric": METRIC,
        "value": rec["value"],
        "unit": rec["unit"],
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": rec["ms_per_step"],
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": DTYPES[args.dtype][3],   # arithmetic type; the state type is config.state
        "data": "synthetic (seeded; RY(x) encoding + RX/RY/RZ layers + CX ring)",
        "config": {"workload": wname, "qubits": w0.spec.n, "state": DTYPES[args.dtype][4],
                   "batch_per_gpu": w0.batch, "gates": len(w0.spec.gates), "num_x": w0.spec.num_x,
                   "num_w": w0.spec.num_w,
                   "parallelism": "dp%d (batch-sharded replicas, dw all-reduce)" % world,
                   "l2": "flushed between steps (256 MiB write) outside the per-step CUDA events",
                   "step": "vqc_forward (final states saved) + vqc_backward from them",
                   "path": rec["path"], "fwd_k": info["fwd_k"], "bwd_k": info["bwd_k"],
                   "fwd_passes": info["fwd_passes"], "bwd_passes": info["bwd_passes"],
                   "fwd_stages": info["fwd_stages"], "bwd_stages": info["bwd_stages"]},
        "fwd": rec["fwd"],
        "bwd": rec.get("bwd"),
        "fused": rec.get("fused"),
        "concurrent": rec.get("concurrent"),
        "time_stats_ms": rec["time_stats_ms"],
        "roofline": {"kernel": kernel_name(info, args.dtype, dom), "bound": rl["bound"],
                     "achieved": main["achieved"], "peak": main["peak"], "unit": main["unit"],
                     "frac": main["frac"], "traffic": traffic_of(wname, dom),
                     "peak_basis": main["basis"],
                     ("bytes_per_call" if rl["bound"] == "hbm" else "flops_per_call"):
                         main.get("bytes", main.get("flops")),
                     "call_ms": rl["call_ms"],
                     "timing": "mean of per-call CUDA-event times on the launch stream (one call = "
                               "every launch of the %s; L2 flushed before each)" % dom,
                     "other_bound": alt, "fwd": rec["roofline"].get("fwd")},
        "fma_measured": fma,
        "e2e": rec["e2e"],
        "gpu_launches": rec["gpu_launches"],
        "clocks": clocks,
        "wall_s_timed_region": t_wall,
    }
    if "cpu_baseline" in rec:
        out["cpu_baseline"] = rec["cpu_baseline"]
        if not args.no_cpu_baseline:
            prate, pdone, pdt, nw = oracle_rate_parallel(w0, seconds=args.cpu_seconds, backward=has_bwd)
            out["cpu_baseline_all_cores"] = {
                "value": prate, "unit": rec["unit"], "cores": nw,
                "kind": "oracle, batch-parallel threads",
                "sample": "%d rows of the workload (cycled), %.1f s" % (pdone, pdt)}
    if subs:
        for r in subs.values():
            if "roofline" in r:
                d = "bwd" if "bwd" in r["roofline"] else "fwd"
                r["roofline_summary"] = {"kernel_call": d, "bound": r["roofline"][d]["bound"],
                                         "frac": r["roofline"][d]["frac"],
                                         "fwd_frac": r["roofline"]["fwd"]["frac"],
                                         "fwd_bound": r["roofline"]["fwd"]["bound"]}
        out["configs"] = subs
    if not args.no_subrecords:
        flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
        out["f4_tensor_core_stage"] = tc_stage_measurement(torch, flush_buf, torch.cuda.current_stream())
        out["cluster_vs_passes"] = cluster_measurement(torch, flush_buf, torch.cuda.current_stream())
    if args.ablation:
        out["ablation"] = ablation(torch, wl_config(2))
    if args.regime:
        out["regime_map"] = regime_map(torch)
    return out


def tc_stage_measurement(torch, flush, stream, repeats=32, n=16, batch=512):
    """One batch-shared 5-qubit stage (the dense 32 x 32 product of five 2x2
    runs) on the tensor cores (tcgen05, tf32 split three products) and on the
    FP32 units (packed FP32 register blocks), applied `repeats` times to states
    kept on chip: device time per application, algorithmic flops (5 runs x 14
    per amplitude, the FP32 form's count) per second, agreement of the two."""
    from paper_2607_11985_gb300 import binding as B
    rng = np.random.default_rng(1616)
    th = rng.uniform(-np.pi, np.pi, (5, 3))

    def u3(t, p, l):
        c, s = np.cos(t / 2), np.sin(t / 2)
        return np.array([[c, -np.exp(1j * l) * s], [np.exp(1j * p) * s, np.exp(1j * (p + l)) * c]])

    factors = np.stack([u3(*t) for t in th])
    z = torch.randn(batch, 1 << n, dtype=torch.complex64, device="cuda")
    z /= torch.linalg.vector_norm(z, dim=1, keepdim=True)
    outs, res = {}, {}
    sp = stream.cuda_stream
    for method, name in ((0, "fp32_cores"), (1, "tcgen05_tf32x3")):
        out = torch.empty_like(z)
        B.vqc_stage_apply(method, batch, n, factors, z.data_ptr(), out.data_ptr(), repeats, sp)
        ms = time_calls(torch, lambda: B.vqc_stage_apply(method, batch, n, factors, z.data_ptr(),
                                                          out.data_ptr(), repeats, sp), 5, flush, stream)
        B.vqc_sync_check(sp)
        per_app = statistics.median(ms) / repeats
        flops = 5 * 14 * float(batch << n)
        res[name] = {"ms_per_application": per_app, "tflops_algorithmic": flops / (per_app / 1e3) / 1e12}
        outs[name] = out
    res["tc_over_fp32_speedup"] = res["fp32_cores"]["ms_per_application"] / res["tcgen05_tf32x3"]["ms_per_application"]
    res["max_abs_diff_after_%d" % repeats] = float((outs["fp32_cores"] - outs["tcgen05_tf32x3"]).abs().max())
    res["workload"] = "%d-qubit states x %d, %d applications on chip per call" % (n, batch, repeats)
    return res


def cluster_measurement(torch, flush, stream, n_calls=3):
    """The thread-block-cluster path against the HBM-tiled passes on the same
    batch (VQC_FORCE_PATH), complex64: forward (final states saved) and backward
    from them, device time per call; the 16-qubit / 8-layer workload and
    layered 8-layer circuits at 14 and 15 qubits (batch 128)."""
    import os
    from paper_2607_11985_gb300.circuit import Circuit
    from paper_2607_11985_gb300 import workloads as wl
    paths = {0: "resident", 1: "hbm-tiled", 2: "cluster"}
    cases = [("16q_8L_B512 (the timed workload)", wl_config(5).spec, 512)]
    for n in (14, 15):
        cases.append(("%dq_8L_B128" % n, wl.layered(n, 8, ("RX", "RY", "RZ"), "CX"), 128))
    saved = os.environ.get("VQC_FORCE_PATH")
    res = {}
    try:
        for name, spec, B in cases:
            rng = np.random.default_rng(7)
            x = torch.tensor(rng.uniform(-np.pi, np.pi, (B, spec.num_x)), dtype=torch.float32, device="cuda")
            w = torch.tensor(rng.uniform(-np.pi, np.pi, spec.num_w), dtype=torch.float32, device="cuda")
            gE = torch.tensor(rng.standard_normal((B, spec.n)), dtype=torch.float32, device="cuda")
            r = {}
            for force in ("hbm", "cluster"):
                os.environ["VQC_FORCE_PATH"] = force
                c = Circuit(spec, "c64")
                inf = c.info(B)
                E, st = c.forward(x, w, want_state=True)
                dx, dw = c.backward(x, w, gE, psi_final=st)
                f = statistics.median(time_calls(torch, lambda: c.forward(x, w, out=E, state_out=st),
                                                 n_calls, flush, stream))
                b = statistics.median(time_calls(torch, lambda: c.backward(x, w, gE, psi_final=st, grad_x=dx,
                                                                           grad_w=dw), n_calls, flush, stream))
                r[force] = {"fwd_ms": f, "bwd_ms": b, "path_fwd_bwd": [paths[inf["fwd_path"]], paths[inf["bwd_path"]]],
                            "dw": dw.double()}
                del c, E, st
            r["dw_max_abs_diff"] = float((r["hbm"].pop("dw") - r["cluster"].pop("dw")).abs().max())
            r["cluster_over_passes_speedup"] = {k: r["hbm"][k + "_ms"] / r["cluster"][k + "_ms"] for k in ("fwd", "bwd")}
            res[name] = r
    finally:
        if saved is None:
            os.environ.pop("VQC_FORCE_PATH", None)
        else:
            os.environ["VQC_FORCE_PATH"] = saved
    return res


def wl_config(k, **kw):
    from paper_2607_11985_gb300 import workloads as wl
    return wl.config(k, **kw)[0]


_DIGEST = None


def info_digest():
    global _DIGEST
    if _DIGEST is None:
        from paper_2607_11985_gb300 import build
        _DIGEST = build._sources_digest()[:16]
    return _DIGEST


def ablation(torch, w_):
    """Internal ablation on this engine (the paper's Table 5 design choices),
    8-qubit workload: compile once vs compile per call; one batched launch vs a
    loop over samples; adjoint gradients vs central finite differences (the
    same forward kernel, 2 calls per parameter).  Device and host time."""
    from paper_2607_11985_gb300.circuit import Circuit
    real = torch.float32
    x = torch.tensor(w_.x, dtype=real, device="cuda")
    w = torch.tensor(w_.w, dtype=real, device="cuda")
    gE = torch.tensor(w_.gE, dtype=real, device="cuda")
    Bt = w_.batch

    def wall(fn, reps):
        fn()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(reps):
            fn()
        torch.cuda.synchronize()
        return (time.perf_counter() - t0) / reps

    c = Circuit(w_.spec, "c64")
    E = c.forward(x, w)
    out = {"workload": w_.name, "batch": Bt}
    t_once = wall(lambda: c.forward(x, w, out=E), 50)
    t_recompile = wall(lambda: Circuit(w_.spec, "c64").forward(x, w, out=E), 20)
    out["compile_once_fwd_s"] = t_once
    out["compile_per_call_fwd_s"] = t_recompile
    out["compile_per_call_slowdown"] = t_recompile / t_once
    rows = min(Bt, 128)
    xs = [x[i:i + 1] for i in range(rows)]
    t_loop = wall(lambda: [c.forward(xi, w) for xi in xs], 3) * Bt / rows
    out["batched_fwd_s"] = t_once
    out["per_sample_loop_fwd_s"] = t_loop
    out["per_sample_loop_slowdown"] = t_loop / t_once
    st = c.forward(x, w, want_state=True)[1]
    t_adj = wall(lambda: c.backward(x, w, gE, psi_final=st), 20)
    h = 1e-2   # central differences in fp32 arithmetic: h balances truncation and rounding

    def fd():
        gx = torch.empty_like(x)
        gw = torch.empty_like(w)
        for j in range(x.shape[1]):
            xp, xm = x.clone(), x.clone()
            xp[:, j] += h
            xm[:, j] -= h
            gx[:, j] = ((c.forward(xp, w) - c.forward(xm, w)) * gE).sum(1) / (2 * h)
        for j in range(w.shape[0]):
            wp, wm = w.clone(), w.clone()
            wp[j] += h
            wm[j] -= h
            gw[j] = ((c.forward(x, wp) - c.forward(x, wm)) * gE).sum() / (2 * h)
        return gx, gw

    t_fd = wall(fd, 3)
    gx_fd, gw_fd = fd()
    dx, dw = c.backward(x, w, gE, psi_final=st)
    torch.cuda.synchronize()
    out["adjoint_bwd_s"] = t_adj
    out["central_fd_grad_s"] = t_fd
    out["central_fd_slowdown"] = t_fd / t_adj
    out["fd_minus_adjoint_max_abs"] = {"dx": float((gx_fd - dx).abs().max()),
                                       "dw": float((gw_fd - dw).abs().max())}
    return out


def regime_map(torch, qubits=(4, 8, 12, 15, 16, 18, 20), batches=(1, 8, 32, 128), layers=4):
    """Qubits x batch sweep (the paper's regime map, Sec. 4.4): RY(x) encoding,
    `layers` x (RX RY RZ per qubit + CX ring), complex64.  Per point: path, passes,
    device workspace bytes of the backward (the memory the caller must provide
    beyond inputs and outputs), forward and fwd+bwd device time (L2 flushed)."""
    from paper_2607_11985_gb300 import binding as Bd
    from paper_2607_11985_gb300.circuit import Circuit
    from paper_2607_11985_gb300 import workloads as wl
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    pts = []
    for n in qubits:
        spec = wl.layered(n, layers, ("RX", "RY", "RZ"), "CX")
        c = Circuit(spec, "c64")
        rng = np.random.default_rng(7000 + n)
        for Bt in batches:
            x = torch.tensor(rng.uniform(-np.pi, np.pi, (Bt, n)), dtype=torch.float32, device="cuda")
            w = torch.tensor(rng.uniform(-np.pi, np.pi, spec.num_w), dtype=torch.float32, device="cuda")
            gE = torch.tensor(rng.standard_normal((Bt, n)), dtype=torch.float32, device="cuda")
            inf = c.info(Bt)
            E, st = c.forward(x, w, want_state=True)
            c.backward(x, w, gE, psi_final=st)
            torch.cuda.synchronize()
            reps = 5 if n <= 16 else 2
            tf = tb = 0.0
            for _ in range(reps):
                flush.zero_()
                a, b2, d = (torch.cuda.Event(enable_timing=True) for _ in range(3))
                a.record()
                c.forward(x, w, out=E, state_out=st)
                b2.record()
                c.backward(x, w, gE, psi_final=st)
                d.record()
                torch.cuda.synchronize()
                tf += a.elapsed_time(b2) / reps
                tb += b2.elapsed_time(d) / reps
            paths = {0: "resident", 1: "hbm-tiled", 2: "cluster"}
            pts.append({"qubits": n, "batch": Bt,
                        "path": paths[inf["fwd_path"]] if inf["fwd_path"] == inf["bwd_path"] else
                        "%s fwd / %s bwd" % (paths[inf["fwd_path"]], paths[inf["bwd_path"]]),
                        "passes_fwd_bwd": [inf["fwd_passes"], inf["bwd_passes"]],
                        "state_bytes": Bt * (8 << n),
                        "bwd_workspace_bytes": int(Bd.vqc_workspace_bytes(c.plan, Bt, 1)),
                        "fwd_ms": tf, "fwd_bwd_ms": tf + tb,
                        "fwd_bwd_evals_per_s": Bt / ((tf + tb) / 1e3)})
            del x, w, gE, E, st
        del c
        torch.cuda.empty_cache()
    return pts


# ------------------------------------------------------------------ reference arm
def run_reference(args, rank, world):
    """The oracle on the host cores, same metric and workload (bounded sample:
    each step evaluates a few rows, sized so the run ends within minutes)."""
    if rank != 0:
        return None
    w_ = dp_shard(args.config, args.dtype, 0, 1)[0]
    backward = w_.backward
    chunk = max(1, min(8, int(2e7 / ((1 << w_.spec.n) * max(1, len(w_.spec.gates))))))
    from oracle import oracle as orc
    orc.build()
    for _ in range(args.warmup):
        orc.forward(w_.spec, w_.x[:1], w_.w)
    times, row = [], 0
    for _ in range(args.steps):
        rows = [(row + i) % w_.batch for i in range(chunk)]
        t0 = time.perf_counter()
        orc.forward(w_.spec, w_.x[rows], w_.w)
        if backward:
            orc.backward(w_.spec, w_.x[rows], w_.w, w_.gE[rows])
        times.append(time.perf_counter() - t0)
        row += chunk
    total = sum(times)
    value = chunk * args.steps / total
    unit = "circuit evals/s (%s)" % ("fwd+adjoint bwd" if backward else "fwd")
    return {"metric": METRIC, "value": value, "unit": unit,
            "impl": "reference", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": total / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)", "config": {"workload": w_.name, "qubits": w_.spec.n,
                                                    "batch_per_step": chunk},
            "cpu_baseline": {"value": value, "unit": unit, "cores": 1, "kind": "oracle",
                             "sample": "%d steps x %d rows of the workload" % (args.steps, chunk)},
            "e2e": {"value": value, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def one_call(args):
    """One forward with the final states saved and one backward of the selected
    workload (launch order: the forward's passes, then the backward's)."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)
    for w_ in dp_shard(args.config, args.dtype, 0, 1):
        b = CircuitBench(torch, w_, torch.cuda.current_stream())
        b.step()
        torch.cuda.synchronize()
        print("one call: %s, E sum %.6g" % (w_.name, float(b.E.double().abs().sum())))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=5, help="timed workload (1..5; default 5, 16 qubits)")
    ap.add_argument("--dtype", default="c64", choices=sorted(DTYPES),
                    help="state type of the timed workload (c128df: complex128 in double-float)")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--sub-cpu-seconds", type=float, default=2.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-subrecords", action="store_true",
                    help="time only the selected workload (no per-configuration sub-records)")
    ap.add_argument("--regime", action="store_true",
                    help="qubits x batch sweep to 20 qubits (HBM-tiled beyond one SM's state)")
    ap.add_argument("--ablation", action="store_true",
                    help="compile-once / batching / adjoint-vs-FD ablation on the 8-qubit workload")
    ap.add_argument("--stage-once", action="store_true",
                    help="no timing: the batch-shared 5-qubit stage once on the FP32 units and once on "
                         "the tensor cores (16-qubit states x 512, 8 applications), for a profiler")
    ap.add_argument("--one-call", action="store_true",
                    help="no timing: one forward (final states saved) and one backward of the selected "
                         "workload, for a profiler to capture")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if "WORLD_SIZE" not in os.environ and args.gpus > 1:
        # N ranks, one per GPU: start this script under torch.distributed.run
        cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
               "--nproc-per-node", str(args.gpus), "--master-addr", "127.0.0.1",
               "--master-port", str(_free_port()), os.path.abspath(__file__)] + sys.argv[1:]
        sys.exit(subprocess.call(cmd))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world != args.gpus:
        ap.error("--gpus %d but the launcher started %d ranks" % (args.gpus, world))
    if args.one_call:
        one_call(args)
        return
    if args.stage_once:
        import torch
        torch.cuda.set_device(0)
        import __graft_entry__
        __graft_entry__.build()
        r = tc_stage_measurement(torch, torch.empty(256 << 20, dtype=torch.uint8, device="cuda"),
                                 torch.cuda.current_stream(), repeats=8)
        print(json.dumps(r))
        return
    if args.impl == "reference":
        out = run_reference(args, rank, world)
        if out is not None:
            print(json.dumps(out))
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    out = run_ours(args, rank, world, local_rank)
    if out is not None:
        print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
