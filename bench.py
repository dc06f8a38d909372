#!/usr/bin/env python
"""Benchmark: circuit evaluations/s of the batched statevector engine on GB300.

One step = one pass of the whole hot path over one batch: forward sweep to
per-qubit <Z> (saving the final state) plus the adjoint backward to dL/dx and
dL/dw, for the 8-qubit / 4-layer / batch-1024 complex64 workload (RY(x)
encoding, RX RY RZ per qubit per layer, CZ ring).  Inputs are seeded and
synthetic.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun (N > 1) every rank runs the same per-rank batch (weak scaling);
the shared-weight gradient is summed across ranks with one all-reduce per step.
Rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
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
NUM_SMS = 152
SM_MAX_MHZ = 2070.0


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "sm_max_mhz": SM_MAX_MHZ}, "fallback"


def fp32_peak_tflops(sm_mhz):
    # FP32 CUDA-core peak: SMs x 128 lanes x 2 flop (FFMA) x clock
    return NUM_SMS * FP32_LANES_PER_SM * 2 * sm_mhz * 1e6 / 1e12


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


def workload(cfg=2, rank=0, world=1, dtype="c64"):
    """This rank's shard of the global batch (world x per-rank batch rows)."""
    from paper_2607_11985_gb300 import workloads as wl
    return wl.config(cfg, dtype=dtype, rank=rank, world=world)[0]


# state type -> (torch real, torch complex, numpy real, arithmetic label, state label)
DTYPES = {"c64": ("float32", "complex64", np.float32, "f32", "complex64"),
          "c128": ("float64", "complex128", np.float64, "f64", "complex128"),
          "c128df": ("float64", "complex128", np.float64, "f32x2 (double-float)", "complex128")}


# ------------------------------------------------------------------ CPU oracle baseline
def oracle_rate(w_, seconds=12.0, chunk=16, backward=True):
    """Oracle fwd(+bwd) evaluations/s on the host (single thread), on a bounded
    sample of the workload's rows."""
    from oracle import oracle as orc
    done, t0, row = 0, time.perf_counter(), 0
    while time.perf_counter() - t0 < seconds:
        rows = [(row + i) % w_.batch for i in range(chunk)]
        x = w_.x[rows]
        orc.forward(w_.spec, x, w_.w)
        if backward:
            orc.backward(w_.spec, x, w_.w, w_.gE[rows])
        done += chunk
        row += chunk
    dt = time.perf_counter() - t0
    return done / dt, done, dt


def oracle_rate_parallel(w_, seconds=12.0, chunk=16, workers=None, backward=True):
    """The same oracle on all host cores: one thread per core, each cycling its
    own rows (the oracle runs in C; ctypes releases the GIL during each call)."""
    import concurrent.futures as cf
    from oracle import oracle as orc
    workers = workers or os.cpu_count() or 1
    orc.forward(w_.spec, w_.x[:1], w_.w)    # load the library before the threads start
    t0 = time.perf_counter()

    def work(k):
        done, row = 0, k * chunk
        while time.perf_counter() - t0 < seconds:
            rows = [(row + i) % w_.batch for i in range(chunk)]
            x = w_.x[rows]
            orc.forward(w_.spec, x, w_.w)
            if backward:
                orc.backward(w_.spec, x, w_.w, w_.gE[rows])
            done += chunk
            row += chunk * workers
        return done

    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        done = sum(ex.map(work, range(workers)))
    dt = time.perf_counter() - t0
    return done / dt, done, dt, workers


# ------------------------------------------------------------------ our engine
def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    import __graft_entry__
    from paper_2607_11985_gb300 import binding as B
    from paper_2607_11985_gb300.circuit import Circuit

    __graft_entry__.build()
    torch.cuda.set_device(local_rank)
    w_ = workload(args.config, rank, world, args.dtype)
    Bt = w_.batch
    c = Circuit(w_.spec, args.dtype)
    info = c.info(Bt)
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    t_real, t_cplx, np_real, arith, state_kind = DTYPES[args.dtype]
    t_real, t_cplx = getattr(torch, t_real), getattr(torch, t_cplx)
    x = torch.tensor(w_.x, dtype=t_real, device="cuda")
    w = torch.tensor(w_.w, dtype=t_real, device="cuda")
    gE = torch.tensor(w_.gE, dtype=t_real, device="cuda")
    E = torch.empty(Bt, w_.spec.n, dtype=t_real, device="cuda")
    st = torch.empty(Bt, 1 << w_.spec.n, dtype=t_cplx, device="cuda")
    dx = torch.empty_like(x)
    dw = torch.empty_like(w)
    ws, wsb = c.workspace(Bt, 1, stream)
    wsf, wsfb = c.workspace(Bt, 0, stream)
    wsf_ptr = wsf.data_ptr() if wsf is not None else None
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")   # > 129 MB L2

    def step():
        B.vqc_forward(c.plan, Bt, x.data_ptr(), w.data_ptr(), None, E.data_ptr(), st.data_ptr(),
                      wsf_ptr, wsfb, sp)
        B.vqc_backward(c.plan, Bt, x.data_ptr(), w.data_ptr(), None, st.data_ptr(), gE.data_ptr(),
                       dx.data_ptr(), dw.data_ptr(), ws.data_ptr(), wsb, sp)

    for _ in range(args.warmup):
        step()
        if world > 1:
            dist.all_reduce(dw)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()

    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    sampler = ClockSampler(local_rank)
    if rank == 0:
        sampler.start()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda._sleep(int(50e-3 * SM_MAX_MHZ * 1e6))   # queue work ahead of the GPU
    t_wall = time.perf_counter()
    for i in range(K):
        flush.zero_()                                   # L2 flush, outside the step events
        e0, e2 = ev[i]
        e0.record(stream)
        step()          # forward, then the backward from the saved final state
        if world > 1:
            dist.all_reduce(dw)
        e2.record(stream)
    torch.cuda.synchronize()
    t_wall = time.perf_counter() - t_wall
    if world > 1:
        dist.barrier()
    clocks = sampler.stop() if rank == 0 else None
    step_ms = [a.elapsed_time(cc) for a, cc in ev]

    # Each call on its own (for the per-kernel rooflines): an event between the
    # forward and the backward would cut the overlap of the backward's launch
    # with the forward's tail that the timed steps above get.
    def timed_calls(fn, n):
        pairs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                 for _ in range(n)]
        for a, b2 in pairs:
            flush.zero_()
            a.record(stream)
            fn()
            b2.record(stream)
        torch.cuda.synchronize()
        return [a.elapsed_time(b2) for a, b2 in pairs]

    n_calls = max(10, min(K, 1000))
    fwd_ms = timed_calls(lambda: B.vqc_forward(c.plan, Bt, x.data_ptr(), w.data_ptr(), None,
                                               E.data_ptr(), st.data_ptr(), wsf_ptr, wsfb, sp), n_calls)
    bwd_ms = timed_calls(lambda: B.vqc_backward(c.plan, Bt, x.data_ptr(), w.data_ptr(), None,
                                                st.data_ptr(), gE.data_ptr(), dx.data_ptr(),
                                                dw.data_ptr(), ws.data_ptr(), wsb, sp), n_calls)
    # the same step as ONE call when gE is known up front (vqc_forward_backward:
    # one launch on the resident path, no state through HBM)
    wsF, wsFb = c.workspace(Bt, 3, stream)
    wsF_ptr = wsF.data_ptr() if wsF is not None else None
    fused_ms = timed_calls(lambda: B.vqc_forward_backward(
        c.plan, Bt, x.data_ptr(), w.data_ptr(), None, gE.data_ptr(), E.data_ptr(), dx.data_ptr(),
        dw.data_ptr(), wsF_ptr, wsFb, sp), n_calls)
    total_ms = float(sum(step_ms))
    tot = torch.tensor([total_ms], dtype=torch.float64, device="cuda")
    if world > 1:
        dist.all_reduce(tot, op=dist.ReduceOp.MAX)
    total_ms = float(tot.item())
    ms_per_step = total_ms / K
    value = world * Bt * K / (total_ms / 1e3)

    # ---- end to end through the C ABI with HOST buffers (vqc_evaluate_host):
    # every step copies x, w, gE in and E, dx, dw out (one packed copy each way)
    xh = np.ascontiguousarray(w_.x, dtype=np_real)
    wh = np.ascontiguousarray(w_.w, dtype=np_real)
    gh = np.ascontiguousarray(w_.gE, dtype=np_real)
    Eh = np.empty((Bt, w_.spec.n), np_real)
    dxh = np.empty_like(xh)
    dwh = np.empty_like(wh)
    h2d = xh.nbytes + wh.nbytes + gh.nbytes
    d2h = Eh.nbytes + dxh.nbytes + dwh.nbytes

    host_step = c.prepare_host(xh, wh, gh, out=(Eh, dxh, dwh), stream=sp)

    def e2e_step():
        host_step()
        if world > 1:   # the data-parallel dw sum of the step
            t = torch.from_numpy(dwh).to("cuda")
            dist.all_reduce(t)
            dwh[:] = t.cpu().numpy()

    for _ in range(max(3, args.warmup // 4)):
        e2e_step()
    Ke = max(10, min(K, 500))
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(Ke):
        e2e_step()
    e2e_s = time.perf_counter() - t0
    t = torch.tensor([e2e_s], dtype=torch.float64, device="cuda")
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    e2e_value = world * Bt * Ke / float(t.item())
    E_check = float(np.max(np.abs(Eh))) if Eh.size else 0.0
    assert np.isfinite(E_check) and np.all(np.isfinite(dwh))

    if rank != 0:
        return None

    pk, pk_kind = peaks()
    hbm_path = info["bwd_path"] == 1
    # library kernels per step: resident forward 1; resident backward = sweep +
    # fixed-order dw sum; HBM-tiled: one launch per pass plus the partial sums
    # (E; dx and dw), the backward starting from the saved final state
    nw, nx = w_.spec.num_w > 0, w_.spec.num_x > 0
    launches_fwd = info["fwd_passes"] + 1 if info["fwd_path"] == 1 else 1
    launches_bwd = (1 + int(nw)) if not hbm_path else info["bwd_passes"] + int(nx) + int(nw)
    launches_per_step = launches_fwd + launches_bwd
    bwd_avg_s = statistics.mean(bwd_ms) / 1e3
    fwd_avg_s = statistics.mean(fwd_ms) / 1e3
    # measured FMA rates (outside the timed region): packed FP32 for complex64
    # sweeps, FP64 for complex128 ones
    fma = {"fp32_tflops": B.vqc_fma_peak(0), "fp64_tflops": B.vqc_fma_peak(1),
           "kernel": "independent FMA chains over every SM (vqc_fma_peak), best of 5 launches"}
    rname = {"c64": "float", "c128": "double", "c128df": "dd"}[args.dtype]
    if hbm_path and args.dtype == "c64":
        # state bytes the passes move through HBM (vqc_plan_info), against copy bandwidth
        peak = pk.get("hbm_gbs", 6800.0)
        bwd_flops = info["bwd_hbm_bytes_per_eval"] * Bt
        fwd_flops = info["fwd_hbm_bytes_per_eval"] * Bt
        ach_bwd = bwd_flops / bwd_avg_s / 1e9
        ach_fwd = fwd_flops / fwd_avg_s / 1e9
    else:
        if args.dtype == "c64":
            peak = fp32_peak_tflops(pk.get("sm_max_mhz", SM_MAX_MHZ))
            basis = ("FP32 FFMA: 152 SMs x 128 lanes x 2 x %.0f MHz (%s sm_max_mhz)"
                     % (pk.get("sm_max_mhz", SM_MAX_MHZ), pk_kind))
        elif args.dtype == "c128":
            peak = fma["fp64_tflops"]
            basis = "measured FP64 FMA rate (vqc_fma_peak); complex128 sweeps are FP64-bound on GB300"
        else:
            peak = fma["fp32_tflops"] / 15.0
            basis = ("measured FP32 FMA rate / 15: a double-float FMA (2 flops) is 15 FP32 "
                     "instructions on the FMA pipe")
        bwd_flops = info["bwd_flops_per_eval"] * Bt
        fwd_flops = info["fwd_flops_per_eval"] * Bt
        ach_bwd = bwd_flops / bwd_avg_s / 1e12
        ach_fwd = fwd_flops / fwd_avg_s / 1e12
    traffic = None
    tpath = os.path.join(ROOT, "profiles", "traffic.txt")
    if os.path.exists(tpath):
        with open(tpath) as f:
            for line in f:
                parts = line.split()
                if len(parts) >= 4 and not line.startswith("#") and parts[0] == w_.name.split("_rank")[0] \
                        and parts[1] == "bwd" and parts[2] == info_digest():
                    traffic = float(parts[3])
    bytes_bound = hbm_path and args.dtype == "c64"
    out = {
        "metric": METRIC,
        "value": value,
        "unit": "circuit evals/s (fwd+adjoint bwd)",
        "n_gpus": world,
        "steps": K,
        "warmup": args.warmup,
        "ms_per_step": ms_per_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": arith,   # arithmetic type; the state type is config.state
        "data": "synthetic (seeded; RY(x) encoding + RX/RY/RZ layers + CZ ring)",
        "config": {"workload": w_.name.split("_rank")[0], "qubits": w_.spec.n, "state": state_kind,
                   "batch_per_gpu": Bt,
                   "gates": len(w_.spec.gates), "num_x": w_.spec.num_x, "num_w": w_.spec.num_w,
                   "parallelism": "dp%d (batch-sharded replicas, dw all-reduce)" % world,
                   "l2": "flushed between steps (256 MiB write) outside the per-step CUDA events",
                   "fwd_k": info["fwd_k"], "bwd_k": info["bwd_k"],
                   "path": "hbm-tiled" if hbm_path else "resident",
                   "fwd_stages": info["fwd_stages"], "bwd_stages": info["bwd_stages"]},
        "fwd": {"value": world * Bt / fwd_avg_s, "unit": "circuit evals/s (fwd)",
                "ms": fwd_avg_s * 1e3, "achieved": ach_fwd},
        # per-call device times (ms) of this rank: median, mean, std (the paper reports mean +- std)
        "time_stats_ms": {name: {"median": statistics.median(v), "mean": statistics.mean(v),
                                 "std": statistics.pstdev(v), "n": len(v)}
                          for name, v in (("step", step_ms), ("fwd", fwd_ms), ("bwd", bwd_ms),
                                          ("fused", fused_ms))},
        "fused": {"value": world * Bt / (statistics.mean(fused_ms) / 1e3),
                  "unit": "circuit evals/s (fwd+adjoint bwd)",
                  "ms_per_step": statistics.mean(fused_ms),
                  "call": "vqc_forward_backward (gE known before the call, e.g. the mean-<Z> "
                          "objective; one launch)"},
        "roofline": {"kernel": ("pass_kernel<%s,K=%d,bwd> x %d passes" % (rname, info["bwd_k"], info["bwd_passes"]))
                     if hbm_path else "sweep_kernel<%s,K=%d,bwd>" % (rname, info["bwd_k"]),
                     "bound": "hbm" if bytes_bound else "alu",
                     "achieved": ach_bwd, "peak": peak, "unit": "GB/s" if bytes_bound else "TFLOP/s",
                     "frac": ach_bwd / peak, "traffic": traffic,
                     "peak_basis": ("copy bandwidth, %s hbm_gbs" % pk_kind) if bytes_bound else basis,
                     ("bytes_per_call" if bytes_bound else "flops_per_launch"): bwd_flops,
                     "launch_ms": bwd_avg_s * 1e3,
                     "fwd_frac": ach_fwd / peak,
                     "frac_of_measured_fma": ach_bwd / fma["fp32_tflops"]
                     if not bytes_bound and args.dtype == "c64" else None},
        "fma_measured": fma,
        "e2e": {"value": e2e_value, "unit": "circuit evals/s (fwd+adjoint bwd, host buffers)",
                "call": "Circuit.prepare_host -> vqc_evaluate_host (pageable numpy in/out; %s)" % (
                    "kernels access the host arrays in place over NVLink-C2C"
                    if B.vqc_host_direct(local_rank) else "one packed copy each way"),
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": Ke},
        "gpu_launches": launches_per_step * K,
        "clocks": clocks,
        "wall_s_timed_loop": t_wall,
    }
    if not args.no_cpu_baseline:
        rate, done, dt = oracle_rate(w_, seconds=args.cpu_seconds)
        out["cpu_baseline"] = {"value": rate, "unit": "circuit evals/s (fwd+adjoint bwd)",
                               "cores": 1, "kind": "oracle",
                               "sample": "%d rows of the workload (cycled), fwd+bwd, %.1f s"
                                         % (done, dt)}
        prate, pdone, pdt, nw = oracle_rate_parallel(w_, seconds=args.cpu_seconds)
        out["cpu_baseline_all_cores"] = {
            "value": prate, "unit": "circuit evals/s (fwd+adjoint bwd)", "cores": nw,
            "kind": "oracle, batch-parallel threads",
            "sample": "%d rows of the workload (cycled), fwd+bwd, %.1f s" % (pdone, pdt)}
    if args.extra:
        out["configs"] = extra_configs(torch, Circuit, B, fma)
    if args.ablation:
        out["ablation"] = ablation(torch, Circuit, w_)
    if args.regime:
        out["regime_map"] = regime_map(torch, Circuit)
    return out


_DIGEST = None


def info_digest():
    global _DIGEST
    if _DIGEST is None:
        from paper_2607_11985_gb300 import build
        _DIGEST = build._sources_digest()[:16]
    return _DIGEST


def ablation(torch, Circuit, w_):
    """Internal ablation on this engine (the paper's Table 5 design choices),
    8-qubit workload: compile once vs compile per call; one batched launch vs a
    loop over samples; adjoint gradients vs central finite differences (the
    same forward kernel, 2 calls per parameter).  Device and host time."""
    import numpy as np
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


def regime_map(torch, Circuit, qubits=(4, 8, 12, 15, 16, 18, 20), batches=(1, 8, 32, 128), layers=4):
    """Qubits x batch sweep (the paper's regime map, Sec. 4.4): RY(x) encoding,
    `layers` x (RX RY RZ per qubit + CX ring), complex64.  Per point: path, passes,
    device workspace bytes of the backward (the memory the caller must provide
    beyond inputs and outputs), forward and fwd+bwd device time (L2 flushed)."""
    import numpy as np
    from paper_2607_11985_gb300 import binding as Bd
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


def extra_configs(torch, Circuit, B, fma=None):
    """Forward and fwd+bwd evaluations/s and roofline fractions of the other
    workloads (device time, L2 flushed before each timed call)."""
    from paper_2607_11985_gb300 import workloads as wl
    pk, _ = peaks()
    fp32 = fp32_peak_tflops(pk.get("sm_max_mhz", SM_MAX_MHZ))
    hbm = pk.get("hbm_gbs", 6800.0)
    fp64 = fma["fp64_tflops"] if fma else None
    res = {}
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    # (name, config, dtype, batch): the 8-qubit circuit also at a large batch, where
    # the sweep is throughput-bound rather than latency-bound
    cases = [("cfg1", 1, None, None), ("cfg2_B65536", 2, None, 65536), ("cfg3", 3, None, None),
             ("cfg3_c128", 3, "c128", None), ("cfg3_c128df", 3, "c128df", None), ("cfg4", 4, None, None),
             ("cfg5_c64", 5, "c64", None), ("cfg5_c128", 5, "c128", None), ("cfg5_c128df", 5, "c128df", None)]
    for key, k, dt, bsz in cases:
        try:
            ws_ = wl.config(k, dtype=dt, batch=bsz)
            tot_f = tot_b = 0.0
            evals = 0
            work_f = work_b = flop_f = flop_b = 0.0
            path = None
            for w_ in ws_:
                real = torch.float32 if w_.dtype == "c64" else torch.float64
                c = Circuit(w_.spec, w_.dtype)
                inf = c.info(w_.batch)
                path = {0: "resident", 1: "hbm-tiled", 2: "cluster"}[inf["fwd_path"]]
                x = torch.tensor(w_.x, dtype=real, device="cuda")
                w = torch.tensor(w_.w, dtype=real, device="cuda") if w_.spec.num_w else None
                gE = torch.tensor(w_.gE, dtype=real, device="cuda")
                E, st = c.forward(x, w, want_state=True)
                if w_.backward:
                    c.backward(x, w, gE, psi_final=st)
                torch.cuda.synchronize()
                n_rep = 3 if k == 5 else 5
                for _ in range(n_rep):
                    flush.zero_()
                    a, b2, d = (torch.cuda.Event(enable_timing=True) for _ in range(3))
                    a.record()
                    c.forward(x, w, out=E, state_out=st)
                    b2.record()
                    if w_.backward:
                        c.backward(x, w, gE, psi_final=st)
                    d.record()
                    torch.cuda.synchronize()
                    tot_f += a.elapsed_time(b2) / 1e3
                    tot_b += b2.elapsed_time(d) / 1e3
                evals += n_rep * w_.batch
                if path == "hbm-tiled":
                    work_f += n_rep * w_.batch * inf["fwd_hbm_bytes_per_eval"]
                    work_b += n_rep * w_.batch * inf["bwd_hbm_bytes_per_eval"] if w_.backward else 0
                flop_f += n_rep * w_.batch * inf["fwd_flops_per_eval"]
                flop_b += n_rep * w_.batch * inf["bwd_flops_per_eval"] if w_.backward else 0
                del c
            r = {"path": path, "circuits": len(ws_), "batch": ws_[0].batch,
                 "qubits": sorted({w_.spec.n for w_ in ws_}), "dtype": ws_[0].dtype,
                 "fwd_evals_per_s": evals / tot_f,
                 "fwd_bwd_evals_per_s": (evals / (tot_f + tot_b)) if flop_b else None}
            if path == "hbm-tiled":
                r["fwd_gbs"] = work_f / tot_f / 1e9
                r["bwd_gbs"] = work_b / tot_b / 1e9 if work_b else None
                r["fwd_frac_hbm"] = r["fwd_gbs"] / hbm
                r["bwd_frac_hbm"] = r["bwd_gbs"] / hbm if work_b else None
            # algorithmic flop rates against the arithmetic ceiling of the state type
            r["fwd_tflops"] = flop_f / tot_f / 1e12
            r["bwd_tflops"] = flop_b / tot_b / 1e12 if flop_b else None
            if r["dtype"] == "c64":
                r["fwd_frac_fp32"] = r["fwd_tflops"] / fp32
                r["bwd_frac_fp32"] = r["bwd_tflops"] / fp32 if flop_b else None
            elif fp64:
                # complex128 flops against the native FP64 ceiling (double-float
                # runs on the FP32 units, so it can exceed 1)
                r["fwd_frac_fp64_measured"] = r["fwd_tflops"] / fp64
                r["bwd_frac_fp64_measured"] = r["bwd_tflops"] / fp64 if flop_b else None
            if r["dtype"] == "c128df" and fma:
                # and against the double-float ceiling: measured FP32 rate / 15
                # (a double-float FMA, 2 flops, is 15 FP32 instructions)
                r["fwd_frac_df_ceiling"] = r["fwd_tflops"] / (fma["fp32_tflops"] / 15.0)
                r["bwd_frac_df_ceiling"] = r["bwd_tflops"] / (fma["fp32_tflops"] / 15.0) if flop_b else None
            if r["dtype"] == "c128df" and key.replace("df", "") in res and "fwd_evals_per_s" in res[key.replace("df", "")]:
                ref = res[key.replace("df", "")]
                r["fwd_speedup_vs_fp64"] = r["fwd_evals_per_s"] / ref["fwd_evals_per_s"]
                if flop_b and ref.get("fwd_bwd_evals_per_s"):
                    r["fwd_bwd_speedup_vs_fp64"] = r["fwd_bwd_evals_per_s"] / ref["fwd_bwd_evals_per_s"]
            res[key] = r
        except Exception as e:   # report, do not hide
            res[key] = {"error": str(e)[:200]}
    return res


# ------------------------------------------------------------------ reference arm
def run_reference(args, rank, world):
    """The oracle on the host cores, same metric and workload (bounded sample)."""
    if rank != 0:
        return None
    w_ = workload(args.config, dtype=args.dtype)
    chunk = 8
    from oracle import oracle as orc
    orc.build()
    for _ in range(args.warmup):
        orc.forward(w_.spec, w_.x[:1], w_.w)
    times, row = [], 0
    for _ in range(args.steps):
        rows = [(row + i) % w_.batch for i in range(chunk)]
        t0 = time.perf_counter()
        orc.forward(w_.spec, w_.x[rows], w_.w)
        orc.backward(w_.spec, w_.x[rows], w_.w, w_.gE[rows])
        times.append(time.perf_counter() - t0)
        row += chunk
    total = sum(times)
    value = chunk * args.steps / total
    return {"metric": METRIC, "value": value, "unit": "circuit evals/s (fwd+adjoint bwd)",
            "impl": "reference", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": total / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)", "config": {"workload": w_.name, "qubits": w_.spec.n,
                                                    "batch_per_step": chunk},
            "cpu_baseline": {"value": value, "unit": "circuit evals/s (fwd+adjoint bwd)",
                             "cores": 1, "kind": "oracle",
                             "sample": "%d steps x %d rows of the workload" % (args.steps, chunk)},
            "e2e": {"value": value, "unit": "circuit evals/s (fwd+adjoint bwd)",
                    "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=2)
    ap.add_argument("--dtype", default="c64", choices=sorted(DTYPES),
                    help="state type of the timed workload (c128df: complex128 in double-float)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--extra", action="store_true", help="also time configs 1, 3, 4 and 5")
    ap.add_argument("--regime", action="store_true",
                    help="qubits x batch sweep to 20 qubits (HBM-tiled beyond one SM's state)")
    ap.add_argument("--ablation", action="store_true",
                    help="compile-once / batching / adjoint-vs-FD ablation on the bench workload")
    args = ap.parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
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
