"""CPU checks of bench.py's arithmetic (no GPU): the algorithmic flop counts
behind the reported roofline fractions, and the roofline bound selection.

Counting rule of the hot-path scope (per amplitude: 14 flops per fused
single-qubit run, 6 per RZZ, 3 per CRZ, 0 for permutations; <Z> adds (3 + n)):
forward F = sum_f 2^n + (3 + n) 2^n; backward = 2 sum_f 2^n + 4 2^n (angle
slots) + (n + 2) 2^n.  The 8-qubit workload has 32 fused runs (RY(x) fuses into
the first layer's runs), 104 angle slots and 2^8 amplitudes:
forward 32*14*256 + 11*256 = 117,504; backward 2*32*14*256 + 4*256*104 +
10*256 = 338,432.
"""
import pytest

import bench
from paper_2607_11985_gb300 import workloads as wl

pytest.importorskip("torch")


def test_flops_per_eval_8_qubit_workload():
    from paper_2607_11985_gb300.circuit import Circuit
    info = Circuit(wl.config(2)[0].spec, "c64").info(1024)
    assert info["num_runs"] == 32 and info["num_terms"] == 104
    fwd, bwd = bench.flops_per_eval(info)
    assert fwd == 117504.0
    assert bwd == 338432.0


def test_roofline_bound_is_the_closer_ceiling():
    fma = {"fp32_tflops": 80.0, "fp64_tflops": 1.0}
    pk = {"hbm_gbs": 6000.0, "sm_max_mhz": 2000.0}
    info = {"num_qubits": 16, "fwd_flops_per_eval": 100e6, "num_terms": 10,
            "fwd_path": 1, "bwd_path": 1, "fwd_hbm_bytes_per_eval": 1e7, "bwd_hbm_bytes_per_eval": 2e7}
    r = bench.rooflines([(info, 100, 1e-3, 2e-3)], "c64", fma, pk, "test")
    for name, secs, nbytes in (("fwd", 1e-3, 1e9), ("bwd", 2e-3, 2e9)):
        hb = r[name]["hbm"]
        assert abs(hb["achieved"] - nbytes / secs / 1e9) < 1e-9
        assert r[name]["bound"] == max(("alu", "hbm"), key=lambda k: r[name][k]["frac"])
        assert r[name]["frac"] == r[name][r[name]["bound"]]["frac"]
    # a resident call has only the arithmetic ceiling
    info2 = dict(info, fwd_path=0, bwd_path=0)
    assert bench.rooflines([(info2, 100, 1e-3, 2e-3)], "c64", fma, pk, "test")["bwd"]["bound"] == "alu"
    # double-float ceiling: the FP32 instruction rate x 14 / 86
    r3 = bench.rooflines([(info2, 100, 1e-3, None)], "c128df", fma, pk, "test")
    assert abs(r3["fwd"]["alu"]["peak"] - 80.0 / 2 * 14 / 86) < 1e-12


def test_launch_count_per_step():
    """gpu_launches: every library kernel of a step (the driver compares this
    claim with the ncu launch list): HBM forward = per-sample tables + passes +
    the <Z> sum; HBM backward = passes + per-sample terms + dx sum + dw sum
    (+ the tables outside complex64); resident forward 1, backward 2 (sweep +
    dw sum); cluster backward 2."""
    class Spec:
        num_x, num_w = 16, 384

    class W:
        spec, backward, dtype = Spec(), True, "c64"

    b = bench.CircuitBench.__new__(bench.CircuitBench)
    b.w_ = W()
    b.info = {"fwd_path": 1, "bwd_path": 1, "fwd_passes": 11, "bwd_passes": 12}
    assert b.launches() == (11 + 1 + 1) + (12 + 1 + 1 + 1)
    b.w_.dtype = "c128"   # the complex128 backward reads the per-sample tables too
    assert b.launches() == (11 + 1 + 1) + (12 + 1 + 1 + 1 + 1)
    b.w_.dtype = "c64"
    b.info = {"fwd_path": 0, "bwd_path": 0, "fwd_passes": 1, "bwd_passes": 1}
    assert b.launches() == 1 + 2
    b.info = {"fwd_path": 0, "bwd_path": 2, "fwd_passes": 1, "bwd_passes": 1}
    assert b.launches() == 1 + 2
