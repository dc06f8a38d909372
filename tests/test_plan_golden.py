"""Plan and index construction, bit-exact (CPU).

vqc_plan_export's bytes (fused ops, table entries and constituents, constant
matrices, gradient terms, accumulators, occurrence lists, and every stage and
pass schedule with its addressing records) must equal those built by an
independent implementation of the compile phase (tests/golden_plan.py, paper
Alg. 1 compile phase), which does not call the library.  Covered: the
workloads up to 14 qubits, random circuits over the whole gate set with
constant, per-sample and shared angles, every gate in both qubit orders, and
the degenerate circuits; complex64, complex128 and double-float plans (the
last export the complex128 bytes); resident and HBM-tiled schedules.
"""
import numpy as np
import pytest

from paper_2607_11985_gb300 import workloads as wl
from tests import golden_plan as gp

pytest.importorskip("torch")


def engine_bytes(spec, dtype):
    from paper_2607_11985_gb300.circuit import Circuit
    return Circuit(spec, dtype).export()


def assert_same(spec, dtype):
    a, b = engine_bytes(spec, dtype), gp.plan_bytes(spec, dtype)
    if a != b:
        first = next((i for i in range(min(len(a), len(b))) if a[i] != b[i]), min(len(a), len(b)))
        raise AssertionError("plan bytes differ at offset %d (engine %d bytes, golden %d)"
                             % (first, len(a), len(b)))


@pytest.fixture(autouse=True)
def default_tiles(monkeypatch):
    monkeypatch.delenv("VQC_HBM_TILE_QUBITS", raising=False)


@pytest.mark.parametrize("dtype", ["c64", "c128", "c128df"])
@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_workload_plans(cfg, dtype):
    assert_same(wl.config(cfg, dtype=dtype)[0].spec, dtype)


@pytest.mark.parametrize("dtype", ["c64", "c128"])
def test_sixteen_qubit_workload_plan(dtype):
    """Cluster schedules (forward and backward, with their CTA-locality flags)
    and the HBM passes of the 16-qubit / 8-layer workload."""
    assert_same(wl.config(5, dtype=dtype)[0].spec, dtype)


@pytest.mark.parametrize("n,dtype", [(13, "c128"), (14, "c64"), (14, "c128"), (15, "c64"), (15, "c128")])
def test_cluster_range_plans(n, dtype):
    """Every state size with a cluster schedule, on a layered circuit with a
    CX ring, a CZ and a phase gate."""
    spec = wl.layered(n, 2, ("RX", "RY"), "CX")
    spec.add("CZ", (0, n - 1)).add("RZZ", (2, n - 2), [("w", 0)]).add("CRZ", (n - 1, 1), [("x", 0)])
    assert_same(spec, dtype)


def test_random_circuit_workload_plans():
    for w_ in wl.config(4)[::4]:
        assert_same(w_.spec, "c64")


@pytest.mark.parametrize("dtype", ["c64", "c128"])
def test_random_circuits_every_gate(dtype):
    seen = set()
    for seed in range(48):
        n = 1 + seed % 13
        w_, _ = wl.small_random(8100 + seed, n, 10 + 9 * seed, batch=1, dtype=dtype)
        seen |= {g[0] for g in w_.spec.gates}
        assert_same(w_.spec, dtype)
    assert seen == set(wl.ALL_GATES)


@pytest.mark.parametrize("dtype", ["c64", "c128"])
def test_each_gate_both_orders_and_sources(dtype):
    for name in wl.ALL_GATES:
        for q in ((0, 6), (6, 0), (2, 5)):
            for src in ("c", "x", "w"):
                spec = wl.CircuitSpec(7, 3, 3)
                spec.add("H", (3,)).add("RY", (q[0],), [("x", 0)])
                params = [(src, 0.4 if src == "c" else 1), ("w", 2), ("c", -0.9)][:wl.NPARAMS.get(name, 0)]
                spec.add(name, q if name in wl.TWO_QUBIT else (q[0],), params)
                spec.add("RX", (q[1],), [("w", 0)]).add("CX", (q[1], 3)).add("T", (q[1],))
                assert_same(spec, dtype)


def test_degenerate_circuits():
    assert_same(wl.CircuitSpec(3, 0, 0), "c64")
    spec = wl.CircuitSpec(8, 0, 0)
    for q in range(7):
        spec.add("CX", (q, q + 1)).add("CZ", (q + 1, q)).add("SWAP", (q, 7 - q) if q != 7 - q else (q, 0))
    assert_same(spec, "c64")
    assert_same(spec, "c128")
    one = wl.CircuitSpec(1, 1, 1).add("RY", (0,), [("x", 0)]).add("RZ", (0,), [("w", 0)])
    assert_same(one, "c64")
