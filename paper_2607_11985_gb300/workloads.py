"""Seeded synthetic workloads: circuits and input arrays, nothing else.

This module holds no simulation arithmetic.  It draws gate lists and angle /
upstream-gradient arrays from numpy's PCG64 generator and returns them in a
neutral form that both the CUDA engine's binding and the CPU oracle marshal
into their own formats.

A circuit is a ``CircuitSpec``: ``gates`` is a list, in time order (first gate
applied first), of ``(name, qubits, params)`` where ``params`` is a tuple of
``(kind, value)`` with kind ``"x"`` (per-sample angle column ``value``), ``"w"``
(shared weight index ``value``) or ``"c"`` (constant angle ``value``).

The five workloads follow the shapes of the paper's variational QML workloads
(Sec. 4.1.1: qnn / vqe families, 4..20 qubits, batched): layered RX/RY/RZ/Rot
ansatze with ring entanglers, plus seeded random static circuits over the
16-gate set.  The paper's own benchmark suite (MQT Bench) is not available
here; these seeded circuits stand in for it.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Tuple

import numpy as np

GATES_1Q_FIXED = ("H", "X", "Y", "Z", "S", "T", "SX")
GATES_1Q_PARAM = ("RX", "RY", "RZ", "U3")
GATES_2Q_FIXED = ("CX", "CZ", "SWAP")
GATES_2Q_PARAM = ("CRZ", "RZZ")
ALL_GATES = GATES_1Q_FIXED + GATES_1Q_PARAM + GATES_2Q_FIXED + GATES_2Q_PARAM
NPARAMS = {"RX": 1, "RY": 1, "RZ": 1, "CRZ": 1, "RZZ": 1, "U3": 3}
TWO_QUBIT = set(GATES_2Q_FIXED + GATES_2Q_PARAM)

Gate = Tuple[str, Tuple[int, ...], Tuple[Tuple[str, float], ...]]


@dataclass
class CircuitSpec:
    n: int
    num_x: int
    num_w: int
    gates: List[Gate] = field(default_factory=list)

    def add(self, name: str, qubits, params=()):
        self.gates.append((name, tuple(int(q) for q in qubits), tuple(params)))
        return self


@dataclass
class Workload:
    name: str
    spec: CircuitSpec
    batch: int
    x: np.ndarray          # [B, num_x] float64 holding dtype-rounded values
    w: np.ndarray          # [num_w]
    gE: np.ndarray         # [B, n]
    dtype: str             # "c64", "c128" or "c128df" (complex128 storage)
    seed: int
    backward: bool = True


def _round(a: np.ndarray, dtype: str) -> np.ndarray:
    """Round to the engine's real type and promote back to float64, so the
    oracle consumes exactly the values the engine sees."""
    if dtype == "c64":
        return np.asarray(a, np.float64).astype(np.float32).astype(np.float64)
    return np.asarray(a, np.float64)


def layered(n: int, layers: int, rotations: Tuple[str, ...], entangler: str,
            reupload: bool = False, ring_range=None) -> CircuitSpec:
    """RY(x_q) encoding (once, or at the start of every layer when ``reupload``),
    then per layer ``rotations`` (time order) on every qubit with shared weights
    w[(l*n + q)*R + r], then a ring of ``entangler`` gates (i, (i + r_l) mod n)
    for i = 0..n-1 applied in increasing i."""
    R = len(rotations)
    spec = CircuitSpec(n=n, num_x=n, num_w=layers * n * R)
    if not reupload:
        for q in range(n):
            spec.add("RY", (q,), (("x", q),))
    for l in range(layers):
        if reupload:
            for q in range(n):
                spec.add("RY", (q,), (("x", q),))
        for q in range(n):
            for r, rot in enumerate(rotations):
                spec.add(rot, (q,), (("w", (l * n + q) * R + r),))
        rng_r = 1 if ring_range is None else ring_range(l)
        for i in range(n):
            spec.add(entangler, (i, (i + rng_r) % n))
    return spec


def random_circuit(rng: np.random.Generator, n: int, num_gates: int,
                   p_two: float = 0.3, p_param: float = 0.4,
                   weight_fraction: float = 0.0, const_fraction: float = 0.0) -> CircuitSpec:
    """Random static circuit over the 16-gate set.  Two-qubit-ness and
    parametrisedness are independent Bernoulli draws; the gate is uniform within
    its category; q0 ~ U[0,n), q1 ~ U([0,n) minus q0).  Every angle gets its own
    source: a new x column by default, a new shared weight with probability
    ``weight_fraction``, or a constant U(-pi, pi) angle with probability
    ``const_fraction``."""
    spec = CircuitSpec(n=n, num_x=0, num_w=0)
    for _ in range(num_gates):
        two = rng.random() < p_two
        par = rng.random() < p_param
        if n < 2:
            two = False
        cat = (GATES_2Q_PARAM if par else GATES_2Q_FIXED) if two else \
              (GATES_1Q_PARAM if par else GATES_1Q_FIXED)
        name = cat[int(rng.integers(len(cat)))]
        q0 = int(rng.integers(n))
        qubits = (q0,)
        if two:
            qubits = (q0, (q0 + 1 + int(rng.integers(n - 1))) % n)
        params = []
        for _p in range(NPARAMS.get(name, 0)):
            u = rng.random()
            if u < const_fraction:
                params.append(("c", float(rng.uniform(-np.pi, np.pi))))
            elif u < const_fraction + weight_fraction:
                params.append(("w", spec.num_w))
                spec.num_w += 1
            else:
                params.append(("x", spec.num_x))
                spec.num_x += 1
        spec.add(name, qubits, params)
    return spec


CONFIG_NAMES = {
    1: "n4_L2_B64_c64",
    2: "n8_L4_B1024_c64",
    3: "n12_L6_B4096_c64_reupload",
    4: "random32_n10-14_B256_c64_fwd",
    5: "n16_L8_B512",
}


def config(k: int, dtype: Optional[str] = None, batch: Optional[int] = None,
           rank: int = 0, world: int = 1) -> List[Workload]:
    """The five workloads.  Returns a list (config 4 holds 32 circuits).

    With ``world`` > 1 the global batch is ``world`` x batch rows and this returns
    rank ``rank``'s contiguous shard; rank 0 of any world sees the same rows as
    world = 1 (each array has its own PCG64 stream, filled row by row)."""
    if k == 1:
        spec = layered(4, 2, ("RY", "RZ"), "CX")
        return [_draw("cfg1_" + CONFIG_NAMES[1], spec, batch or 64, dtype or "c64", 1001,
                      "uniform", rank, world)]
    if k == 2:
        spec = layered(8, 4, ("RX", "RY", "RZ"), "CZ")
        return [_draw("cfg2_" + CONFIG_NAMES[2], spec, batch or 1024, dtype or "c64", 1002,
                      "uniform", rank, world)]
    if k == 3:
        # Rot(phi, theta, omega) = RZ(omega) RY(theta) RZ(phi): RZ(phi) first.
        spec = layered(12, 6, ("RZ", "RY", "RZ"), "CX", reupload=True,
                       ring_range=lambda l: (l % 11) + 1)
        return [_draw("cfg3_" + CONFIG_NAMES[3], spec, batch or 4096, dtype or "c64", 1003,
                      "normal", rank, world)]
    if k == 4:
        out = []
        B = batch or 256
        for c in range(32):
            rng = np.random.Generator(np.random.PCG64(4000 + c))
            n = int(rng.integers(10, 15))
            G = int(rng.integers(200, 801))
            spec = random_circuit(rng, n, G)
            arng = np.random.Generator(np.random.PCG64(5000 + c))
            dt = dtype or "c64"
            x = _round(arng.uniform(-np.pi, np.pi, (B, spec.num_x)), dt)
            out.append(Workload("cfg4_circuit%02d_n%d_G%d" % (c, n, G), spec, B, x,
                                np.zeros(0), np.zeros((B, n)), dt, 4000 + c, backward=False))
        return out
    if k == 5:
        spec = layered(16, 8, ("RX", "RY", "RZ"), "CX")
        return [_draw("cfg5_" + CONFIG_NAMES[5] + "_" + (dtype or "c64"), spec, batch or 512,
                      dtype or "c64", 1005, "uniform", rank, world)]
    raise ValueError("config must be 1..5")


def _draw(name, spec, B, dtype, seed, xdist, rank=0, world=1) -> Workload:
    sx, sw, sg = np.random.SeedSequence(seed).spawn(3)
    rx, rw, rg = (np.random.Generator(np.random.PCG64(s)) for s in (sx, sw, sg))
    rows = B * (rank + 1)            # fill up to the end of this rank's shard
    if xdist == "normal":
        x = rx.standard_normal((rows, spec.num_x))
    else:
        x = rx.uniform(-np.pi, np.pi, (rows, spec.num_x))
    w = rw.uniform(-np.pi, np.pi, spec.num_w)
    gE = rg.standard_normal((rows, spec.n))
    x, gE = x[B * rank:], gE[B * rank:]
    if world > 1:
        name = "%s_rank%dof%d" % (name, rank, world)
    return Workload(name, spec, B, _round(x, dtype), _round(w, dtype), _round(gE, dtype),
                    dtype, seed)


def small_random(seed: int, n: int, num_gates: int, batch: int, dtype: str = "c128",
                 weight_fraction: float = 0.5, const_fraction: float = 0.1,
                 with_psi0: bool = False):
    """A small random circuit plus inputs, for parity tests at sizes the oracle
    finishes quickly.  Returns (Workload, psi0 or None)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    spec = random_circuit(rng, n, num_gates, weight_fraction=weight_fraction,
                          const_fraction=const_fraction)
    x = _round(rng.uniform(-np.pi, np.pi, (batch, spec.num_x)), dtype)
    w = _round(rng.uniform(-np.pi, np.pi, spec.num_w), dtype)
    gE = _round(rng.standard_normal((batch, n)), dtype)
    psi0 = None
    if with_psi0:
        z = rng.standard_normal((batch, 1 << n)) + 1j * rng.standard_normal((batch, 1 << n))
        z /= np.linalg.norm(z, axis=1, keepdims=True)
        if dtype == "c64":
            z = z.astype(np.complex64).astype(np.complex128)
        psi0 = z
    return Workload("random_n%d_G%d_s%d" % (n, num_gates, seed), spec, batch, x, w, gE,
                    dtype, seed), psi0
