"""Pins for the CPU oracle, independent of the oracle's own code paths.

Each check ties the oracle to something it does not compute itself:
  * gate matrices: matrix exponentials of Pauli generators (scipy.linalg.expm),
    algebraic identities (H Z H = X, S^2 = Z, T^2 = S, SX^2 = X, ...), Qiskit's
    U-gate special cases, finite differences for the derivative matrices;
  * gate application: dense 2^n x 2^n operators built from Kronecker products of
    embedded single-qubit operators, multiplied in time order (brute force);
  * closed forms: RY(t)|0> gives <Z> = cos t, encoding layers give cos x, GHZ,
    all-zero angles give |0...0>, Z-diagonal layers leave <Z> = cos x;
  * invariants: norm, circuit followed by its inverse, batch independence,
    qubit relabelling;
  * gradients: two-term parameter-shift rule (exact for exp(-i t P / 2) with
    P^2 = I), CRZ through its CX/RZ decomposition, central finite differences.

The oracle evaluates Alg. 1 (statevector + Pauli-Z expectation) and the exact
gradient of L = sum gE * E (Sec. 3); these tests never call anything under the
package's CUDA path.
"""
import json
import os

import numpy as np
import pytest
import scipy.linalg

from oracle import oracle as orc
from paper_2607_11985_gb300 import workloads as wl

HERE = os.path.dirname(os.path.abspath(__file__))

I2 = np.eye(2, dtype=complex)
PX = np.array([[0, 1], [1, 0]], dtype=complex)
PZ = np.array([[1, 0], [0, -1]], dtype=complex)
PY = 1j * PX @ PZ          # = [[0,-i],[i,0]]
P0 = np.array([[1, 0], [0, 0]], dtype=complex)
P1 = np.array([[0, 0], [0, 1]], dtype=complex)
ANGLES = [0.0, 0.3, -1.1, np.pi / 2, 2.7, -np.pi]


def kron_local(A0, A1):
    """4x4 operator A0 on the first qubit (bit b0) and A1 on the second (b1),
    in the local index s = b0 + 2*b1 used for 2q gates."""
    return np.kron(A1, A0)


# ----------------------------------------------------------------------------- gates

def test_pauli_constants():
    assert np.allclose(PY, [[0, -1j], [1j, 0]])
    assert np.allclose(orc.gate_matrix("X"), PX)
    assert np.allclose(orc.gate_matrix("Z"), PZ)
    assert np.allclose(orc.gate_matrix("Y"), 1j * PX @ PZ)


@pytest.mark.parametrize("name", wl.ALL_GATES)
def test_gates_unitary(name):
    rng = np.random.default_rng(7)
    for _ in range(5):
        U = orc.gate_matrix(name, rng.uniform(-np.pi, np.pi, 3))
        assert np.allclose(U @ U.conj().T, np.eye(U.shape[0]), atol=1e-14)


@pytest.mark.parametrize("t", ANGLES)
def test_rotations_are_exponentials(t):
    assert np.allclose(orc.gate_matrix("RX", (t,)), scipy.linalg.expm(-0.5j * t * PX), atol=1e-14)
    assert np.allclose(orc.gate_matrix("RY", (t,)), scipy.linalg.expm(-0.5j * t * PY), atol=1e-14)
    assert np.allclose(orc.gate_matrix("RZ", (t,)), scipy.linalg.expm(-0.5j * t * PZ), atol=1e-14)
    assert np.allclose(orc.gate_matrix("RZZ", (t,)),
                       scipy.linalg.expm(-0.5j * t * kron_local(PZ, PZ)), atol=1e-14)
    # CRZ: control = first qubit, generator |1><1|_c (x) Z_t
    assert np.allclose(orc.gate_matrix("CRZ", (t,)),
                       scipy.linalg.expm(-0.5j * t * kron_local(P1, PZ)), atol=1e-14)


def test_fixed_gate_identities():
    H, S, T, SX = (orc.gate_matrix(g) for g in ("H", "S", "T", "SX"))
    assert np.allclose(H @ H, I2)
    assert np.allclose(H @ PZ @ H, PX)
    assert np.allclose(H @ PX @ H, PZ)
    assert H[0, 0].real > 0 and H[0, 1].real > 0      # H|0> = |+>
    assert np.allclose(S @ S, PZ)
    assert np.allclose(S[0, 0], 1) and np.allclose(S[1, 1], 1j)
    assert np.allclose(T @ T, S)
    assert np.allclose(T[0, 0], 1)
    assert np.allclose(SX @ SX, PX)
    assert np.allclose(SX, np.exp(1j * np.pi / 4) * scipy.linalg.expm(-0.25j * np.pi * PX))


def test_two_qubit_fixed_gates():
    CX, CZ, SWAP = (orc.gate_matrix(g) for g in ("CX", "CZ", "SWAP"))
    assert np.allclose(CX, kron_local(P0, I2) + kron_local(P1, PX))
    assert np.allclose(CZ, kron_local(P0, I2) + kron_local(P1, PZ))
    rng = np.random.default_rng(3)
    A = rng.standard_normal((2, 2)) + 1j * rng.standard_normal((2, 2))
    B = rng.standard_normal((2, 2)) + 1j * rng.standard_normal((2, 2))
    assert np.allclose(SWAP @ kron_local(A, B) @ SWAP, kron_local(B, A))
    assert np.allclose(SWAP @ SWAP, np.eye(4))


@pytest.mark.parametrize("t", ANGLES)
def test_u3(t):
    rng = np.random.default_rng(11)
    ph, lam = rng.uniform(-np.pi, np.pi, 2)
    RZ = lambda a: orc.gate_matrix("RZ", (a,))
    RY = lambda a: orc.gate_matrix("RY", (a,))
    U = orc.gate_matrix("U3", (t, ph, lam))
    assert np.allclose(U, np.exp(0.5j * (ph + lam)) * RZ(ph) @ RY(t) @ RZ(lam), atol=1e-14)
    assert np.allclose(orc.gate_matrix("U3", (t, -np.pi / 2, np.pi / 2)), orc.gate_matrix("RX", (t,)))
    assert np.allclose(orc.gate_matrix("U3", (t, 0, 0)), orc.gate_matrix("RY", (t,)))
    assert orc.gate_matrix("U3", (t, ph, lam))[0, 0].imag == 0


def test_crz_decomposition():
    # CRZ(t) = CX . RZ_t(-t/2) . CX . RZ_t(t/2)  (operator product; RZ(t/2) first)
    for t in ANGLES:
        CX = orc.gate_matrix("CX")
        rz = lambda a: kron_local(I2, orc.gate_matrix("RZ", (a,)))
        assert np.allclose(orc.gate_matrix("CRZ", (t,)), CX @ rz(-t / 2) @ CX @ rz(t / 2), atol=1e-14)


@pytest.mark.parametrize("name", ["RX", "RY", "RZ", "U3", "CRZ", "RZZ"])
def test_derivative_matrices_fd(name):
    rng = np.random.default_rng(5)
    h = 1e-6
    for _ in range(4):
        th = rng.uniform(-np.pi, np.pi, 3)
        for p in range(wl.NPARAMS[name]):
            tp, tm = th.copy(), th.copy()
            tp[p] += h
            tm[p] -= h
            fd = (orc.gate_matrix(name, tp) - orc.gate_matrix(name, tm)) / (2 * h)
            assert np.allclose(orc.gate_matrix_deriv(name, th, p), fd, atol=1e-8)


# ----------------------------------------------------------------------------- brute force

def embed1(n, q, A):
    """I (x) ... (x) A (x) ... (x) I with A at bit q (little endian)."""
    return np.kron(np.kron(np.eye(1 << (n - q - 1)), A), np.eye(1 << q))


def dense_gate(n, name, qubits, th):
    M = orc.gate_matrix(name, th)
    if M.shape[0] == 2:
        return embed1(n, qubits[0], M)
    q0, q1 = qubits
    full = np.zeros((1 << n, 1 << n), dtype=complex)
    for so in range(4):
        for si in range(4):
            if M[so, si] == 0:
                continue
            e0 = np.zeros((2, 2)); e0[so & 1, si & 1] = 1
            e1 = np.zeros((2, 2)); e1[so >> 1, si >> 1] = 1
            full += M[so, si] * embed1(n, q0, e0) @ embed1(n, q1, e1)
    return full


def resolve(params, xb, w):
    th = np.zeros(3)
    for p, (kind, v) in enumerate(params):
        th[p] = v if kind == "c" else (xb[int(v)] if kind == "x" else w[int(v)])
    return th


def dense_circuit(spec, xb, w):
    U = np.eye(1 << spec.n, dtype=complex)
    for name, qubits, params in spec.gates:
        U = dense_gate(spec.n, name, qubits, resolve(params, xb, w)) @ U
    return U


@pytest.mark.parametrize("n,seed", [(1, 1), (2, 2), (3, 3), (4, 4), (5, 5)])
def test_forward_matches_dense_kronecker(n, seed):
    w_, psi0 = wl.small_random(seed, n, 40, batch=3, dtype="c128", with_psi0=True)
    spec = w_.spec
    E, st = orc.forward(spec, w_.x, w_.w, psi0=psi0, want_state=True)
    for b in range(3):
        U = dense_circuit(spec, w_.x[b] if spec.num_x else None, w_.w)
        ref = U @ psi0[b]
        assert np.allclose(st[b], ref, atol=1e-12)
        for j in range(n):
            Zj = embed1(n, j, PZ)
            assert abs(E[b, j] - np.vdot(ref, Zj @ ref).real) < 1e-12


def test_every_gate_every_placement():
    n = 4
    rng = np.random.default_rng(0)
    psi = rng.standard_normal(16) + 1j * rng.standard_normal(16)
    psi /= np.linalg.norm(psi)
    for name in wl.ALL_GATES:
        pairs = [(a, b) for a in range(n) for b in range(n) if a != b] if name in wl.TWO_QUBIT \
            else [(a,) for a in range(n)]
        for qs in pairs:
            th = rng.uniform(-np.pi, np.pi, 3)
            spec = wl.CircuitSpec(n, 0, 0).add(name, qs, [("c", t) for t in th[:wl.NPARAMS.get(name, 0)]])
            _, st = orc.forward(spec, None, None, psi0=psi[None], want_state=True)
            ref = dense_gate(n, name, qs, th) @ psi
            assert np.allclose(st[0], ref, atol=1e-13), (name, qs)


# ----------------------------------------------------------------------------- closed forms

@pytest.mark.parametrize("t", ANGLES)
def test_single_rotation_closed_form(t):
    for g in ("RY", "RX"):
        spec = wl.CircuitSpec(1, 1, 0).add(g, (0,), [("x", 0)])
        E = orc.forward(spec, np.array([[t]]), None)
        assert abs(E[0, 0] - np.cos(t)) < 1e-14
    spec = wl.CircuitSpec(1, 1, 0).add("RZ", (0,), [("x", 0)])
    assert abs(orc.forward(spec, np.array([[t]]), None)[0, 0] - 1.0) < 1e-14


def test_encoding_layer_gives_cos_x():
    n = 5
    spec = wl.CircuitSpec(n, n, 0)
    for q in range(n):
        spec.add("RY", (q,), [("x", q)])
    x = np.random.default_rng(1).uniform(-np.pi, np.pi, (7, n))
    assert np.allclose(orc.forward(spec, x, None), np.cos(x), atol=1e-14)


@pytest.mark.parametrize("k", [1, 2, 3])
def test_zero_angles_leave_ground_state(k):
    w_ = wl.config(k, dtype="c128", batch=2)[0]
    E, st = orc.forward(w_.spec, np.zeros_like(w_.x), np.zeros_like(w_.w), want_state=True)
    assert np.allclose(E, 1.0, atol=1e-13)
    assert np.allclose(np.abs(st[:, 0]), 1.0, atol=1e-13)


def test_zero_angles_config5_single_sample():
    w_ = wl.config(5, dtype="c128", batch=1)[0]
    E = orc.forward(w_.spec, np.zeros_like(w_.x), np.zeros_like(w_.w))
    assert np.allclose(E, 1.0, atol=1e-13)


def test_ghz():
    for n in (2, 3, 6):
        spec = wl.CircuitSpec(n, 0, 0).add("H", (0,))
        for q in range(n - 1):
            spec.add("CX", (q, q + 1))
        E, st = orc.forward(spec, None, None, want_state=True)
        assert np.allclose(E, 0.0, atol=1e-15)
        ref = np.zeros(1 << n, complex)
        ref[0] = ref[-1] = 1 / np.sqrt(2)
        assert np.allclose(st[0], ref, atol=1e-15)


def test_z_diagonal_layers_keep_cos_x():
    # config-2 structure with RX = RY = 0: only RZ and CZ after the encoding.
    w_ = wl.config(2, dtype="c128", batch=5)[0]
    w = w_.w.copy()
    w[0::3] = 0.0
    w[1::3] = 0.0
    assert np.allclose(orc.forward(w_.spec, w_.x, w), np.cos(w_.x), atol=1e-13)


def test_golden_fixtures():
    with open(os.path.join(HERE, "golden", "closed_forms.json")) as f:
        cases = json.load(f)["cases"]
    assert len(cases) >= 5
    for case in cases:
        spec = wl.CircuitSpec(case["n"], 0, 0)
        for g in case["gates"]:
            spec.add(g[0], g[1], [("c", float(eval(str(t), {"pi": np.pi}))) for t in g[2]])
        E, st = orc.forward(spec, None, None, want_state=True)
        assert np.allclose(E[0], case["expz"], atol=1e-12), case["name"]
        if "state" in case:
            ref = np.array([complex(a[0], a[1]) for a in case["state"]])
            assert np.allclose(st[0], ref, atol=1e-12), case["name"]


# ----------------------------------------------------------------------------- invariants

def inverse_spec(spec, xb, w):
    inv = wl.CircuitSpec(spec.n, 0, 0)
    for name, qubits, params in reversed(spec.gates):
        th = resolve(params, xb, w)
        if name in ("H", "X", "Y", "Z", "CX", "CZ", "SWAP"):
            inv.add(name, qubits)
        elif name == "S":
            for _ in range(3):
                inv.add("S", qubits)
        elif name == "T":
            for _ in range(7):
                inv.add("T", qubits)
        elif name == "SX":
            for _ in range(3):
                inv.add("SX", qubits)
        elif name == "U3":
            inv.add("U3", qubits, [("c", -th[0]), ("c", -th[2]), ("c", -th[1])])
        else:
            inv.add(name, qubits, [("c", -th[0])])
    return inv


def test_norm_and_inverse():
    for seed, n in [(21, 3), (22, 5), (23, 6)]:
        w_, psi0 = wl.small_random(seed, n, 60, batch=2, with_psi0=True)
        _, st = orc.forward(w_.spec, w_.x, w_.w, psi0=psi0, want_state=True)
        assert np.allclose(np.linalg.norm(st, axis=1), 1.0, atol=1e-12)
        for b in range(2):
            inv = inverse_spec(w_.spec, w_.x[b] if w_.spec.num_x else None, w_.w)
            _, back = orc.forward(inv, None, None, psi0=st[b][None], want_state=True)
            assert np.allclose(back[0], psi0[b], atol=1e-12)


def test_batch_rows_independent():
    w_, psi0 = wl.small_random(31, 5, 50, batch=4, with_psi0=True)
    E = orc.forward(w_.spec, w_.x, w_.w, psi0=psi0)
    for b in range(4):
        Eb = orc.forward(w_.spec, w_.x[b:b + 1], w_.w, psi0=psi0[b:b + 1])
        assert np.array_equal(E[b], Eb[0])


def test_qubit_relabelling_permutes_expectations():
    w_, _ = wl.small_random(41, 5, 50, batch=3)
    perm = [3, 0, 4, 1, 2]
    spec2 = wl.CircuitSpec(w_.spec.n, w_.spec.num_x, w_.spec.num_w)
    for name, qubits, params in w_.spec.gates:
        spec2.add(name, [perm[q] for q in qubits], params)
    E1 = orc.forward(w_.spec, w_.x, w_.w)
    E2 = orc.forward(spec2, w_.x, w_.w)
    assert np.allclose(E2[:, perm], E1, atol=1e-13)


# ----------------------------------------------------------------------------- gradients

def test_adjoint_sign_single_ry():
    for t in ANGLES:
        spec = wl.CircuitSpec(1, 1, 0).add("RY", (0,), [("x", 0)])
        dx, _ = orc.backward(spec, np.array([[t]]), None, np.array([[1.0]]))
        assert abs(dx[0, 0] + np.sin(t)) < 1e-14


def untie(spec, xb, w):
    """Give every angle occurrence its own x column (constants stay constant).
    Returns (spec, values, owner) with owner[j] = ('x'|'w', index) or None.
    CRZ(t) is expanded into RZ_t(t/2), CX, RZ_t(-t/2), CX, whose angles carry
    derivative factors +1/2 and -1/2."""
    out = wl.CircuitSpec(spec.n, 0, 0)
    vals, owner, factor = [], [], []

    def angle(kind, v, fac):
        col = len(vals)
        vals.append(v)
        owner.append(kind)
        factor.append(fac)
        return ("x", col)

    for name, qubits, params in spec.gates:
        th = resolve(params, xb, w)
        srcs = [(k, int(v)) if k != "c" else None for k, v in params]
        if name == "CRZ":
            c, t = qubits
            out.add("RZ", (t,), [angle(srcs[0], th[0] / 2, 0.5)])
            out.add("CX", (c, t))
            out.add("RZ", (t,), [angle(srcs[0], -th[0] / 2, -0.5)])
            out.add("CX", (c, t))
        else:
            out.add(name, qubits, [angle(srcs[p], th[p], 1.0) for p in range(len(params))])
    out.num_x = len(vals)
    return out, np.array(vals), owner, factor


def shift_gradient(spec, xb, w, gEb, psi0b=None):
    """dL/dx_b and dL/dw for one sample with the two-term shift rule."""
    uspec, vals, owner, factor = untie(spec, xb, w)
    dx = np.zeros(spec.num_x)
    dw = np.zeros(spec.num_w)
    p0 = None if psi0b is None else psi0b[None]
    for j in range(len(vals)):
        if owner[j] is None:
            continue
        vp, vm = vals.copy(), vals.copy()
        vp[j] += np.pi / 2
        vm[j] -= np.pi / 2
        Ep = orc.forward(uspec, vp[None], None, psi0=p0)[0]
        Em = orc.forward(uspec, vm[None], None, psi0=p0)[0]
        g = factor[j] * float(np.dot(gEb, (Ep - Em) / 2))
        kind, idx = owner[j]
        if kind == "x":
            dx[idx] += g
        else:
            dw[idx] += g
    return dx, dw


@pytest.mark.parametrize("seed,n", [(51, 1), (52, 2), (53, 3), (54, 4)])
def test_adjoint_matches_parameter_shift(seed, n):
    w_, psi0 = wl.small_random(seed, n, 30, batch=2, weight_fraction=0.5,
                               const_fraction=0.2, with_psi0=(seed % 2 == 0))
    dx, dw = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
    dw_ref = np.zeros_like(dw)
    for b in range(2):
        xb = w_.x[b] if w_.spec.num_x else np.zeros(0)
        sdx, sdw = shift_gradient(w_.spec, xb, w_.w, w_.gE[b], None if psi0 is None else psi0[b])
        assert np.allclose(dx[b], sdx, atol=1e-11)
        dw_ref += sdw
    assert np.allclose(dw, dw_ref, atol=1e-11)


def test_reuploaded_x_gradient_sums_occurrences():
    w_ = wl.config(3, dtype="c128", batch=1)[0]
    # shrink to 4 qubits / 2 layers with the same re-uploading structure
    spec = wl.layered(4, 2, ("RZ", "RY", "RZ"), "CX", reupload=True, ring_range=lambda l: (l % 3) + 1)
    rng = np.random.default_rng(2)
    x = rng.standard_normal((1, 4))
    w = rng.uniform(-np.pi, np.pi, spec.num_w)
    gE = rng.standard_normal((1, 4))
    dx, dw = orc.backward(spec, x, w, gE)
    sdx, sdw = shift_gradient(spec, x[0], w, gE[0])
    assert np.allclose(dx[0], sdx, atol=1e-12)
    assert np.allclose(dw, sdw, atol=1e-12)


def test_gradient_finite_difference_mean_objective():
    # the paper's objective: mean of <Z_i>  (gE = 1/n)
    w_ = wl.config(1, dtype="c128", batch=3)[0]
    n = w_.spec.n
    gE = np.full((3, n), 1.0 / n)
    dx, dw = orc.backward(w_.spec, w_.x, w_.w, gE)
    h = 1e-6
    L = lambda x, w: float(np.sum(gE * orc.forward(w_.spec, x, w)))
    for j in range(w_.spec.num_w):
        wp, wm = w_.w.copy(), w_.w.copy()
        wp[j] += h
        wm[j] -= h
        assert abs(dw[j] - (L(w_.x, wp) - L(w_.x, wm)) / (2 * h)) < 1e-8
    for b in range(3):
        for j in range(n):
            xp, xm = w_.x.copy(), w_.x.copy()
            xp[b, j] += h
            xm[b, j] -= h
            assert abs(dx[b, j] - (L(xp, w_.w) - L(xm, w_.w)) / (2 * h)) < 1e-8


@pytest.mark.parametrize("t", [1e3, -1e5, 131072.0, 1e6, -3e7])
def test_large_angle_rotations_closed_form(t):
    """Angles far outside [-pi, pi] (the range the GPU trig test covers): the
    oracle's RY, RX and RZ states equal the closed forms from the float64
    half-angle, and the adjoint gradient of <Z> after RY(t) RX(s) equals its
    closed form (d/dt cos t cos s = -sin t cos s)."""
    c, s = np.cos(t / 2), np.sin(t / 2)
    for name, want in (("RY", [c, s]), ("RX", [c, -1j * s]), ("RZ", [c - 1j * s, 0])):
        spec = wl.CircuitSpec(1, 1, 0).add(name, (0,), [("x", 0)])
        _, st = orc.forward(spec, np.array([[t]]), None, want_state=True)
        assert np.allclose(st[0], want, atol=1e-12, rtol=0), name
    u = 0.37 * t
    spec = wl.CircuitSpec(1, 2, 0).add("RY", (0,), [("x", 0)]).add("RX", (0,), [("x", 1)])
    x = np.array([[t, u]])
    assert abs(orc.forward(spec, x, None)[0, 0] - np.cos(t) * np.cos(u)) <= 1e-12
    dx, _ = orc.backward(spec, x, None, np.ones((1, 1)))
    assert np.allclose(dx[0], [-np.sin(t) * np.cos(u), -np.cos(t) * np.sin(u)], atol=1e-11, rtol=0)
