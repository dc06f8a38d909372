"""OpenQASM 2 front end (vqc_parse_qasm / vqc_compile_qasm), CPU only.

* a program lowers to exactly the gate records a hand-written gate list gives;
* the U3 special cases (u1, p, u2, sdg, tdg) reproduce their textbook matrices
  through the oracle's gate definitions, and a parsed program's oracle state
  equals the hand-written circuit's;
* broadcasts over whole registers, several registers, comments, expressions;
* errors: codes and the offending line;
* vqc_compile_qasm == vqc_compile on the parsed list (plan bytes), parameter
  counts inferred or checked.
"""
import numpy as np
import pytest

from oracle import oracle as orc
from paper_2607_11985_gb300 import binding as B
from paper_2607_11985_gb300 import workloads as wl


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_11985_gb300 import build
    build.build()


def records(arr, n):
    return [(g.op, g.q0, g.q1 if B.GATE_OPS[g.op] in ("CX", "CZ", "SWAP", "CRZ", "RZZ") else 0,
             tuple(g.pkind[:B.NUM_ANGLES.get(B.GATE_OPS[g.op], 0)]),
             tuple(g.pidx[k] if g.pkind[k] in (2, 3) else 0 for k in range(B.NUM_ANGLES.get(B.GATE_OPS[g.op], 0))),
             tuple(round(g.pconst[k], 12) if g.pkind[k] == 1 else 0.0
                   for k in range(B.NUM_ANGLES.get(B.GATE_OPS[g.op], 0))))
            for g in arr[:n]]


def to_spec(arr, n, nq, nx, nw):
    """The parsed records as a neutral circuit description (for the oracle)."""
    spec = wl.CircuitSpec(nq, nx, nw)
    kinds = {1: "c", 2: "x", 3: "w"}
    for g in arr[:n]:
        name = B.GATE_OPS[g.op]
        qs = (g.q0, g.q1) if name in ("CX", "CZ", "SWAP", "CRZ", "RZZ") else (g.q0,)
        ps = []
        for k in range(B.NUM_ANGLES.get(name, 0)):
            kind = kinds[g.pkind[k]]
            ps.append((kind, g.pconst[k] if kind == "c" else g.pidx[k]))
        spec.add(name, qs, ps)
    return spec


PROGRAM = """OPENQASM 2.0;
include "qelib1.inc";
// two registers: a[0..1] are qubits 0..1, b[0..2] are qubits 2..4
qreg a[2];
qreg b[3];
creg c[5];
h a[0];
ry(x[0]) a[1];
rz(w[2]) b[0];
u3(pi/2, -pi/4, 0.3) b[1];
rx(2*pi/3 - 0.5) b[2];
cx a[0], b[2];
cz a[1], b[0];
crz(x[1]) b[1], a[0];
rzz(w[0]) b[2], a[1];
swap a[0], b[1];
sx b[0];
s a[1]; t b[2]; y a[0]; z b[0]; x b[1];
barrier a, b;
measure a[0] -> c[0];
"""


def hand_spec():
    s = wl.CircuitSpec(5, 2, 3)
    s.add("H", (0,)).add("RY", (1,), [("x", 0)]).add("RZ", (2,), [("w", 2)])
    s.add("U3", (3,), [("c", np.pi / 2), ("c", -np.pi / 4), ("c", 0.3)])
    s.add("RX", (4,), [("c", 2 * np.pi / 3 - 0.5)])
    s.add("CX", (0, 4)).add("CZ", (1, 2)).add("CRZ", (3, 0), [("x", 1)])
    s.add("RZZ", (4, 1), [("w", 0)]).add("SWAP", (0, 3)).add("SX", (2,))
    s.add("S", (1,)).add("T", (4,)).add("Y", (0,)).add("Z", (2,)).add("X", (3,))
    return s


def test_program_lowers_to_the_hand_written_list():
    arr, n, nq, nx, nw = B.vqc_parse_qasm(PROGRAM)
    assert (nq, nx, nw) == (5, 2, 3)
    h = hand_spec()
    harr = B.gates_array(h)
    assert records(arr, n) == records(harr, len(h.gates))
    rng = np.random.default_rng(5)
    x = rng.uniform(-np.pi, np.pi, (2, 2))
    w = rng.uniform(-np.pi, np.pi, 3)
    _, s1 = orc.forward(to_spec(arr, n, nq, nx, nw), x, w, want_state=True)
    _, s2 = orc.forward(h, x, w, want_state=True)
    assert np.allclose(s1, s2, atol=1e-14)


@pytest.mark.parametrize("text,angles", [
    ("u1(0.7) q[0];", (0.0, 0.0, 0.7)),
    ("p(-1.1) q[0];", (0.0, 0.0, -1.1)),
    ("u2(0.2, 0.9) q[0];", (np.pi / 2, 0.2, 0.9)),
    ("sdg q[0];", (0.0, 0.0, -np.pi / 2)),
    ("tdg q[0];", (0.0, 0.0, -np.pi / 4)),
])
def test_u3_special_cases(text, angles):
    arr, n, nq, _, _ = B.vqc_parse_qasm("OPENQASM 2.0;\nqreg q[1];\n" + text + "\n")
    assert n == 1 and B.GATE_OPS[arr[0].op] == "U3"
    assert np.allclose([arr[0].pconst[k] for k in range(3)], angles)
    M = orc.gate_matrix("U3", np.array(angles))
    lam = angles[2]
    if text.startswith(("u1", "p(", "sdg", "tdg")):   # diag(1, e^{i lambda}) exactly
        assert np.allclose(M, np.diag([1, np.exp(1j * lam)]), atol=1e-15)
    else:                                             # u2 = [[1, -e^{il}], [e^{ip}, e^{i(p+l)}]] / sqrt 2
        p = angles[1]
        ref = np.array([[1, -np.exp(1j * lam)], [np.exp(1j * p), np.exp(1j * (p + lam))]]) / np.sqrt(2)
        assert np.allclose(M, ref, atol=1e-15)
    sd = {"sdg": np.diag([1, -1j]), "tdg": np.diag([1, np.exp(-1j * np.pi / 4)])}
    for k, v in sd.items():
        if text.startswith(k):
            assert np.allclose(M, v, atol=1e-15)


def test_broadcast_and_expressions():
    arr, n, nq, nx, nw = B.vqc_parse_qasm(
        "OPENQASM 2.0;\nqreg q[3];\nqreg r[3];\nh q;\ncx q, r;\nrz(-(1+2)^2/4 + sin(pi/6)) r[1];\nid q[0];\n")
    assert nq == 6 and n == 3 + 3 + 1
    assert [(g.op, g.q0) for g in arr[:3]] == [(B.GATE_CODE["H"], q) for q in range(3)]
    assert [(g.q0, g.q1) for g in arr[3:6]] == [(0, 3), (1, 4), (2, 5)]
    assert arr[6].pconst[0] == pytest.approx(-9 / 4 + 0.5)


@pytest.mark.parametrize("body,code,line", [
    ("ccx q[0], q[1], q[2];", 2, 3),
    ("rx(2*x[0]) q[0];", 1, 3),
    ("rx(x[0] + 1) q[0];", 1, 3),
    ("h q[3];", 3, 3),
    ("cx q[1], q[1];", 3, 3),
    ("gate g a { h a; }", 2, 3),
    ("reset q[0];", 2, 3),
    ("h q[0];\nrx(0.1, 0.2) q[1];", 1, 4),
    ("h z[0];", 3, 3),
    # only terminal measurements (Sec. 3 "Static Circuit Scope"): nothing acts
    # on a qubit after its measure
    ("creg c[3];\nmeasure q[0] -> c[0];\nh q[0];", 2, 5),
    ("creg c[3];\nmeasure q -> c;\ncx q[1], q[2];", 2, 5),
    ("creg c[3];\nmeasure q[2] -> c[2];\nbarrier q;", 2, 5),
    ("creg c[3];\nmeasure q[1] -> c[1];\nrzz(0.3) q[0], q[1];", 2, 5),
])
def test_errors_name_the_line(body, code, line):
    with pytest.raises(B.VQCError) as e:
        B.vqc_parse_qasm("OPENQASM 2.0;\nqreg q[3];\n" + body + "\n")
    assert e.value.status == code
    assert "line %d" % line in str(e.value)


def test_terminal_measurements_accepted():
    # measuring one qubit leaves the others free; measurements at the end pass
    arr, n, nq, nx, nw = B.vqc_parse_qasm(
        "OPENQASM 2.0;\nqreg q[3];\ncreg c[3];\nh q[0];\nmeasure q[0] -> c[0];\n"
        "cx q[1], q[2];\nbarrier q[1], q[2];\nmeasure q[1] -> c[1];\nmeasure q[2] -> c[2];\n")
    assert n == 2 and nq == 3
    assert [(g.op, g.q0, g.q1) for g in arr[:n]] == [(B.GATE_CODE["H"], 0, 0),
                                                     (B.GATE_CODE["CX"], 1, 2)]


def test_header_required():
    with pytest.raises(B.VQCError):
        B.vqc_parse_qasm("qreg q[2];\nh q[0];\n")
    with pytest.raises(B.VQCError):
        B.vqc_parse_qasm("OPENQASM 3.0;\nqreg q[2];\n")


def test_compile_qasm_matches_compile():
    arr, n, nq, nx, nw = B.vqc_parse_qasm(PROGRAM)
    p1 = B.vqc_compile_qasm(PROGRAM)
    p2 = B.vqc_compile(arr, n, nq, nx, nw, 0)
    assert B.vqc_plan_export(p1) == B.vqc_plan_export(p2)
    info = B.vqc_plan_info(B.vqc_compile_qasm(PROGRAM, 7, 9), 1)
    assert (info["num_x"], info["num_w"]) == (7, 9)
    with pytest.raises(B.VQCError) as e:
        B.vqc_compile_qasm(PROGRAM, 1, -1)
    assert e.value.status == 5
    B.vqc_free(p1)
    B.vqc_free(p2)
