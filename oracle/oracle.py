"""TEST INFRASTRUCTURE ONLY: ctypes wrapper around the plain C complex128 oracle.

Only the test suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg may import this module.  It shares no code with the CUDA engine: it
marshals the neutral circuit description (gate names, qubits, parameter sources)
produced by the seeded input generators into the oracle's own array format.

What the oracle computes is stated in ``vqc_oracle.c`` (paper, Alg. 1 and Sec. 3).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "vqc_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

# Oracle opcode numbering (must match the enum in vqc_oracle.c).
OPS = ["H", "X", "Y", "Z", "S", "T", "SX", "RX", "RY", "RZ", "U3",
       "CX", "CZ", "SWAP", "CRZ", "RZZ"]
OPCODE = {name: i for i, name in enumerate(OPS)}
NPARAMS = {"RX": 1, "RY": 1, "RZ": 1, "CRZ": 1, "RZZ": 1, "U3": 3}
TWO_QUBIT = {"CX", "CZ", "SWAP", "CRZ", "RZZ"}
_KIND = {"c": 1, "x": 2, "w": 3}

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with the host C compiler (gcc, plain C11, no ISA flags)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp.%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SRC,
                               "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i = ctypes.c_int
            lib.oracle_forward.argtypes = [i, i, P, P, P, P, P, P, i, i, i, P, P, P, P, P]
            lib.oracle_forward.restype = i
            lib.oracle_backward.argtypes = [i, i, P, P, P, P, P, P, i, i, i, P, P, P, P, P, P]
            lib.oracle_backward.restype = i
            lib.oracle_gate_matrix.argtypes = [i, P, P]
            lib.oracle_gate_matrix.restype = i
            lib.oracle_gate_matrix_deriv.argtypes = [i, P, i, P]
            lib.oracle_gate_matrix_deriv.restype = i
            lib.oracle_num_ops.restype = i
            assert lib.oracle_num_ops() == len(OPS)
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


class _Arrays:
    """The oracle's own array form of a circuit."""

    def __init__(self, spec):
        G = len(spec.gates)
        self.n, self.G = int(spec.n), G
        self.Px, self.Pw = int(spec.num_x), int(spec.num_w)
        self.op = np.zeros(G, np.int32)
        self.q0 = np.zeros(G, np.int32)
        self.q1 = np.zeros(G, np.int32)
        self.pkind = np.zeros(G * 3, np.int32)
        self.pidx = np.zeros(G * 3, np.int32)
        self.pconst = np.zeros(G * 3, np.float64)
        for g, (name, qubits, params) in enumerate(spec.gates):
            self.op[g] = OPCODE[name]
            self.q0[g] = qubits[0]
            self.q1[g] = qubits[1] if len(qubits) > 1 else 0
            for p, (kind, val) in enumerate(params):
                self.pkind[g * 3 + p] = _KIND[kind]
                if kind == "c":
                    self.pconst[g * 3 + p] = float(val)
                else:
                    self.pidx[g * 3 + p] = int(val)

    def args(self):
        return (self.n, self.G, _ptr(self.op), _ptr(self.q0), _ptr(self.q1),
                _ptr(self.pkind), _ptr(self.pidx), _ptr(self.pconst), self.Px, self.Pw)


def _f64(a, shape):
    if a is None:
        return None
    a = np.ascontiguousarray(np.asarray(a, dtype=np.float64))
    return a.reshape(shape)


def _psi0(psi0, B, dim):
    if psi0 is None:
        return None
    p = np.asarray(psi0)
    if np.iscomplexobj(p):
        p = np.stack([p.real, p.imag], axis=-1)
    return _f64(p, (B, dim, 2))


def forward(spec, x, w, psi0=None, want_state=False):
    """E [B, n] (float64) and, if asked, the final states [B, 2^n] (complex128)."""
    lib = _load()
    a = _Arrays(spec)
    dim = 1 << a.n
    x = _f64(x, (-1, a.Px)) if a.Px else None
    B = x.shape[0] if x is not None else (np.asarray(psi0).shape[0] if psi0 is not None else 1)
    w = _f64(w, (a.Pw,)) if a.Pw else np.zeros(1)
    p0 = _psi0(psi0, B, dim)
    E = np.zeros((B, a.n), np.float64)
    st = np.zeros((B, dim, 2), np.float64) if want_state else None
    rc = lib.oracle_forward(*a.args(), B, _ptr(x), _ptr(w), _ptr(p0), _ptr(E), _ptr(st))
    if rc:
        raise ValueError("oracle_forward rejected the circuit (code %d)" % rc)
    if want_state:
        return E, st[..., 0] + 1j * st[..., 1]
    return E


def backward(spec, x, w, gE, psi0=None):
    """(dx [B, Px], dw [Pw]) of L = sum gE * E, float64."""
    lib = _load()
    a = _Arrays(spec)
    dim = 1 << a.n
    gE = _f64(gE, (-1, a.n))
    B = gE.shape[0]
    x = _f64(x, (B, a.Px)) if a.Px else None
    w = _f64(w, (a.Pw,)) if a.Pw else np.zeros(1)
    p0 = _psi0(psi0, B, dim)
    dx = np.zeros((B, max(a.Px, 1)), np.float64)
    dw = np.zeros(max(a.Pw, 1), np.float64)
    rc = lib.oracle_backward(*a.args(), B, _ptr(x), _ptr(w), _ptr(p0), _ptr(gE),
                             _ptr(dx), _ptr(dw))
    if rc:
        raise ValueError("oracle_backward rejected the circuit (code %d)" % rc)
    return dx[:, :a.Px], dw[:a.Pw]


def gate_matrix(name, theta=(0.0, 0.0, 0.0)):
    """Dense matrix of one gate (2x2 or 4x4; 4x4 local index s = b0 + 2*b1)."""
    lib = _load()
    th = np.zeros(3, np.float64)
    th[:len(theta)] = theta
    out = np.zeros(32, np.float64)
    d = lib.oracle_gate_matrix(OPCODE[name], _ptr(th), _ptr(out))
    m = out[:2 * d * d:2] + 1j * out[1:2 * d * d:2]
    return m.reshape(d, d)


def gate_matrix_deriv(name, theta, p):
    lib = _load()
    th = np.zeros(3, np.float64)
    th[:len(theta)] = theta
    out = np.zeros(32, np.float64)
    d = lib.oracle_gate_matrix_deriv(OPCODE[name], _ptr(th), p, _ptr(out))
    if d == 0:
        raise ValueError("gate %s has no parameter %d" % (name, p))
    m = out[:2 * d * d:2] + 1j * out[1:2 * d * d:2]
    return m.reshape(d, d)


# ------------------------------------------------------------------ batch-parallel calls
def _row_chunks(B, workers):
    """Contiguous row ranges, about four per worker thread."""
    parts = max(1, min(B, 4 * workers))
    edges = np.linspace(0, B, parts + 1).astype(int)
    return [(int(a), int(b)) for a, b in zip(edges[:-1], edges[1:]) if b > a]


def _pool_map(fn, items, workers):
    import concurrent.futures as cf
    _load()   # build and load the library before the threads start
    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        return list(ex.map(fn, items))


def forward_parallel(spec, x, w, psi0=None, want_state=False, workers=None):
    """forward() over row chunks on a thread pool: samples are independent and the
    C oracle releases the GIL during each call, so every host core works on its
    own rows.  Same results as forward() on the whole batch."""
    workers = workers or os.cpu_count() or 1
    Px = int(spec.num_x)
    x = None if not Px else np.asarray(x)
    B = x.shape[0] if x is not None else np.asarray(psi0).shape[0]

    def one(rg):
        a, b = rg
        return forward(spec, None if x is None else x[a:b], w,
                       psi0=None if psi0 is None else np.asarray(psi0)[a:b], want_state=want_state)

    outs = _pool_map(one, _row_chunks(B, workers), workers)
    if want_state:
        return (np.concatenate([o[0] for o in outs]), np.concatenate([o[1] for o in outs]))
    return np.concatenate(outs)


def backward_parallel(spec, x, w, gE, psi0=None, workers=None):
    """backward() over row chunks on a thread pool: dx rows are independent and
    dw is the sum of the chunks' dw (in chunk order, float64)."""
    workers = workers or os.cpu_count() or 1
    gE = np.asarray(gE)
    B = gE.shape[0]
    Px = int(spec.num_x)

    def one(rg):
        a, b = rg
        return backward(spec, None if not Px else np.asarray(x)[a:b], w, gE[a:b],
                        psi0=None if psi0 is None else np.asarray(psi0)[a:b])

    outs = _pool_map(one, _row_chunks(B, workers), workers)
    dx = np.concatenate([o[0] for o in outs])
    dw = np.zeros(int(spec.num_w), np.float64)
    for o in outs:
        dw += o[1]
    return dx, dw
