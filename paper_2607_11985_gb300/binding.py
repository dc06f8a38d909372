"""ctypes binding of the C ABI in ``include/vqc.h`` (argument marshalling only).

Every function here has the name of the C entry point it calls.  Pointers are
plain integers (device addresses, e.g. ``tensor.data_ptr()``) or ctypes
buffers; no torch type crosses the ABI.  Loading fails loudly when the
library has not been built: there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libvqc.so")

# vqc_gate_op
GATE_OPS = ["H", "X", "Y", "Z", "S", "T", "SX", "RX", "RY", "RZ", "U3",
            "CX", "CZ", "SWAP", "CRZ", "RZZ"]
GATE_CODE = {g: i for i, g in enumerate(GATE_OPS)}
NUM_ANGLES = {"RX": 1, "RY": 1, "RZ": 1, "CRZ": 1, "RZZ": 1, "U3": 3}
PKIND = {"c": 1, "x": 2, "w": 3}

VQC_C64, VQC_C128, VQC_C128_DF = 0, 1, 2
STATUS = {0: "VQC_OK", 1: "VQC_ERR_INVALID_ARG", 2: "VQC_ERR_UNSUPPORTED_GATE",
          3: "VQC_ERR_QUBIT_RANGE", 4: "VQC_ERR_TOO_MANY_QUBITS", 5: "VQC_ERR_PARAM_RANGE",
          6: "VQC_ERR_OUT_OF_MEMORY", 7: "VQC_ERR_CUDA", 8: "VQC_ERR_WORKSPACE",
          9: "VQC_ERR_DEVICE_CHECK", 10: "VQC_ERR_UNSUPPORTED"}


class vqc_gate(ctypes.Structure):
    _fields_ = [("op", ctypes.c_uint8), ("q0", ctypes.c_uint8), ("q1", ctypes.c_uint8),
                ("pkind", ctypes.c_uint8 * 3), ("reserved", ctypes.c_uint8 * 2),
                ("pidx", ctypes.c_int32 * 3), ("reserved2", ctypes.c_int32),
                ("pconst", ctypes.c_double * 3)]


class vqc_plan_stats(ctypes.Structure):
    _fields_ = [(name, ctypes.c_int32) for name in (
        "num_qubits", "num_x", "num_w", "dtype", "num_gates_in", "num_ops", "num_runs",
        "num_terms", "fwd_path", "bwd_path", "fwd_k", "bwd_k", "fwd_stages", "bwd_stages",
        "fwd_passes", "bwd_passes", "fwd_threads_per_sample", "bwd_threads_per_sample",
        "fwd_tile_qubits", "bwd_tile_qubits")] + [
        (name, ctypes.c_double) for name in (
            "fwd_flops_per_eval", "bwd_flops_per_eval", "recompute_flops_per_eval",
            "fwd_hbm_bytes_per_eval", "bwd_hbm_bytes_per_eval")]

    def as_dict(self):
        return {name: getattr(self, name) for name, _ in self._fields_}


assert ctypes.sizeof(vqc_gate) == 48


class VQCError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__("%s: %s" % (STATUS.get(status, status), msg))
        self.status = status


_lib = None

# C entry points and their signatures: (name, restype, argtypes)
_P, _I, _S = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
SIGNATURES = [
    ("vqc_compile", _I, [ctypes.POINTER(vqc_gate), _I, _I, _I, _I, _I, ctypes.POINTER(_P)]),
    ("vqc_free", None, [_P]),
    ("vqc_workspace_bytes", _S, [_P, _I, _I]),
    ("vqc_workspace_init", _I, [_P, _S, _P]),
    ("vqc_forward", _I, [_P, _I, _P, _P, _P, _P, _P, _P, _S, _P]),
    ("vqc_backward", _I, [_P, _I, _P, _P, _P, _P, _P, _P, _P, _P, _S, _P]),
    ("vqc_backward_noalloc", _I, [_P, _I, _P, _P, _P, _P, _P, _P, _P, _P]),
    ("vqc_stage_apply", _I, [_I, _I, _I, ctypes.POINTER(ctypes.c_double), _P, _P, _I, _P]),
    ("vqc_plan_info", _I, [_P, _I, ctypes.POINTER(vqc_plan_stats)]),
    ("vqc_plan_export", _I, [_P, _P, ctypes.POINTER(_S)]),
    ("vqc_sync_check", _I, [_P]),
    ("vqc_last_error", ctypes.c_char_p, []),
    ("vqc_abi_version", _I, []),
    ("vqc_probabilities", _I, [_P, _I, _P, _P, _P, _P, _P, _S, _P]),
    ("vqc_parse_qasm", _I, [ctypes.c_char_p, ctypes.POINTER(vqc_gate), ctypes.POINTER(_I),
                            ctypes.POINTER(_I), ctypes.POINTER(_I), ctypes.POINTER(_I)]),
    ("vqc_compile_qasm", _I, [ctypes.c_char_p, _I, _I, _I, ctypes.POINTER(_P)]),
    ("vqc_evaluate_host", _I, [_P, _I, _P, _P, _P, _P, _P, _P, _P]),
    ("vqc_host_direct", _I, [_I]),
    ("vqc_fma_peak", _I, [_I, ctypes.POINTER(ctypes.c_double)]),
    ("vqc_forward_backward", _I, [_P, _I, _P, _P, _P, _P, _P, _P, _P, _P, _S, _P]),
]


def lib():
    """Load libvqc.so (raises if it is missing: no CPU fallback exists)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libvqc.so is not built (run __graft_entry__.build() or "
                               "python -m paper_2607_11985_gb300.build)")
        L = ctypes.CDLL(LIB_PATH)
        for name, res, args in SIGNATURES:
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(status):
    if status != 0:
        raise VQCError(status, lib().vqc_last_error().decode(errors="replace"))


def gates_array(spec):
    """Marshal a neutral circuit description into a vqc_gate array."""
    arr = (vqc_gate * max(len(spec.gates), 1))()
    for g, (name, qubits, params) in enumerate(spec.gates):
        rec = arr[g]
        rec.op = GATE_CODE[name]
        rec.q0 = qubits[0]
        rec.q1 = qubits[1] if len(qubits) > 1 else 0
        for k, (kind, val) in enumerate(params):
            rec.pkind[k] = PKIND[kind]
            if kind == "c":
                rec.pconst[k] = float(val)
            else:
                rec.pidx[k] = int(val)
    return arr


def vqc_compile(gates, num_gates, num_qubits, num_x, num_w, dtype):
    plan = ctypes.c_void_p()
    _check(lib().vqc_compile(gates, num_gates, num_qubits, num_x, num_w, dtype, ctypes.byref(plan)))
    return plan.value


def vqc_parse_qasm(source):
    """(gates array, num_gates, num_qubits, num_x, num_w) of an OpenQASM 2 program."""
    src = source.encode() if isinstance(source, str) else source
    n, nq, nx, nw = _I(0), _I(0), _I(0), _I(0)
    _check(lib().vqc_parse_qasm(src, None, ctypes.byref(n), ctypes.byref(nq), ctypes.byref(nx),
                                ctypes.byref(nw)))
    arr = (vqc_gate * max(n.value, 1))()
    _check(lib().vqc_parse_qasm(src, arr, ctypes.byref(n), ctypes.byref(nq), ctypes.byref(nx),
                                ctypes.byref(nw)))
    return arr, n.value, nq.value, nx.value, nw.value


def vqc_compile_qasm(source, num_x=-1, num_w=-1, dtype=0):
    src = source.encode() if isinstance(source, str) else source
    plan = ctypes.c_void_p()
    _check(lib().vqc_compile_qasm(src, num_x, num_w, dtype, ctypes.byref(plan)))
    return plan.value


def vqc_free(plan):
    lib().vqc_free(plan)


def vqc_workspace_bytes(plan, batch, mode):
    return lib().vqc_workspace_bytes(plan, batch, mode)


def vqc_workspace_init(workspace, nbytes, stream):
    _check(lib().vqc_workspace_init(workspace, nbytes, stream))


def vqc_forward(plan, batch, x, w, psi0, expz_out, state_out, workspace, workspace_bytes, stream):
    _check(lib().vqc_forward(plan, batch, x, w, psi0, expz_out, state_out, workspace,
                             workspace_bytes, stream))


def vqc_probabilities(plan, batch, x, w, psi0, probs_out, workspace, workspace_bytes, stream):
    _check(lib().vqc_probabilities(plan, batch, x, w, psi0, probs_out, workspace, workspace_bytes,
                                   stream))


def vqc_backward(plan, batch, x, w, psi0, psi_final, grad_expz, grad_x, grad_w, workspace,
                 workspace_bytes, stream):
    _check(lib().vqc_backward(plan, batch, x, w, psi0, psi_final, grad_expz, grad_x, grad_w,
                              workspace, workspace_bytes, stream))


def vqc_forward_backward(plan, batch, x, w, psi0, grad_expz, expz_out, grad_x, grad_w, workspace,
                         workspace_bytes, stream):
    _check(lib().vqc_forward_backward(plan, batch, x, w, psi0, grad_expz, expz_out, grad_x, grad_w,
                                      workspace, workspace_bytes, stream))


def vqc_backward_noalloc(plan, batch, x, w, psi0, psi_final, grad_expz, grad_x, grad_w, stream):
    _check(lib().vqc_backward_noalloc(plan, batch, x, w, psi0, psi_final, grad_expz, grad_x,
                                      grad_w, stream))


def vqc_stage_apply(method, batch, num_qubits, factors, psi_in, psi_out, repeats, stream):
    """factors: 5 complex 2x2 matrices (any array of shape [5, 2, 2]), factor q
    on qubit q; psi_in / psi_out device addresses of complex64 states."""
    import numpy as np
    f = np.ascontiguousarray(np.stack([np.asarray(factors, np.complex128).real,
                                       np.asarray(factors, np.complex128).imag], -1).reshape(5, 8))
    _check(lib().vqc_stage_apply(method, batch, num_qubits,
                                 f.ctypes.data_as(ctypes.POINTER(ctypes.c_double)), psi_in, psi_out,
                                 repeats, stream))


def vqc_evaluate_host(plan, batch, x, w, grad_expz, expz_out, grad_x, grad_w, stream):
    """Host-memory evaluation: x, w, grad_expz, expz_out, grad_x, grad_w are
    host addresses (e.g. ``ndarray.ctypes.data``) or None."""
    _check(lib().vqc_evaluate_host(plan, batch, x, w, grad_expz, expz_out, grad_x, grad_w, stream))


def vqc_host_direct(device):
    return int(lib().vqc_host_direct(device))


def vqc_fma_peak(dtype):
    """Measured FMA rate (TFLOP/s) of the current device for dtype's arithmetic."""
    out = ctypes.c_double(0.0)
    _check(lib().vqc_fma_peak(dtype, ctypes.byref(out)))
    return out.value


def vqc_plan_info(plan, batch):
    st = vqc_plan_stats()
    _check(lib().vqc_plan_info(plan, batch, ctypes.byref(st)))
    return st.as_dict()


def vqc_plan_export(plan):
    n = ctypes.c_size_t(0)
    _check(lib().vqc_plan_export(plan, None, ctypes.byref(n)))
    buf = (ctypes.c_uint8 * n.value)()
    _check(lib().vqc_plan_export(plan, buf, ctypes.byref(n)))
    return bytes(buf)


def vqc_sync_check(stream):
    _check(lib().vqc_sync_check(stream))


def vqc_last_error():
    return lib().vqc_last_error().decode(errors="replace")


def vqc_abi_version():
    return lib().vqc_abi_version()
