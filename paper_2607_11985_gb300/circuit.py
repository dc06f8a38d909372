"""PyTorch-facing wrapper: compile once, then run batches through the C ABI.

``Circuit`` holds one compiled plan (paper, Alg. 1 compile phase: the gate
list is lowered once and the result cached) and calls ``vqc_forward`` /
``vqc_backward`` on torch CUDA tensors.  Torch supplies device memory and the
current stream only; every step of the sweep runs in the library's kernels.
``VQCFunction`` makes the forward differentiable with the adjoint backward.
"""
from __future__ import annotations

import torch

from . import binding as B

_DT = {"c64": (B.VQC_C64, torch.float32, torch.complex64),
       "c128": (B.VQC_C128, torch.float64, torch.complex128),
       # complex128 storage, double-float arithmetic on the FP32 units
       "c128df": (B.VQC_C128_DF, torch.float64, torch.complex128)}


def _ptr(t):
    return None if t is None else t.data_ptr()


class Circuit:
    """A compiled static circuit (see ``workloads.CircuitSpec`` for the format)."""

    def __init__(self, spec, dtype: str = "c64"):
        if dtype not in _DT:
            raise ValueError("dtype must be 'c64', 'c128' or 'c128df'")
        self.spec = spec
        self.n, self.num_x, self.num_w = int(spec.n), int(spec.num_x), int(spec.num_w)
        self.dtype = dtype
        self.code, self.real, self.cplx = _DT[dtype]
        self._gates = B.gates_array(spec)
        self.plan = B.vqc_compile(self._gates, len(spec.gates), self.n, self.num_x, self.num_w,
                                  self.code)
        self._ws = {}

    @classmethod
    def from_qasm(cls, source: str, dtype: str = "c64", num_x: int = -1, num_w: int = -1):
        """Compile an OpenQASM 2 program (gate set, parameter references x[i] /
        w[j]: see vqc_compile_qasm in include/vqc.h)."""
        if dtype not in _DT:
            raise ValueError("dtype must be 'c64', 'c128' or 'c128df'")
        self = cls.__new__(cls)
        self.spec = None
        self.dtype = dtype
        self.code, self.real, self.cplx = _DT[dtype]
        self._gates = None
        self.plan = B.vqc_compile_qasm(source, num_x, num_w, self.code)
        info = B.vqc_plan_info(self.plan, 1)
        self.n, self.num_x, self.num_w = info["num_qubits"], info["num_x"], info["num_w"]
        self._ws = {}
        return self

    def __del__(self):
        plan = getattr(self, "plan", None)
        if plan:
            try:
                torch.cuda.synchronize()
            except Exception:
                pass
            B.vqc_free(plan)
            self.plan = None

    # ------------------------------------------------------------------ helpers
    def info(self, batch: int = 1) -> dict:
        return B.vqc_plan_info(self.plan, batch)

    def export(self) -> bytes:
        return B.vqc_plan_export(self.plan)

    def _check(self, t, dtype, shape, name):
        if t is None:
            return None
        if not t.is_cuda or t.dtype != dtype or tuple(t.shape) != tuple(shape):
            raise ValueError("%s must be a CUDA %s tensor of shape %s (got %s %s %s)"
                             % (name, dtype, tuple(shape), t.device, t.dtype, tuple(t.shape)))
        return t.contiguous()

    def workspace(self, batch: int, mode: int, stream=None):
        nbytes = B.vqc_workspace_bytes(self.plan, batch, mode)
        if nbytes == 0:
            return None, 0
        stream = stream or torch.cuda.current_stream()
        key = (mode, stream.cuda_stream, torch.cuda.current_device())
        buf = self._ws.get(key)
        if buf is None or buf.numel() < nbytes:
            buf = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
            B.vqc_workspace_init(buf.data_ptr(), nbytes, stream.cuda_stream)
            self._ws[key] = buf
        return buf, buf.numel()

    # ------------------------------------------------------------------ calls
    def forward(self, x, w, psi0=None, want_state=False, out=None, state_out=None):
        """E [B, n] (and the final states [B, 2^n] when ``want_state``)."""
        batch = x.shape[0] if x is not None and x.dim() == 2 else (psi0.shape[0] if psi0 is not None else 1)
        x = self._check(x, self.real, (batch, self.num_x), "x") if self.num_x else None
        w = self._check(w, self.real, (self.num_w,), "w") if self.num_w else None
        psi0 = self._check(psi0, self.cplx, (batch, 1 << self.n), "psi0")
        E = out if out is not None else torch.empty(batch, self.n, dtype=self.real, device="cuda")
        st = state_out
        if want_state and st is None:
            st = torch.empty(batch, 1 << self.n, dtype=self.cplx, device="cuda")
        stream = torch.cuda.current_stream()
        ws, wsb = self.workspace(batch, 0, stream)
        B.vqc_forward(self.plan, batch, _ptr(x), _ptr(w), _ptr(psi0), _ptr(E), _ptr(st),
                      _ptr(ws), wsb, stream.cuda_stream)
        return (E, st) if want_state else E

    def probabilities(self, x, w, psi0=None, out=None):
        """|psi_b[k]|^2 of the final states, [B, 2^n] real."""
        batch = x.shape[0] if x is not None and x.dim() == 2 else (psi0.shape[0] if psi0 is not None else 1)
        x = self._check(x, self.real, (batch, self.num_x), "x") if self.num_x else None
        w = self._check(w, self.real, (self.num_w,), "w") if self.num_w else None
        psi0 = self._check(psi0, self.cplx, (batch, 1 << self.n), "psi0")
        P = out if out is not None else torch.empty(batch, 1 << self.n, dtype=self.real, device="cuda")
        stream = torch.cuda.current_stream()
        ws, wsb = self.workspace(batch, 2, stream)
        B.vqc_probabilities(self.plan, batch, _ptr(x), _ptr(w), _ptr(psi0), _ptr(P), _ptr(ws), wsb,
                            stream.cuda_stream)
        return P

    def backward(self, x, w, grad_expz, psi0=None, psi_final=None, need_x=True, need_w=True,
                 grad_x=None, grad_w=None):
        """(dL/dx [B, num_x], dL/dw [num_w]) for L = sum(grad_expz * E)."""
        batch = grad_expz.shape[0]
        x = self._check(x, self.real, (batch, self.num_x), "x") if self.num_x else None
        w = self._check(w, self.real, (self.num_w,), "w") if self.num_w else None
        gE = self._check(grad_expz, self.real, (batch, self.n), "grad_expz")
        psi0 = self._check(psi0, self.cplx, (batch, 1 << self.n), "psi0")
        psi_final = self._check(psi_final, self.cplx, (batch, 1 << self.n), "psi_final")
        dx = grad_x
        if dx is None and need_x and self.num_x:
            dx = torch.empty(batch, self.num_x, dtype=self.real, device="cuda")
        dw = grad_w
        if dw is None and need_w and self.num_w:
            dw = torch.empty(self.num_w, dtype=self.real, device="cuda")
        stream = torch.cuda.current_stream()
        ws, wsb = self.workspace(batch, 1, stream)
        B.vqc_backward(self.plan, batch, _ptr(x), _ptr(w), _ptr(psi0), _ptr(psi_final),
                       _ptr(gE), _ptr(dx), _ptr(dw), _ptr(ws), wsb, stream.cuda_stream)
        return dx, dw

    def forward_backward(self, x, w, grad_expz, psi0=None, out=None):
        """(E [B, n], dL/dx [B, num_x], dL/dw [num_w]) for L = sum(grad_expz * E)
        with grad_expz known up front (vqc_forward_backward: one launch on the
        resident path).  ``out`` = (E, dx, dw) preallocated CUDA tensors."""
        batch = grad_expz.shape[0]
        x = self._check(x, self.real, (batch, self.num_x), "x") if self.num_x else None
        w = self._check(w, self.real, (self.num_w,), "w") if self.num_w else None
        gE = self._check(grad_expz, self.real, (batch, self.n), "grad_expz")
        psi0 = self._check(psi0, self.cplx, (batch, 1 << self.n), "psi0")
        if out is None:
            E = torch.empty(batch, self.n, dtype=self.real, device="cuda")
            dx = torch.empty(batch, self.num_x, dtype=self.real, device="cuda") if self.num_x else None
            dw = torch.empty(self.num_w, dtype=self.real, device="cuda") if self.num_w else None
        else:
            E, dx, dw = out
        stream = torch.cuda.current_stream()
        ws, wsb = self.workspace(batch, 3, stream)
        B.vqc_forward_backward(self.plan, batch, _ptr(x), _ptr(w), _ptr(psi0), _ptr(gE), _ptr(E),
                               _ptr(dx), _ptr(dw), _ptr(ws), wsb, stream.cuda_stream)
        return E, dx, dw

    def evaluate_host(self, x, w, grad_expz=None, out=None, stream=None):
        """One evaluation from and to host memory (numpy arrays): E [B, n] and,
        given grad_expz [B, n], (dL/dx [B, num_x], dL/dw [num_w]) for
        L = sum(grad_expz * E).  One copy in, one copy out (vqc_evaluate_host).
        ``out`` = (E, dx, dw) preallocated host arrays to fill."""
        import numpy as np
        rdt = np.float32 if self.dtype == "c64" else np.float64

        def arr(a, shape, name):
            if a is None:
                return None
            if not isinstance(a, np.ndarray) or a.dtype != rdt or a.shape != tuple(shape) \
                    or not a.flags.c_contiguous:
                raise ValueError("%s must be a C-contiguous %s array of shape %s"
                                 % (name, np.dtype(rdt).name, tuple(shape)))
            return a

        batch = x.shape[0] if x is not None and self.num_x else \
            (grad_expz.shape[0] if grad_expz is not None else 1)
        x = arr(x, (batch, self.num_x), "x") if self.num_x else None
        w = arr(w, (self.num_w,), "w") if self.num_w else None
        gE = arr(grad_expz, (batch, self.n), "grad_expz")
        if out is None:
            E = np.empty((batch, self.n), rdt)
            dx = np.empty((batch, self.num_x), rdt) if gE is not None and self.num_x else None
            dw = np.empty((self.num_w,), rdt) if gE is not None and self.num_w else None
        else:
            E, dx, dw = out
            E = arr(E, (batch, self.n), "E")
            dx = arr(dx, (batch, self.num_x), "dx")
            dw = arr(dw, (self.num_w,), "dw")
        hp = lambda a: None if a is None else a.ctypes.data   # noqa: E731
        if stream is None:
            stream = torch.cuda.current_stream().cuda_stream
        B.vqc_evaluate_host(self.plan, batch, hp(x), hp(w), hp(gE), hp(E), hp(dx), hp(dw), stream)
        return E if gE is None else (E, dx, dw)

    def prepare_host(self, x, w, grad_expz=None, out=None, stream=None):
        """A prepared ``evaluate_host`` on fixed host arrays: the arrays are
        checked and their addresses taken once; each call of the returned
        ``HostStep`` evaluates whatever the arrays hold then (refill them in
        place between calls) and returns the output arrays."""
        return HostStep(self, x, w, grad_expz, out, stream)

    def __call__(self, x, w, psi0=None):
        return VQCFunction.apply(x, w, self, psi0)


class HostStep:
    """``Circuit.prepare_host``: one vqc_evaluate_host call on fixed host arrays."""

    def __init__(self, circuit, x, w, grad_expz=None, out=None, stream=None):
        import numpy as np
        c = circuit
        rdt = np.float32 if c.dtype == "c64" else np.float64
        batch = x.shape[0] if x is not None and c.num_x else \
            (grad_expz.shape[0] if grad_expz is not None else 1)

        def arr(a, shape, name):
            if a is None:
                return None
            if not isinstance(a, np.ndarray) or a.dtype != rdt or a.shape != tuple(shape) \
                    or not a.flags.c_contiguous:
                raise ValueError("%s must be a C-contiguous %s array of shape %s"
                                 % (name, np.dtype(rdt).name, tuple(shape)))
            return a

        x = arr(x, (batch, c.num_x), "x") if c.num_x else None
        w = arr(w, (c.num_w,), "w") if c.num_w else None
        gE = arr(grad_expz, (batch, c.n), "grad_expz")
        if out is None:
            out = (np.empty((batch, c.n), rdt),
                   np.empty((batch, c.num_x), rdt) if gE is not None and c.num_x else None,
                   np.empty((c.num_w,), rdt) if gE is not None and c.num_w else None)
        E, dx, dw = out
        E = arr(E, (batch, c.n), "E")
        dx = arr(dx, (batch, c.num_x), "dx")
        dw = arr(dw, (c.num_w,), "dw")
        self.circuit = c                              # keeps the plan alive
        self.arrays = (x, w, gE, E, dx, dw)           # keeps the addresses valid
        hp = lambda a: None if a is None else a.ctypes.data   # noqa: E731
        if stream is None:
            stream = torch.cuda.current_stream().cuda_stream
        self._args = (c.plan, batch) + tuple(hp(a) for a in self.arrays) + (stream,)
        self._fn = B.lib().vqc_evaluate_host
        self.result = E if gE is None else (E, dx, dw)

    def __call__(self):
        st = self._fn(*self._args)
        if st != 0:
            B._check(st)
        return self.result


class VQCFunction(torch.autograd.Function):
    """E = circuit(x, w); backward by the adjoint method from the saved final state."""

    @staticmethod
    def forward(ctx, x, w, circuit, psi0=None):
        E, st = circuit.forward(x.detach() if x is not None else None,
                                w.detach() if w is not None else None, psi0=psi0, want_state=True)
        ctx.circuit = circuit
        ctx.save_for_backward(x, w, psi0, st)
        return E

    @staticmethod
    def backward(ctx, gE):
        x, w, psi0, st = ctx.saved_tensors
        c = ctx.circuit
        need_x = x is not None and ctx.needs_input_grad[0]
        need_w = w is not None and ctx.needs_input_grad[1]
        dx, dw = c.backward(x, w, gE.contiguous(), psi0=psi0, psi_final=st,
                            need_x=need_x, need_w=need_w)
        return (dx if need_x else None), (dw if need_w else None), None, None
