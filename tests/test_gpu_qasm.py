"""GPU: circuits compiled from OpenQASM and the probabilities output, against
the oracle (complex64 / complex128 tolerances as in test_gpu_parity)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc  # noqa: E402
from paper_2607_11985_gb300 import binding as B  # noqa: E402
from paper_2607_11985_gb300 import workloads as wl  # noqa: E402
from tests.test_gpu_parity import TOL, dev, devc, maxerr  # noqa: E402
from tests.test_qasm_cpu import PROGRAM, to_spec  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def qasm_ring(n, layers):
    """A variational program: RY(x) encoding, RX(w) RZ(w) layers, CX ring."""
    lines = ["OPENQASM 2.0;", 'include "qelib1.inc";', "qreg q[%d];" % n]
    lines += ["ry(x[%d]) q[%d];" % (q, q) for q in range(n)]
    k = 0
    for _ in range(layers):
        for q in range(n):
            lines.append("rx(w[%d]) q[%d];" % (k, q))
            lines.append("rz(w[%d]) q[%d];" % (k + 1, q))
            k += 2
        lines += ["cx q[%d], q[%d];" % (q, (q + 1) % n) for q in range(n)]
    lines.append("u1(pi/8) q;")
    return "\n".join(lines) + "\n"


@pytest.mark.parametrize("dtype", ["c64", "c128", "c128df"])
@pytest.mark.parametrize("source", ["program", "ring6", "ring11"])
def test_qasm_forward_backward(dtype, source):
    from paper_2607_11985_gb300.circuit import Circuit
    text = {"program": PROGRAM, "ring6": qasm_ring(6, 3), "ring11": qasm_ring(11, 2)}[source]
    arr, n, nq, nx, nw = B.vqc_parse_qasm(text)
    spec = to_spec(arr, n, nq, nx, nw)
    rng = np.random.default_rng(77 + nq)
    Bt = 9
    x = wl._round(rng.uniform(-np.pi, np.pi, (Bt, nx)), dtype)
    w = wl._round(rng.uniform(-np.pi, np.pi, nw), dtype)
    gE = wl._round(rng.standard_normal((Bt, nq)), dtype)
    c = Circuit.from_qasm(text, dtype)
    assert (c.n, c.num_x, c.num_w) == (nq, nx, nw)
    E, st = c.forward(dev(x, dtype), dev(w, dtype), want_state=True)
    dx, dw = c.backward(dev(x, dtype), dev(w, dtype), dev(gE, dtype), psi_final=st)
    torch.cuda.synchronize()
    E_ref, st_ref = orc.forward(spec, x, w, want_state=True)
    dx_ref, dw_ref = orc.backward(spec, x, w, gE)
    tol = TOL[dtype]
    assert maxerr(E.cpu().numpy(), E_ref) <= tol["E"]
    assert maxerr(st.cpu().numpy(), st_ref) <= tol["state"]
    assert maxerr(dx.cpu().numpy(), dx_ref) <= tol["grad"]
    assert maxerr(dw.cpu().numpy(), dw_ref) <= tol["grad"]


@pytest.mark.parametrize("dtype", ["c64", "c128", "c128df"])
@pytest.mark.parametrize("force_hbm", [False, True])
def test_probabilities(monkeypatch, dtype, force_hbm):
    from paper_2607_11985_gb300.circuit import Circuit
    if force_hbm:
        monkeypatch.setenv("VQC_HBM_TILE_QUBITS", "6")
        monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
    w_, psi0 = wl.small_random(31, 9, 150, batch=5, dtype=dtype, with_psi0=True)
    c = Circuit(w_.spec, dtype)
    assert c.info(w_.batch)["fwd_path"] == (1 if force_hbm else 0)
    x = dev(w_.x, dtype) if w_.spec.num_x else None
    w = dev(w_.w, dtype) if w_.spec.num_w else None
    for p0 in (None, psi0):
        P = c.probabilities(x, w, psi0=devc(p0, dtype) if p0 is not None else None)
        torch.cuda.synchronize()
        _, st_ref = orc.forward(w_.spec, w_.x, w_.w, psi0=p0, want_state=True)
        P_ref = np.abs(st_ref) ** 2
        Pn = P.cpu().numpy()
        assert maxerr(Pn, P_ref) <= TOL[dtype]["state"]
        assert np.allclose(Pn.sum(1), 1.0, atol=1e-5 if dtype == "c64" else 1e-12)
