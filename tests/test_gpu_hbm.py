"""GPU parity of the HBM-tiled pass path (states too large for one SM).

* the 16-qubit / 8-layer / batch-512 workload in complex64, complex128 and
  double-float complex128: the full batch against the batch-parallel oracle
  (E, every amplitude, dx, dw);
* small circuits forced onto the HBM path with 6-qubit tiles (many passes,
  tile-outer controls and phases), against the oracle, with and without psi0
  and the saved final state, ragged batches; the smallest circuits with the
  path forced (recomputing backward and the one-call forward+backward);
* cross-path agreement: the 12-qubit workload on the resident and HBM paths;
* the largest plan (24 qubits): forward against the oracle, backward against
  central differences of the complex128 forward;
* the thread-block-cluster forward (VQC_FORCE_PATH=cluster) at 14-16 qubits
  against the oracle and against the HBM passes, and on the 16-qubit workload.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc  # noqa: E402
from paper_2607_11985_gb300 import workloads as wl  # noqa: E402
from tests.test_gpu_parity import TOL, C, dev, devc, maxerr, oracle_full, report, run_bwd, run_fwd  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


_CFG5_REF = {}


def cfg5_reference(w_):
    """Oracle results of the 16-qubit workload's full batch (E, final states, dx,
    dw), computed once per input rounding: complex128 and double-float plans see
    the same float64 inputs."""
    key = "c64" if w_.dtype == "c64" else "c128"
    if key not in _CFG5_REF:
        _CFG5_REF[key] = oracle_full(w_, want_state=True)
    return _CFG5_REF[key]


@pytest.mark.parametrize("dtype", ["c64", "c128", "c128df"])
def test_config5_full_batch(dtype):
    """The 16-qubit / 8-layer workload at its full batch (512 rows, the launches
    the benchmark times): E, every final amplitude, dx and dw element by element
    against the oracle, from the saved final state and recomputing it."""
    w_ = wl.config(5, dtype=dtype)[0]
    c = C(w_.spec, dtype)
    info = c.info(w_.batch)
    # 16 qubits: forward and backward in HBM-tiled passes
    assert info["fwd_path"] == 1 and info["bwd_path"] == 1 and info["bwd_passes"] > 1
    ref = cfg5_reference(w_)
    E, st = run_fwd(c, w_)
    tol = TOL[dtype]
    errs = dict(E=maxerr(E, ref["E"]), state=maxerr(st, ref["st"]))
    dx, dw = run_bwd(c, w_, psi_final=devc(st, dtype))
    del st
    errs.update(dx=maxerr(dx, ref["dx"]), dw=maxerr(dw, ref["dw"]))
    dx2, dw2 = run_bwd(c, w_)
    errs.update(dx_recompute=maxerr(dx2, ref["dx"]), dw_recompute=maxerr(dw2, ref["dw"]))
    report(w_.name, **errs)
    for k, v in errs.items():
        bound = tol["E"] if k == "E" else tol["state"] if k == "state" else tol["grad"]
        assert v <= bound, (k, v)


SMALL = [(601, 8, 160), (602, 9, 200), (603, 10, 240), (604, 11, 200)]


@pytest.mark.parametrize("dtype", ["c64", "c128", "c128df"])
@pytest.mark.parametrize("seed,n,G", SMALL)
def test_forced_hbm_small_tiles(monkeypatch, seed, n, G, dtype):
    monkeypatch.setenv("VQC_HBM_TILE_QUBITS", "6")
    monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
    w_, psi0 = wl.small_random(seed, n, G, batch=21, dtype=dtype, with_psi0=(seed % 2 == 0))
    c = C(w_.spec, dtype)
    info = c.info(w_.batch)
    assert info["fwd_path"] == 1 and info["fwd_passes"] >= 2
    tol = TOL[dtype]
    E, st = run_fwd(c, w_, psi0)
    E_ref, st_ref = orc.forward(w_.spec, w_.x, w_.w, psi0=psi0, want_state=True)
    assert maxerr(E, E_ref) <= tol["E"]
    assert maxerr(st, st_ref) <= tol["state"]
    E2 = run_fwd(c, w_, psi0, want_state=False)          # last pass writes no state
    assert maxerr(E2, E_ref) <= tol["E"]
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
    dx, dw = run_bwd(c, w_, psi0)                          # recompute the final state
    assert maxerr(dx, dx_ref) <= tol["grad"] and maxerr(dw, dw_ref) <= tol["grad"]
    dx, dw = run_bwd(c, w_, psi0, psi_final=devc(st, dtype))
    assert maxerr(dx, dx_ref) <= tol["grad"] and maxerr(dw, dw_ref) <= tol["grad"]


@pytest.mark.parametrize("dtype,n", [("c64", 6), ("c128", 5), ("c64", 7), ("c128df", 5)])
def test_forced_hbm_smallest_circuits(monkeypatch, dtype, n):
    # at these sizes the backward's tile fits a pass kernel but the forward's
    # does not: the compiler then keeps both on the resident path, and the
    # recomputing backward and the one-call forward+backward still run
    monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
    w_, psi0 = wl.small_random(640 + n, n, 60, batch=5, dtype=dtype, with_psi0=True)
    c = C(w_.spec, dtype)
    info = c.info(w_.batch)
    assert (info["bwd_path"] == 1) <= (info["fwd_path"] == 1)
    tol = TOL[dtype]
    E_ref = orc.forward(w_.spec, w_.x, w_.w, psi0=psi0)
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
    dx, dw = run_bwd(c, w_, psi0)
    assert maxerr(dx, dx_ref) <= tol["grad"] and maxerr(dw, dw_ref) <= tol["grad"]
    x = dev(w_.x, dtype) if w_.spec.num_x else None
    w = dev(w_.w, dtype) if w_.spec.num_w else None
    E, dx, dw = c.forward_backward(x, w, dev(w_.gE, dtype), psi0=devc(psi0, dtype))
    torch.cuda.synchronize()
    assert maxerr(E.cpu().numpy(), E_ref) <= tol["E"]
    if dx is not None:
        assert maxerr(dx.cpu().numpy(), dx_ref) <= tol["grad"]
    if dw is not None:
        assert maxerr(dw.cpu().numpy(), dw_ref) <= tol["grad"]


def test_forced_hbm_ragged_batches(monkeypatch):
    monkeypatch.setenv("VQC_HBM_TILE_QUBITS", "7")
    monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
    w0, _ = wl.small_random(611, 9, 150, batch=1, dtype="c64")
    c = C(w0.spec, "c64")
    for B in (1, 3, 17, 64):
        wb, _ = wl.small_random(611, 9, 150, batch=B, dtype="c64")
        E = run_fwd(c, wb, want_state=False)
        assert maxerr(E, orc.forward(wb.spec, wb.x, wb.w)) <= 1e-4
        dx, dw = run_bwd(c, wb)
        dx_ref, dw_ref = orc.backward(wb.spec, wb.x, wb.w, wb.gE)
        assert maxerr(dx, dx_ref) <= 5e-4 and maxerr(dw, dw_ref) <= 5e-4


def test_resident_and_hbm_paths_agree(monkeypatch):
    w_ = wl.config(3, batch=256)[0]
    c = C(w_.spec, "c64")
    E1, st1 = run_fwd(c, w_)
    dx1, dw1 = run_bwd(c, w_)
    monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
    c2 = C(w_.spec, "c64")
    assert c2.info(w_.batch)["fwd_path"] == 1
    E2, st2 = run_fwd(c2, w_)
    dx2, dw2 = run_bwd(c2, w_)
    assert maxerr(E1, E2) <= 2e-5 and maxerr(st1, st2) <= 2e-5
    assert maxerr(dx1, dx2) <= 2e-4 and maxerr(dw1, dw2) <= 1e-3


def test_hbm_18_qubits_sampled():
    """18 qubits (2 MB complex64 state per sample, 32 tiles per sample per pass):
    E and dx of two rows against the oracle, dw of the whole batch of 3."""
    n = 18
    spec = wl.layered(n, 2, ("RX", "RY", "RZ"), "CX")
    rng = np.random.default_rng(1800)
    B = 3
    x = wl._round(rng.uniform(-np.pi, np.pi, (B, n)), "c64")
    w = wl._round(rng.uniform(-np.pi, np.pi, spec.num_w), "c64")
    gE = wl._round(rng.standard_normal((B, n)), "c64")
    w_ = wl.Workload("layered_n18", spec, B, x, w, gE, "c64", 1800)
    c = C(spec, "c64")
    info = c.info(B)
    assert info["fwd_path"] == 1 and info["bwd_path"] == 1
    E = run_fwd(c, w_, want_state=False)
    E_ref = orc.forward(spec, x, w)
    assert maxerr(E, E_ref) <= 1e-4
    dx, dw = run_bwd(c, w_)
    dx_ref, dw_ref = orc.backward(spec, x, w, gE)
    assert maxerr(dx, dx_ref) <= 5e-4 and maxerr(dw, dw_ref) <= 5e-4


def test_max_qubits_24():
    """The largest plan the ABI accepts (24 qubits: 128 MiB complex64 / 256 MiB
    complex128 per state).  Forward: E of one row against the oracle (complex64,
    batch of 2).  Backward, where the oracle would take minutes: the adjoint
    directional derivatives dL/dw . v and dL/dx . u match central differences
    of L = sum gE * E computed with the complex128 forward (a property that
    holds at any size; the forward itself is pinned above)."""
    n = 24
    spec = wl.layered(n, 1, ("RX", "RY", "RZ"), "CX")
    rng = np.random.default_rng(2400)
    x = wl._round(rng.uniform(-np.pi, np.pi, (2, n)), "c64")
    w = wl._round(rng.uniform(-np.pi, np.pi, spec.num_w), "c64")
    gE = wl._round(rng.standard_normal((2, n)), "c64")
    c = C(spec, "c64")
    assert c.info(2)["fwd_path"] == 1
    E = run_fwd(c, wl.Workload("n24", spec, 2, x, w, gE, "c64", 2400), want_state=False)
    assert maxerr(E[:1], orc.forward(spec, x[:1], w)) <= 1e-4
    assert np.all(np.abs(E) <= 1 + 1e-5)
    del c
    torch.cuda.empty_cache()

    c = C(spec, "c128")
    x1, g1 = x[:1], gE[:1]
    dx, dw = run_bwd(c, wl.Workload("n24", spec, 1, x1, w, g1, "c128", 2400))

    def loss(xv, wv):
        Ev = run_fwd(c, wl.Workload("n24", spec, 1, xv, wv, g1, "c128", 2400), want_state=False)
        return float(np.sum(g1 * Ev))

    v = rng.standard_normal(spec.num_w)
    u = rng.standard_normal((1, n))
    h = 1e-4
    fd_w = (loss(x1, w + h * v) - loss(x1, w - h * v)) / (2 * h)
    fd_x = (loss(x1 + h * u, w) - loss(x1 - h * u, w)) / (2 * h)
    assert abs(fd_w - float(dw @ v)) <= 1e-6 * max(1.0, abs(fd_w))
    assert abs(fd_x - float(np.sum(dx * u))) <= 1e-6 * max(1.0, abs(fd_x))


@pytest.mark.parametrize("dtype,n", [("c64", 15), ("c64", 16), ("c128", 14), ("c128", 15), ("c128", 16),
                                     ("c128df", 14), ("c128df", 16)])
def test_cluster_forward(monkeypatch, dtype, n):
    """Forward with the state spread over a thread-block cluster (2, 4 or 8 CTAs):
    E and the final states against the oracle, from |0...0> and from a given
    psi0, with and without the state output; the same batch through the
    HBM-tiled passes agrees."""
    spec = wl.layered(n, 2, ("RX", "RY", "RZ"), "CX", ring_range=lambda l: 2 * l + 1)
    rng = np.random.default_rng(1500 + n)
    B = 3
    x = wl._round(rng.uniform(-np.pi, np.pi, (B, n)), dtype)
    w = wl._round(rng.uniform(-np.pi, np.pi, spec.num_w), dtype)
    gE = wl._round(rng.standard_normal((B, n)), dtype)
    z = rng.standard_normal((B, 1 << n)) + 1j * rng.standard_normal((B, 1 << n))
    z /= np.linalg.norm(z, axis=1, keepdims=True)
    if dtype == "c64":
        z = z.astype(np.complex64).astype(np.complex128)
    w_ = wl.Workload("cluster_n%d" % n, spec, B, x, w, gE, dtype, 1500 + n)
    c = C(spec, dtype)
    # default: the cluster for 2-CTA clusters (complex64 15 qubits, complex128 14), else the passes
    two_cta = (dtype, n) in (("c64", 15), ("c128", 14), ("c128df", 14))
    assert c.info(B)["fwd_path"] == (2 if two_cta else 1)
    monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
    assert c.info(B)["fwd_path"] == 2
    tol = TOL[dtype]
    for psi0 in (None, z):
        E_ref, st_ref = orc.forward(spec, x, w, psi0=psi0, want_state=True)
        E, st = run_fwd(c, w_, psi0)
        assert maxerr(E, E_ref) <= tol["E"] and maxerr(st, st_ref) <= tol["state"]
        E2 = run_fwd(c, w_, psi0, want_state=False)
        assert maxerr(E2, E_ref) <= tol["E"]
        monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
        E3, st3 = run_fwd(c, w_, psi0)
        monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
        assert maxerr(E3, E) <= tol["E"] and maxerr(st3, st) <= tol["state"]


@pytest.mark.parametrize("dtype", ["c64", "c128", "c128df"])
def test_config5_cluster_forward(monkeypatch, dtype):
    """The 16-qubit, 8-layer batch through the cluster forward: sampled rows
    against the oracle."""
    monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
    w_ = wl.config(5, dtype=dtype)[0]
    c = C(w_.spec, dtype)
    assert c.info(w_.batch)["fwd_path"] == 2
    E, st = run_fwd(c, w_)
    rows = [0, 257, w_.batch - 1]
    E_ref, st_ref = orc.forward(w_.spec, w_.x[rows], w_.w, want_state=True)
    assert maxerr(E[rows], E_ref) <= TOL[dtype]["E"]
    assert maxerr(st[rows], st_ref) <= TOL[dtype]["state"]
