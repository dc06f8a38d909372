"""GPU: vqc_evaluate_host (inputs and outputs in host memory, one copy each
way) against the oracle and against the device-memory calls.

* the 8-qubit / 4-layer workload (full batch 1024 and a ragged 37-row slice):
  E, dL/dx, dL/dw equal to vqc_forward + vqc_backward on the same inputs (same
  kernels, same order: bit-identical) and within tolerance of the oracle;
* forward only (no gE), complex128, a batch that grows and shrinks (the arena
  is reallocated and its workspaces re-initialised), batch 0;
* a 16-qubit circuit on the HBM-tiled path (both workspaces in the arena);
* a 14-qubit circuit whose backward runs on thread-block clusters;
* argument errors.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc  # noqa: E402
from paper_2607_11985_gb300 import binding as B  # noqa: E402
from paper_2607_11985_gb300 import workloads as wl  # noqa: E402
from tests.test_gpu_parity import TOL, C, maxerr, run_bwd, run_fwd  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def rows(w_, idx):
    return wl.Workload(w_.name, w_.spec, len(idx), w_.x[idx], w_.w, w_.gE[idx], w_.dtype, w_.seed)


def host(a, dtype):
    return np.ascontiguousarray(a, dtype=np.float32 if dtype == "c64" else np.float64)


@pytest.fixture(params=["direct", "staged"])
def access(request, monkeypatch):
    """Both transfer modes: kernels on the host arrays in place (where the
    device supports it) and the pinned staging copies."""
    if request.param == "staged":
        monkeypatch.setenv("VQC_HOST_DIRECT", "0")
        assert B.vqc_host_direct(0) == 0
    elif not B.vqc_host_direct(0):
        pytest.skip("this device does not access pageable host memory")
    return request.param


@pytest.mark.parametrize("batch", [1024, 37])
def test_matches_device_calls_and_oracle(access, batch):
    w_ = wl.config(2)[0]
    if batch != w_.batch:
        w_ = rows(w_, np.arange(batch) * 7 % w_.batch)
    c = C(w_.spec, "c64")
    E, dx, dw = c.evaluate_host(host(w_.x, "c64"), host(w_.w, "c64"), host(w_.gE, "c64"))
    E_d, st = run_fwd(c, w_)
    dx_d, dw_d = run_bwd(c, w_, psi_final=torch.tensor(st, device="cuda"))
    assert np.array_equal(E, E_d) and np.array_equal(dx, dx_d) and np.array_equal(dw, dw_d)
    sub = rows(w_, [0, batch // 2, batch - 1])
    E_ref = orc.forward(w_.spec, sub.x, sub.w)
    dx_ref, _ = orc.backward(w_.spec, sub.x, sub.w, sub.gE)
    assert maxerr(E[[0, batch // 2, batch - 1]], E_ref) <= TOL["c64"]["E"]
    assert maxerr(dx[[0, batch // 2, batch - 1]], dx_ref) <= TOL["c64"]["grad"]
    if batch == 37:
        _, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE)
        assert maxerr(dw, dw_ref) <= TOL["c64"]["grad"]


@pytest.mark.parametrize("dt", ["c128", "c128df"])
def test_forward_only_c128_and_batch_changes(access, dt):
    w_ = wl.config(1, dtype=dt)[0]
    c = C(w_.spec, dt)
    for b in (5, 64, 3, 64):
        sub = rows(w_, np.arange(b) % w_.batch)
        E = c.evaluate_host(host(sub.x, dt), host(sub.w, dt))
        assert E.shape == (b, w_.spec.n)
        assert maxerr(E, orc.forward(w_.spec, sub.x, sub.w)) <= TOL[dt]["E"]
        E2, dx, dw = c.evaluate_host(host(sub.x, dt), host(sub.w, dt), host(sub.gE, dt))
        # the one-call forward+backward writes the same E as the forward alone
        # (complex128: bit for bit; double-float: the fused kernel's own forward)
        assert maxerr(E, E2) <= (0.0 if dt == "c128" else 1e-13)
        dx_ref, dw_ref = orc.backward(w_.spec, sub.x, sub.w, sub.gE)
        assert maxerr(dx, dx_ref) <= TOL[dt]["grad"] and maxerr(dw, dw_ref) <= TOL[dt]["grad"]
    # batch 0: nothing to evaluate, dw is zero
    dw0 = np.full(w_.spec.num_w, 7.0)
    B.vqc_evaluate_host(c.plan, 0, None, host(w_.w, "c128").ctypes.data,
                        host(w_.gE[:1], "c128").ctypes.data, np.zeros((1, w_.spec.n)).ctypes.data,
                        None, dw0.ctypes.data, torch.cuda.current_stream().cuda_stream)
    assert not dw0.any()


def test_hbm_path_circuit(access):
    n = 16
    spec = wl.layered(n, 2, ("RX", "RY", "RZ"), "CX", ring_range=lambda l: 2 * l + 1)
    rng = np.random.default_rng(1616)
    b = 3
    x = rng.uniform(-np.pi, np.pi, (b, n)).astype(np.float32)
    w = rng.uniform(-np.pi, np.pi, spec.num_w).astype(np.float32)
    gE = rng.standard_normal((b, n)).astype(np.float32)
    c = C(spec, "c64")
    info = c.info(b)
    assert info["fwd_path"] == 1 and info["bwd_path"] == 1
    E, dx, dw = c.evaluate_host(x, w, gE)
    w_ = wl.Workload("hbm16", spec, b, x.astype(np.float64), w.astype(np.float64),
                     gE.astype(np.float64), "c64", 1616)
    E_d, st = run_fwd(c, w_)
    dx_d, dw_d = run_bwd(c, w_, psi_final=torch.tensor(st, device="cuda"))
    assert np.array_equal(E, E_d) and np.array_equal(dx, dx_d) and np.array_equal(dw, dw_d)
    E_ref = orc.forward(spec, x.astype(np.float64), w.astype(np.float64))
    assert maxerr(E, E_ref) <= TOL["c64"]["E"]


def test_cluster_backward_circuit(access):
    """14 qubits complex64: resident forward, backward on 2-CTA thread-block
    clusters (the final states in the arena's workspace); three calls, so the
    later ones replay the captured graph."""
    n = 14
    spec = wl.layered(n, 2, ("RX", "RY", "RZ"), "CX", ring_range=lambda l: 2 * l + 1)
    rng = np.random.default_rng(1414)
    b = 5
    x = rng.uniform(-np.pi, np.pi, (b, n)).astype(np.float32)
    w = rng.uniform(-np.pi, np.pi, spec.num_w).astype(np.float32)
    gE = rng.standard_normal((b, n)).astype(np.float32)
    c = C(spec, "c64")
    info = c.info(b)
    assert info["fwd_path"] == 0 and info["bwd_path"] == 2
    w_ = wl.Workload("cluster14", spec, b, x.astype(np.float64), w.astype(np.float64),
                     gE.astype(np.float64), "c64", 1414)
    E_d, st = run_fwd(c, w_)
    dx_d, dw_d = run_bwd(c, w_, psi_final=torch.tensor(st, device="cuda"))
    for _ in range(3):
        E, dx, dw = c.evaluate_host(x, w, gE)
        assert np.array_equal(E, E_d) and np.array_equal(dx, dx_d) and np.array_equal(dw, dw_d)
    dx_ref, dw_ref = orc.backward(spec, x.astype(np.float64), w.astype(np.float64), gE.astype(np.float64))
    assert maxerr(dx, dx_ref) <= TOL["c64"]["grad"] and maxerr(dw, dw_ref) <= TOL["c64"]["grad"]


def test_argument_errors():
    w_ = wl.config(2, batch=4)[0]
    c = C(w_.spec, "c64")
    s = torch.cuda.current_stream().cuda_stream
    E = np.zeros((4, w_.spec.n), np.float32)
    w = host(w_.w, "c64")
    with pytest.raises(B.VQCError) as e:   # x missing although the circuit uses x
        B.vqc_evaluate_host(c.plan, 4, None, w.ctypes.data, None, E.ctypes.data, None, None, s)
    assert e.value.status == 1
    x = host(w_.x, "c64")
    with pytest.raises(B.VQCError) as e:   # no output
        B.vqc_evaluate_host(c.plan, 4, x.ctypes.data, w.ctypes.data, None, None, None, None, s)
    assert e.value.status == 1
    with pytest.raises(ValueError):        # wrong dtype at the Python layer
        c.evaluate_host(w_.x, w)


def test_graph_replay_sees_new_inputs(access, monkeypatch):
    """From the second call of one shape on, the device work is a replayed CUDA
    graph: it must read each call's inputs (new arrays, or new contents of the
    same arrays), and agree bit for bit with plain launches (VQC_HOST_GRAPH=0)."""
    w_ = wl.config(2, batch=64)[0]
    c = C(w_.spec, "c64")
    x1, w1, g1 = host(w_.x, "c64"), host(w_.w, "c64"), host(w_.gE, "c64")
    x2 = np.ascontiguousarray(x1[::-1])
    w2 = np.ascontiguousarray(w1 * 0.5)
    outs = tuple(np.empty_like(a) for a in (np.empty((64, w_.spec.n), np.float32), x1, w1))
    first = [a.copy() for a in c.evaluate_host(x1, w1, g1, out=outs)]
    again = [a.copy() for a in c.evaluate_host(x1, w1, g1, out=outs)]   # captured here
    xs, ws_ = x1.copy(), w1.copy()
    x1[:] = x2
    w1[:] = w2
    other = [a.copy() for a in c.evaluate_host(x1, w1, g1, out=outs)]   # replayed, new contents
    x1[:] = xs
    w1[:] = ws_
    for a, b in zip(first, again):
        assert np.array_equal(a, b)
    monkeypatch.setenv("VQC_HOST_GRAPH", "0")
    c2 = C(w_.spec, "c64")
    direct = c2.evaluate_host(x2, w2, g1)
    for a, b in zip(other, direct):
        assert np.array_equal(a, b)
    sub = wl.Workload(w_.name, w_.spec, 64, x2.astype(np.float64), w2.astype(np.float64),
                      g1.astype(np.float64), "c64", w_.seed)
    assert maxerr(other[0], orc.forward(w_.spec, sub.x, sub.w)) <= TOL["c64"]["E"]


def test_prepared_host_step_refills(access):
    """Circuit.prepare_host: the arrays are bound once; refilling them in place
    between calls gives the results evaluate_host gives on the new contents."""
    w_ = wl.config(2, batch=64)[0]
    c = C(w_.spec, "c64")
    x, w, g = host(w_.x, "c64"), host(w_.w, "c64"), host(w_.gE, "c64")
    step = c.prepare_host(x, w, g)
    E1, dx1, dw1 = [a.copy() for a in step()]
    ref1 = c.evaluate_host(host(w_.x, "c64"), host(w_.w, "c64"), host(w_.gE, "c64"))
    x[:] = x[::-1].copy()
    g *= -0.5
    E2, dx2, dw2 = [a.copy() for a in step()]
    ref2 = c.evaluate_host(x.copy(), w.copy(), g.copy())
    for a, b in zip((E1, dx1, dw1, E2, dx2, dw2), tuple(ref1) + tuple(ref2)):
        assert np.array_equal(a, b)
    assert not np.array_equal(E1, E2)
    with pytest.raises(ValueError):
        c.prepare_host(w_.x, w, g)          # float64 x for a complex64 plan
