"""vqc_backward_noalloc against vqc_backward, through the C ABI (GPU).

vqc_backward_noalloc serves callers that cannot allocate device memory (a
plugin whose host application owns every device allocation, a real-time loop
that cannot afford cudaMalloc's latency and implicit synchronisation, code under
a fixed device-memory budget): it takes no workspace and uses scratch built
into the library instead.  It runs the same kernels with the same fixed-order
reductions as the workspace entry point, so its gradients must be bit-identical
to those of vqc_backward, on two calls in a row (the second call finds the first
call's leftovers in the shared scratch): on the resident path, on the
HBM-tiled passes (15 qubits) and on the thread-block-cluster backward (14
qubits), from a saved final state and recomputing it.  A
batch whose scratch need exceeds the built-in size must be rejected with
VQC_ERR_WORKSPACE.

This file is collected last so that a run stopping at its first failure has
already run every other test; it also passes on its own in a fresh process.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2607_11985_gb300 import workloads as wl  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _inputs(w_, real=torch.float32):
    f = lambda a: torch.tensor(np.asarray(a), dtype=real, device="cuda")
    return f(w_.x), f(w_.w), f(w_.gE)


def _ptr(t):
    return None if t is None else t.data_ptr()


def _workspace_backward(B, c, x, w, gE, st):
    dx = torch.empty_like(x)
    dw = torch.empty_like(w)
    stream = torch.cuda.current_stream()
    ws, wsb = c.workspace(x.shape[0], 1, stream)
    B.vqc_backward(c.plan, x.shape[0], x.data_ptr(), w.data_ptr(), None, _ptr(st),
                   gE.data_ptr(), dx.data_ptr(), dw.data_ptr(), ws.data_ptr(), wsb,
                   stream.cuda_stream)
    return dx, dw


def _noalloc_backward(B, c, x, w, gE, st):
    dx = torch.full_like(x, float("nan"))
    dw = torch.full_like(w, float("nan"))
    B.vqc_backward_noalloc(c.plan, x.shape[0], x.data_ptr(), w.data_ptr(), None, _ptr(st),
                           gE.data_ptr(), dx.data_ptr(), dw.data_ptr(),
                           torch.cuda.current_stream().cuda_stream)
    return dx, dw


@pytest.mark.parametrize("k", [2, 3])
def test_noalloc_backward_matches_workspace_backward_twice(k):
    from paper_2607_11985_gb300 import binding as B
    from paper_2607_11985_gb300.circuit import Circuit
    w_ = wl.config(k)[0]
    c = Circuit(w_.spec, "c64")
    x, w, gE = _inputs(w_)
    E, st = c.forward(x, w, want_state=True)
    dx_ref, dw_ref = _workspace_backward(B, c, x, w, gE, st)
    for _ in range(2):
        dx, dw = _noalloc_backward(B, c, x, w, gE, st)
        torch.cuda.synchronize()
        assert torch.isfinite(dx).all() and torch.isfinite(dw).all()
        assert torch.equal(dx, dx_ref) and torch.equal(dw, dw_ref)


@pytest.mark.parametrize("saved_state", [True, False])
def test_noalloc_backward_hbm_passes(saved_state):
    # 15 qubits complex64: the backward runs HBM-tiled passes whose psi / lam
    # working states (about 0.5 MiB at batch 1) live in the built-in scratch
    from paper_2607_11985_gb300 import binding as B
    from paper_2607_11985_gb300.circuit import Circuit
    spec = wl.layered(15, 1, ("RX", "RY", "RZ"), "CX")
    rng = np.random.default_rng(1515)
    c = Circuit(spec, "c64")
    assert c.info(1)["bwd_path"] == 1
    assert B.vqc_workspace_bytes(c.plan, 1, 1) <= (1 << 20)
    x = torch.tensor(rng.uniform(-3, 3, (1, 15)), dtype=torch.float32, device="cuda")
    w = torch.tensor(rng.uniform(-3, 3, spec.num_w), dtype=torch.float32, device="cuda")
    gE = torch.tensor(rng.standard_normal((1, 15)), dtype=torch.float32, device="cuda")
    st = c.forward(x, w, want_state=True)[1] if saved_state else None
    dx_ref, dw_ref = _workspace_backward(B, c, x, w, gE, st)
    for _ in range(2):
        dx, dw = _noalloc_backward(B, c, x, w, gE, st)
        torch.cuda.synchronize()
        assert torch.isfinite(dx).all() and torch.isfinite(dw).all()
        assert torch.equal(dx, dx_ref) and torch.equal(dw, dw_ref)


@pytest.mark.parametrize("saved_state", [True, False])
def test_noalloc_backward_cluster(saved_state):
    # 14 qubits complex64: the backward runs on 2-CTA thread-block clusters; the
    # built-in scratch holds its per-cluster dw partials
    from paper_2607_11985_gb300 import binding as B
    from paper_2607_11985_gb300.circuit import Circuit
    spec = wl.layered(14, 2, ("RX", "RY", "RZ"), "CX")
    rng = np.random.default_rng(1414)
    b = 40
    c = Circuit(spec, "c64")
    assert c.info(b)["bwd_path"] == 2
    x = torch.tensor(rng.uniform(-3, 3, (b, 14)), dtype=torch.float32, device="cuda")
    w = torch.tensor(rng.uniform(-3, 3, spec.num_w), dtype=torch.float32, device="cuda")
    gE = torch.tensor(rng.standard_normal((b, 14)), dtype=torch.float32, device="cuda")
    st = c.forward(x, w, want_state=True)[1] if saved_state else None
    dx_ref, dw_ref = _workspace_backward(B, c, x, w, gE, st)
    for _ in range(2):
        dx, dw = _noalloc_backward(B, c, x, w, gE, st)
        torch.cuda.synchronize()
        assert torch.isfinite(dx).all() and torch.isfinite(dw).all()
        assert torch.equal(dx, dx_ref) and torch.equal(dw, dw_ref)


@pytest.mark.parametrize("dt", ["c128", "c128df"])
def test_noalloc_backward_complex128(dt):
    # complex128 storage (native FP64 and double-float kernels): the workspace
    # backward's gradients
    from paper_2607_11985_gb300 import binding as B
    from paper_2607_11985_gb300.circuit import Circuit
    w_ = wl.config(1, dtype=dt)[0]
    c = Circuit(w_.spec, dt)
    x, w, gE = _inputs(w_, torch.float64)
    E, st = c.forward(x, w, want_state=True)
    dx_ref, dw_ref = _workspace_backward(B, c, x, w, gE, st)
    for _ in range(2):
        dx, dw = _noalloc_backward(B, c, x, w, gE, st)
        torch.cuda.synchronize()
        assert torch.isfinite(dx).all() and torch.isfinite(dw).all()
        assert torch.equal(dx, dx_ref) and torch.equal(dw, dw_ref)


def test_noalloc_rejects_batches_beyond_the_builtin_scratch():
    from paper_2607_11985_gb300 import binding as B
    from paper_2607_11985_gb300.circuit import Circuit
    # 6000 shared weights: the per-CTA dw partials of a full grid exceed 1 MiB
    spec = wl.CircuitSpec(6, 6, 6000)
    for q in range(6):
        spec.add("RY", (q,), [("x", q)])
    for j in range(6000):
        spec.add("RZ", (j % 6,), [("w", j)])
    c = Circuit(spec, "c64")
    batch = 4096
    need = B.vqc_workspace_bytes(c.plan, batch, 1)
    assert need > (1 << 20)
    x = torch.zeros(batch, 6, device="cuda")
    w = torch.zeros(6000, device="cuda")
    gE = torch.ones(batch, 6, device="cuda")
    dx = torch.empty_like(x)
    dw = torch.empty_like(w)
    with pytest.raises(B.VQCError) as err:
        B.vqc_backward_noalloc(c.plan, batch, x.data_ptr(), w.data_ptr(), None, None,
                               gE.data_ptr(), dx.data_ptr(), dw.data_ptr(),
                               torch.cuda.current_stream().cuda_stream)
    assert err.value.status == 8
    assert "scratch" in str(err.value)
