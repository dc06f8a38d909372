"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Tolerances (stated for this engine): complex64 path -- expectations and
amplitudes max-abs <= 1e-4, gradients max-abs <= 5e-4; complex128 path --
<= 1e-10 for all of them.  Inputs are seeded and generated in fp64, rounded to
the engine's real type, and the oracle consumes the rounded values promoted to
fp64, so the comparison measures kernel error only.
"""
import os

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc  # noqa: E402
from paper_2607_11985_gb300 import workloads as wl  # noqa: E402
from paper_2607_11985_gb300 import binding as B  # noqa: E402

pytestmark = pytest.mark.gpu

TOL = {"c64": dict(E=1e-4, state=1e-4, grad=5e-4), "c128": dict(E=1e-10, state=1e-10, grad=1e-10),
       "c128df": dict(E=1e-10, state=1e-10, grad=1e-10)}   # complex128 storage, double-float arithmetic


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def C(spec, dtype):
    from paper_2607_11985_gb300.circuit import Circuit
    return Circuit(spec, dtype)


def dev(a, dtype):
    real = torch.float32 if dtype == "c64" else torch.float64
    return torch.tensor(np.asarray(a), dtype=real, device="cuda")


def devc(a, dtype):
    cplx = torch.complex64 if dtype == "c64" else torch.complex128
    return torch.tensor(np.asarray(a), dtype=cplx, device="cuda")


def run_fwd(c, w_, psi0=None, want_state=True):
    x = dev(w_.x, w_.dtype) if w_.spec.num_x else None
    w = dev(w_.w, w_.dtype) if w_.spec.num_w else None
    p0 = devc(psi0, w_.dtype) if psi0 is not None else None
    if x is None and p0 is None:
        # batch is carried by x; circuits without x get a zero-column x
        pass
    out = c.forward(x, w, psi0=p0, want_state=want_state)
    torch.cuda.synchronize()
    if want_state:
        return out[0].cpu().numpy(), out[1].cpu().numpy()
    return out.cpu().numpy()


def run_bwd(c, w_, psi0=None, psi_final=None):
    x = dev(w_.x, w_.dtype) if w_.spec.num_x else None
    w = dev(w_.w, w_.dtype) if w_.spec.num_w else None
    gE = dev(w_.gE, w_.dtype)
    p0 = devc(psi0, w_.dtype) if psi0 is not None else None
    dx, dw = c.backward(x, w, gE, psi0=p0, psi_final=psi_final)
    torch.cuda.synchronize()
    return (dx.cpu().numpy() if dx is not None else np.zeros((w_.batch, 0)),
            dw.cpu().numpy() if dw is not None else np.zeros(0))


def maxerr(a, b):
    a, b = np.asarray(a), np.asarray(b)
    return float(np.max(np.abs(a - b))) if a.size else 0.0


# ------------------------------------------------------------------ small random circuits
SMALL = [(201, 1, 10), (202, 2, 40), (203, 3, 80), (204, 4, 120), (205, 5, 160), (206, 6, 200),
         (207, 7, 200), (208, 8, 240), (209, 9, 200), (210, 10, 160)]


@pytest.mark.parametrize("dtype", ["c64", "c128", "c128df"])
@pytest.mark.parametrize("seed,n,G", SMALL)
def test_random_forward_and_gradients(seed, n, G, dtype):
    w_, psi0 = wl.small_random(seed, n, G, batch=37, dtype=dtype, with_psi0=(seed % 2 == 0))
    if w_.spec.num_x == 0:
        pytest.skip("needs x to carry the batch")
    c = C(w_.spec, dtype)
    E, st = run_fwd(c, w_, psi0)
    E_ref, st_ref = orc.forward(w_.spec, w_.x, w_.w, psi0=psi0, want_state=True)
    tol = TOL[dtype]
    assert maxerr(E, E_ref) <= tol["E"]
    assert maxerr(st, st_ref) <= tol["state"]
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
    dx, dw = run_bwd(c, w_, psi0)                       # recompute psi_final in the kernel
    assert maxerr(dx, dx_ref) <= tol["grad"]
    assert maxerr(dw, dw_ref) <= tol["grad"]
    dx2, dw2 = run_bwd(c, w_, psi0, psi_final=devc(st, dtype))   # from the saved state
    assert maxerr(dx2, dx_ref) <= tol["grad"]
    assert maxerr(dw2, dw_ref) <= tol["grad"]


@pytest.mark.parametrize("mode_env", ["VQC_FORCE_K_FWD", "VQC_FORCE_K_BWD"])
@pytest.mark.parametrize("K", [1, 2, 3, 4, 5])
def test_every_register_block_size(monkeypatch, mode_env, K):
    w_, psi0 = wl.small_random(300 + K, 8, 200, batch=19, dtype="c64", with_psi0=True)
    monkeypatch.setenv(mode_env, str(K))
    c = C(w_.spec, "c64")
    E, st = run_fwd(c, w_, psi0)
    E_ref, st_ref = orc.forward(w_.spec, w_.x, w_.w, psi0=psi0, want_state=True)
    assert maxerr(E, E_ref) <= 1e-4
    assert maxerr(st, st_ref) <= 1e-4
    dx, dw = run_bwd(c, w_, psi0)
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
    assert maxerr(dx, dx_ref) <= 5e-4
    assert maxerr(dw, dw_ref) <= 5e-4


# ------------------------------------------------------------------ the five workloads
def test_config1_full():
    w_ = wl.config(1)[0]
    c = C(w_.spec, "c64")
    E, st = run_fwd(c, w_)
    assert maxerr(E, orc.forward(w_.spec, w_.x, w_.w)) <= 1e-4
    dx, dw = run_bwd(c, w_, psi_final=devc(st, "c64"))
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE)
    assert maxerr(dx, dx_ref) <= 5e-4
    assert maxerr(dw, dw_ref) <= 5e-4


def test_config2_full():
    w_ = wl.config(2)[0]
    c = C(w_.spec, "c64")
    E, st = run_fwd(c, w_)
    assert maxerr(E, orc.forward(w_.spec, w_.x, w_.w)) <= 1e-4
    dx, dw = run_bwd(c, w_, psi_final=devc(st, "c64"))
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE)
    assert maxerr(dx, dx_ref) <= 5e-4
    assert maxerr(dw, dw_ref) <= 5e-4


def test_config2_paper_objective_mean_z():
    # the paper's scalar objective: mean of <Z_i>  (upstream gradient 1/n)
    w_ = wl.config(2, batch=64)[0]
    w_.gE = np.full_like(w_.gE, np.float32(1.0 / w_.spec.n))
    c = C(w_.spec, "c64")
    dx, dw = run_bwd(c, w_)
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE)
    assert maxerr(dx, dx_ref) <= 5e-4
    assert maxerr(dw, dw_ref) <= 5e-4


def oracle_full(w_, psi0=None, want_state=False, backward=True):
    """The oracle on a whole batch, batch-parallel over the host cores (rows are
    independent): E (and final states), dx and dw of the workload's inputs."""
    out = {}
    if want_state:
        out["E"], out["st"] = orc.forward_parallel(w_.spec, w_.x, w_.w, psi0=psi0, want_state=True)
    else:
        out["E"] = orc.forward_parallel(w_.spec, w_.x, w_.w, psi0=psi0)
    if backward:
        out["dx"], out["dw"] = orc.backward_parallel(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
    return out


def report(name, **errs):
    print("PARITY %s %s" % (name, " ".join("%s=%.3e" % kv for kv in errs.items())))


def test_config3_full_batch():
    """The 12-qubit re-uploading workload at its full batch (4096 rows, the
    launch the benchmark times): E, dx and dw element by element against the
    oracle on the same inputs; the forward+backward call too."""
    w_ = wl.config(3)[0]
    c = C(w_.spec, "c64")
    ref = oracle_full(w_)
    E, st = run_fwd(c, w_)
    dx, dw = run_bwd(c, w_, psi_final=devc(st, "c64"))
    dx2, dw2 = run_bwd(c, w_)                          # recomputing the final states
    x, w, gE = dev(w_.x, "c64"), dev(w_.w, "c64"), dev(w_.gE, "c64")
    Ef, dxf, dwf = (t.cpu().numpy() for t in c.forward_backward(x, w, gE))
    errs = dict(E=maxerr(E, ref["E"]), dx=maxerr(dx, ref["dx"]), dw=maxerr(dw, ref["dw"]),
                dx_recompute=maxerr(dx2, ref["dx"]), dw_recompute=maxerr(dw2, ref["dw"]),
                E_fused=maxerr(Ef, ref["E"]), dx_fused=maxerr(dxf, ref["dx"]),
                dw_fused=maxerr(dwf, ref["dw"]))
    report(w_.name, **errs)
    for k, v in errs.items():
        assert v <= (1e-4 if k.startswith("E") else 5e-4), (k, v)


def test_config4_random_circuits_full_state():
    """All 32 random circuits, every one of the 256 rows: E and the full final
    statevectors element by element, and the fidelity, against the oracle."""
    worst = {"E": 0.0, "state": 0.0, "infidelity": 0.0}
    for w_ in wl.config(4):
        c = C(w_.spec, "c64")
        E, st = run_fwd(c, w_)
        ref = oracle_full(w_, want_state=True, backward=False)
        eE, es = maxerr(E, ref["E"]), maxerr(st, ref["st"])
        fid = np.abs(np.sum(np.conj(ref["st"]) * st, axis=1)) ** 2
        worst["E"] = max(worst["E"], eE)
        worst["state"] = max(worst["state"], es)
        worst["infidelity"] = max(worst["infidelity"], float(1 - fid.min()))
        assert eE <= 1e-4, w_.name
        assert es <= 1e-4, w_.name
        assert np.all(fid >= 1 - 1e-5), w_.name
        del c, st, ref
    report("cfg4_random32_B256", **worst)


# ------------------------------------------------------------------ edge cases
def test_zero_batch_and_ragged_batches():
    w_, _ = wl.small_random(401, 6, 80, batch=1, dtype="c64")
    c = C(w_.spec, "c64")
    x = torch.empty(0, w_.spec.num_x, device="cuda")
    w = dev(w_.w, "c64")
    E = c.forward(x, w)
    assert E.shape == (0, 6)
    for B in (1, 2, 3, 5, 31, 33, 129, 257):
        wb, _ = wl.small_random(401, 6, 80, batch=B, dtype="c64")
        E = run_fwd(c, wb, want_state=False)
        assert maxerr(E, orc.forward(wb.spec, wb.x, wb.w)) <= 1e-4
        dx, dw = run_bwd(c, wb)
        dx_ref, dw_ref = orc.backward(wb.spec, wb.x, wb.w, wb.gE)
        assert maxerr(dx, dx_ref) <= 5e-4 and maxerr(dw, dw_ref) <= 5e-4


def test_batch_rows_independent():
    w_, psi0 = wl.small_random(402, 7, 150, batch=9, dtype="c64", with_psi0=True)
    c = C(w_.spec, "c64")
    E = run_fwd(c, w_, psi0, want_state=False)
    for b in (0, 4, 8):
        one = wl.Workload(w_.name, w_.spec, 1, w_.x[b:b + 1], w_.w, w_.gE[b:b + 1], "c64", 0)
        Eb = run_fwd(c, one, psi0[b:b + 1], want_state=False)
        assert maxerr(Eb[0], E[b]) <= 1e-6


def test_only_two_qubit_gates_and_constants():
    spec = wl.CircuitSpec(6, 1, 0)
    spec.add("RY", (0,), [("x", 0)])
    for q in range(5):
        spec.add("CX", (q, q + 1))
    spec.add("SWAP", (0, 5)).add("CZ", (2, 4)).add("CRZ", (1, 3), [("c", 0.7)])
    spec.add("RZZ", (5, 2), [("c", -1.3)]).add("H", (4,)).add("T", (4,)).add("SX", (1,))
    rng = np.random.default_rng(5)
    x = wl._round(rng.uniform(-np.pi, np.pi, (11, 1)), "c64")
    w_ = wl.Workload("twoq", spec, 11, x, np.zeros(0), wl._round(rng.standard_normal((11, 6)), "c64"), "c64", 0)
    c = C(spec, "c64")
    E, st = run_fwd(c, w_)
    E_ref, st_ref = orc.forward(spec, x, None, want_state=True)
    assert maxerr(E, E_ref) <= 1e-4 and maxerr(st, st_ref) <= 1e-4
    dx, _ = run_bwd(c, w_)
    dx_ref, _ = orc.backward(spec, x, None, w_.gE)
    assert maxerr(dx, dx_ref) <= 5e-4


def test_single_rotation_closed_form_on_gpu():
    spec = wl.CircuitSpec(1, 1, 0).add("RY", (0,), [("x", 0)])
    t = np.linspace(-np.pi, np.pi, 65)[:, None]
    w_ = wl.Workload("ry", spec, 65, wl._round(t, "c128"), np.zeros(0), np.ones((65, 1)), "c128", 0)
    c = C(spec, "c128")
    E, _ = run_fwd(c, w_)
    assert np.max(np.abs(E[:, 0] - np.cos(t[:, 0]))) <= 1e-12
    dx, _ = run_bwd(c, w_)
    assert np.max(np.abs(dx[:, 0] + np.sin(t[:, 0]))) <= 1e-12


def test_autograd_function():
    w_ = wl.config(1, batch=16)[0]
    c = C(w_.spec, "c64")
    x = dev(w_.x, "c64").requires_grad_(True)
    w = dev(w_.w, "c64").requires_grad_(True)
    E = c(x, w)
    (E * dev(w_.gE, "c64")).sum().backward()
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE)
    assert maxerr(x.grad.cpu().numpy(), dx_ref) <= 5e-4
    assert maxerr(w.grad.cpu().numpy(), dw_ref) <= 5e-4


def test_deterministic_dw():
    w_ = wl.config(2)[0]
    c = C(w_.spec, "c64")
    _, dw1 = run_bwd(c, w_)
    _, dw2 = run_bwd(c, w_)
    assert np.array_equal(dw1, dw2)


# ------------------------------------------------------------------ folded CX, multi-warp groups
@pytest.mark.parametrize("n", [11, 12, 13])
def test_folded_cx_multiwarp_groups(n):
    """CX rings folded into stage store maps while a sample is spread over
    several warps (2^(n-K) >= 64 threads): a permuting store writes slots other
    warps load in the same stage, so the kernels order every load of the stage
    before the stores.  Repeated calls against the oracle, forward and
    backward."""
    spec = wl.layered(n, 3, ("RX", "RY"), "CX", ring_range=lambda l: l + 1)
    rng = np.random.default_rng(900 + n)
    B = 24
    x = wl._round(rng.uniform(-np.pi, np.pi, (B, n)), "c64")
    w = wl._round(rng.uniform(-np.pi, np.pi, spec.num_w), "c64")
    gE = wl._round(rng.standard_normal((B, n)), "c64")
    w_ = wl.Workload("cx_ring_n%d" % n, spec, B, x, w, gE, "c64", 900 + n)
    c = C(spec, "c64")
    info = c.info(B)
    assert info["fwd_path"] == 0 and info["fwd_threads_per_sample"] >= 64
    E_ref, st_ref = orc.forward(spec, x, w, want_state=True)
    dx_ref, dw_ref = orc.backward(spec, x, w, gE)
    for _ in range(3):
        E, st = run_fwd(c, w_)
        assert maxerr(E, E_ref) <= TOL["c64"]["E"] and maxerr(st, st_ref) <= TOL["c64"]["state"]
        dx, dw = run_bwd(c, w_)                       # recomputed forward inside the backward
        report("cx_ring_n%d_recompute" % n, dx=maxerr(dx, dx_ref), dw=maxerr(dw, dw_ref))
        assert maxerr(dx, dx_ref) <= 5e-4 and maxerr(dw, dw_ref) <= 5e-4
        dx, dw = run_bwd(c, w_, psi_final=devc(st, "c64"))
        report("cx_ring_n%d_saved" % n, dx=maxerr(dx, dx_ref), dw=maxerr(dw, dw_ref))
        assert maxerr(dx, dx_ref) <= 5e-4 and maxerr(dw, dw_ref) <= 5e-4


def test_largest_resident_forward_n14():
    """14 qubits at batch 3: the largest resident forward (register blocks of 32
    amplitudes, 512 threads per sample, folded CX rings); the backward runs
    HBM-tiled passes."""
    n = 14
    spec = wl.layered(n, 2, ("RY", "RZ"), "CX")
    rng = np.random.default_rng(914)
    B = 3
    x = wl._round(rng.uniform(-np.pi, np.pi, (B, n)), "c64")
    w = wl._round(rng.uniform(-np.pi, np.pi, spec.num_w), "c64")
    gE = wl._round(rng.standard_normal((B, n)), "c64")
    w_ = wl.Workload("cx_ring_n14", spec, B, x, w, gE, "c64", 914)
    c = C(spec, "c64")
    info = c.info(B)
    assert info["fwd_path"] == 0 and info["fwd_threads_per_sample"] == 512
    E_ref, st_ref = orc.forward(spec, x, w, want_state=True)
    dx_ref, dw_ref = orc.backward(spec, x, w, gE)
    E, st = run_fwd(c, w_)
    assert maxerr(E, E_ref) <= TOL["c64"]["E"] and maxerr(st, st_ref) <= TOL["c64"]["state"]
    for psi_final in (None, devc(st, "c64")):
        dx, dw = run_bwd(c, w_, psi_final=psi_final)
        assert maxerr(dx, dx_ref) <= 5e-4 and maxerr(dw, dw_ref) <= 5e-4


# ------------------------------------------------------------------ fused forward + backward
@pytest.mark.parametrize("case", ["cfg1", "cfg2", "cfg3_rows", "rand_c128_psi0", "rand_c128df_psi0", "hbm16"])
def test_forward_backward_fused(case, monkeypatch):
    """vqc_forward_backward (one launch on the resident path: the backward kernel
    sweeps forward itself and writes E) against the oracle and against the
    separate vqc_forward + vqc_backward.  Covers sub-warp groups (4 qubits),
    one-warp groups (8), multi-warp groups (12), complex128 with psi0, and a
    16-qubit plan that runs as forward passes + recomputing backward passes."""
    psi0 = None
    if case == "cfg1":
        w_ = wl.config(1)[0]
    elif case == "cfg2":
        w_ = wl.config(2)[0]
    elif case == "cfg3_rows":
        full = wl.config(3)[0]
        idx = np.arange(40) * 97 % full.batch
        w_ = wl.Workload(full.name, full.spec, 40, full.x[idx], full.w, full.gE[idx], "c64", full.seed)
    elif case in ("rand_c128_psi0", "rand_c128df_psi0"):
        w_, psi0 = wl.small_random(777, 9, 180, batch=6, dtype=case[5:-5], with_psi0=True)
    else:
        spec = wl.layered(16, 1, ("RX", "RY", "RZ"), "CX")
        rng = np.random.default_rng(1616)
        w_ = wl.Workload("hbm16", spec, 2, wl._round(rng.uniform(-3, 3, (2, 16)), "c64"),
                         wl._round(rng.uniform(-3, 3, spec.num_w), "c64"),
                         wl._round(rng.standard_normal((2, 16)), "c64"), "c64", 1616)
    dt = w_.dtype
    c = C(w_.spec, dt)
    x = dev(w_.x, dt) if w_.spec.num_x else None
    w = dev(w_.w, dt) if w_.spec.num_w else None
    gE = dev(w_.gE, dt)
    p0 = devc(psi0, dt) if psi0 is not None else None
    E, dx, dw = c.forward_backward(x, w, gE, psi0=p0)
    torch.cuda.synchronize()
    E, dx, dw = E.cpu().numpy(), (dx.cpu().numpy() if dx is not None else None), \
        (dw.cpu().numpy() if dw is not None else None)
    E2 = run_fwd(c, w_, psi0, want_state=False)
    dx2, dw2 = run_bwd(c, w_, psi0)
    tol = TOL[dt]
    close = 1e-5 if dt == "c64" else 1e-12
    assert maxerr(E, E2) <= close
    if dx is not None:
        assert maxerr(dx, dx2) <= 10 * close
    if dw is not None:
        assert maxerr(dw, dw2) <= 10 * close * max(1.0, float(np.abs(dw2).max()))
    rows = [0, w_.batch - 1]
    E_ref = orc.forward(w_.spec, w_.x[rows], w_.w, psi0=None if psi0 is None else psi0[rows])
    dx_ref, _ = orc.backward(w_.spec, w_.x[rows], w_.w, w_.gE[rows],
                             psi0=None if psi0 is None else psi0[rows])
    assert maxerr(E[rows], E_ref) <= tol["E"]
    if dx is not None:
        assert maxerr(dx[rows], dx_ref) <= tol["grad"]
    if w_.batch <= 64 and dw is not None:
        _, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
        assert maxerr(dw, dw_ref) <= tol["grad"]


@pytest.mark.parametrize("case", ["cfg3_rows", "rand_psi0"])
def test_double_float_agrees_with_fp64(case):
    """complex128 with double-float arithmetic against native FP64 on the same
    inputs: E, final states and gradients agree far inside the complex128
    parity bound (48-bit double-float against 53-bit double)."""
    if case == "cfg3_rows":
        full = wl.config(3, dtype="c128")[0]
        idx = np.arange(64) * 61 % full.batch
        w_ = wl.Workload(full.name, full.spec, 64, full.x[idx], full.w, full.gE[idx], "c128", full.seed)
        psi0 = None
    else:
        w_, psi0 = wl.small_random(778, 10, 220, batch=8, dtype="c128", with_psi0=True)
    out = {}
    for dt in ("c128", "c128df"):
        c = C(w_.spec, dt)
        E, st = run_fwd(c, w_, psi0)
        dx, dw = run_bwd(c, w_, psi0)
        out[dt] = (E, st, dx, dw)
    for a, b in zip(out["c128"], out["c128df"]):
        scale = max(1.0, float(np.abs(a).max())) if a.size else 1.0
        assert maxerr(a, b) <= 1e-12 * scale


# ------------------------------------------------------------------ degenerate circuits
@pytest.mark.parametrize("dtype", ["c64", "c128", "c128df"])
@pytest.mark.parametrize("which", ["empty", "no_params", "one_long_run"])
def test_degenerate_circuits(dtype, which):
    """An empty gate list (E = <Z> of psi0; the state passes through), a circuit
    without any angle parameter (gradients have no entries), and one qubit
    carrying a single fused run of 40 rotations (far more than a table entry's
    four constituents) with a gradient for every angle: forward, backward and
    the fused call against the oracle, with and without psi0."""
    rng = np.random.default_rng({"empty": 11, "no_params": 12, "one_long_run": 13}[which])
    if which == "empty":
        spec = wl.CircuitSpec(3, 0, 0)
    elif which == "no_params":
        spec = wl.CircuitSpec(5, 0, 0).add("H", (0,)).add("CX", (0, 4)).add("T", (4,)) \
            .add("SWAP", (1, 3)).add("U3", (2,), [("c", 0.3), ("c", -1.1), ("c", 2.0)]).add("CZ", (2, 4))
    else:
        spec = wl.CircuitSpec(4, 2, 20).add("H", (1,)).add("CX", (1, 2))
        for k in range(40):
            g = ("RX", "RY", "RZ")[k % 3]
            spec.add(g, (2,), [("x", k % 2)] if k % 4 == 0 else [("w", k % 20)])
        spec.add("CRZ", (2, 3), [("w", 3)])
    Bt = 5
    x = wl._round(rng.uniform(-np.pi, np.pi, (Bt, spec.num_x)), dtype)
    w = wl._round(rng.uniform(-np.pi, np.pi, spec.num_w), dtype)
    gE = wl._round(rng.standard_normal((Bt, spec.n)), dtype)
    z = rng.standard_normal((Bt, 1 << spec.n)) + 1j * rng.standard_normal((Bt, 1 << spec.n))
    z /= np.linalg.norm(z, axis=1, keepdims=True)
    if dtype == "c64":
        z = z.astype(np.complex64).astype(np.complex128)
    c = C(spec, dtype)
    tol = TOL[dtype]
    real = torch.float32 if dtype == "c64" else torch.float64
    xd = torch.tensor(x, dtype=real, device="cuda")   # [B, 0] when there is no x: carries B
    wd = dev(w, dtype) if spec.num_w else None
    gd = dev(gE, dtype)
    for psi0 in (None, z):
        p0 = devc(psi0, dtype) if psi0 is not None else None
        E, st = c.forward(xd, wd, psi0=p0, want_state=True)
        dx, dw = c.backward(xd if spec.num_x else None, wd, gd, psi0=p0)
        Ef, dxf, dwf = c.forward_backward(xd if spec.num_x else None, wd, gd, psi0=p0)
        torch.cuda.synchronize()
        E_ref, st_ref = orc.forward(spec, x, w, psi0=psi0, want_state=True)
        dx_ref, dw_ref = orc.backward(spec, x, w, gE, psi0=psi0)
        assert maxerr(E.cpu().numpy(), E_ref) <= tol["E"]
        assert maxerr(Ef.cpu().numpy(), E_ref) <= tol["E"]
        assert maxerr(st.cpu().numpy(), st_ref) <= tol["state"]
        if which == "empty":
            assert maxerr(st.cpu().numpy(), psi0 if psi0 is not None else
                          np.eye(1, 1 << spec.n).repeat(Bt, 0)) <= tol["state"]
        for got, ref in ((dx, dx_ref), (dw, dw_ref), (dxf, dx_ref), (dwf, dw_ref)):
            if got is None:
                assert np.asarray(ref).size == 0
            else:
                assert maxerr(got.cpu().numpy(), ref) <= tol["grad"]


def test_two_streams_share_a_plan():
    """One plan used on two CUDA streams at once (each with its own workspace,
    different batches): results equal those of the same calls made one after
    the other on the default stream."""
    w_ = wl.config(2)[0]
    c = C(w_.spec, "c64")
    x = dev(w_.x, "c64")
    w = dev(w_.w, "c64")
    gE = dev(w_.gE, "c64")
    halves = [slice(0, 400), slice(400, 1024)]
    ref = []
    for h in halves:
        E, st = c.forward(x[h], w, want_state=True)
        dx, dw = c.backward(x[h], w, gE[h], psi_final=st)
        ref.append((E.clone(), dx.clone(), dw.clone()))
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    got = []
    for _ in range(3):
        got.clear()
        for h, s in zip(halves, streams):
            with torch.cuda.stream(s):
                E, st = c.forward(x[h], w, want_state=True)
                dx, dw = c.backward(x[h], w, gE[h], psi_final=st)
                got.append((E, dx, dw))
        torch.cuda.synchronize()
        for (E, dx, dw), (E0, dx0, dw0) in zip(got, ref):
            assert torch.equal(E, E0) and torch.equal(dx, dx0) and torch.equal(dw, dw0)


def test_sync_check_after_every_kernel_kind(monkeypatch):
    """vqc_sync_check reads every plan's error word: after resident forward,
    backward and fused launches, HBM passes, the cluster forward and the
    probabilities kernel, no launch self-check has tripped."""
    w_ = wl.config(2, batch=64)[0]
    c = C(w_.spec, "c64")
    x, w, gE = dev(w_.x, "c64"), dev(w_.w, "c64"), dev(w_.gE, "c64")
    E, st = c.forward(x, w, want_state=True)
    c.backward(x, w, gE, psi_final=st)
    c.forward_backward(x, w, gE)
    c.probabilities(x, w)
    spec = wl.layered(15, 1, ("RX", "RY", "RZ"), "CX")
    rng = np.random.default_rng(15)
    c2 = C(spec, "c64")
    x2 = dev(rng.uniform(-3, 3, (2, 15)), "c64")
    w2 = dev(rng.uniform(-3, 3, spec.num_w), "c64")
    g2 = dev(rng.standard_normal((2, 15)), "c64")
    monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
    assert c2.info(2)["fwd_path"] == 1
    E2, st2 = c2.forward(x2, w2, want_state=True)          # HBM passes
    c2.backward(x2, w2, g2, psi_final=st2)
    monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
    assert c2.info(2)["fwd_path"] == 2
    c2.forward(x2, w2)                                      # cluster forward
    B.vqc_sync_check(torch.cuda.current_stream().cuda_stream)


def test_argument_errors_before_any_launch():
    """Every argument check of the device calls fails before anything is
    launched: NULL / misaligned pointers, negative batch, short or misaligned
    workspace, NULL plan.  The stream stays clean (vqc_sync_check)."""
    w_ = wl.config(2, batch=8)[0]
    c = C(w_.spec, "c64")
    s = torch.cuda.current_stream().cuda_stream
    x, w, gE = dev(w_.x, "c64"), dev(w_.w, "c64"), dev(w_.gE, "c64")
    E = torch.empty(8, w_.spec.n, device="cuda")
    st = torch.empty(8, 1 << w_.spec.n, dtype=torch.complex64, device="cuda")
    dx, dw = torch.empty_like(x), torch.empty_like(w)
    ws, wsb = c.workspace(8, 1, torch.cuda.current_stream())
    ws3, ws3b = c.workspace(8, 3, torch.cuda.current_stream())

    def P(t, off=0):
        return t.data_ptr() + off

    fwd = lambda **k: B.vqc_forward(k.get("plan", c.plan), k.get("b", 8), k.get("x", P(x)), P(w), None,   # noqa: E731
                                    k.get("E", P(E)), k.get("st"), None, 0, s)
    bwd = lambda **k: B.vqc_backward(c.plan, 8, P(x), P(w), None, k.get("psi", P(st)), k.get("g", P(gE)),   # noqa: E731
                                     k.get("dx", P(dx)), P(dw), k.get("ws", P(ws)), k.get("wsb", wsb), s)
    fb = lambda **k: B.vqc_forward_backward(c.plan, 8, P(x), P(w), None, k.get("g", P(gE)),   # noqa: E731
                                            k.get("E", P(E)), P(dx), k.get("dw", P(dw)),
                                            P(ws3) if ws3 is not None else None, ws3b, s)
    cases = [
        (lambda: fwd(plan=None), 1), (lambda: fwd(b=-1), 1), (lambda: fwd(x=None), 1),
        (lambda: fwd(E=None), 1), (lambda: fwd(x=P(x, 2)), 1), (lambda: fwd(E=P(E, 2)), 1),
        (lambda: fwd(st=P(st, 4)), 1),
        (lambda: bwd(g=None), 1), (lambda: bwd(dx=P(dx, 2)), 1), (lambda: bwd(psi=P(st, 4)), 1),
        (lambda: bwd(wsb=16), 8), (lambda: bwd(ws=P(ws, 16), wsb=wsb - 16), 8), (lambda: bwd(ws=None), 8),
        (lambda: fb(E=None), 1), (lambda: fb(g=None), 1), (lambda: fb(dw=P(dw, 2)), 1),
    ]
    for i, (call, code) in enumerate(cases):
        with pytest.raises(B.VQCError) as e:
            call()
        assert e.value.status == code, (i, str(e.value))
    B.vqc_sync_check(s)


def test_geometries_sharing_a_kernel(monkeypatch):
    """Two launch geometries of the same kernel instantiation with different
    shared-memory needs, used alternately (here: the default CTA size, then a
    smaller one, then the default again from the geometry cache; the same
    happens with two plans): every launch keeps working and gives the same
    result."""
    w_ = wl.config(1)[0]
    c = C(w_.spec, "c64")
    x, w, gE = dev(w_.x, "c64"), dev(w_.w, "c64"), dev(w_.gE, "c64")
    E0 = c.forward(x, w)
    dx0, dw0 = c.backward(x, w, gE)
    monkeypatch.setenv("VQC_CTA_THREADS", "64")
    E1 = c.forward(x, w)
    dx1, dw1 = c.backward(x, w, gE)
    monkeypatch.delenv("VQC_CTA_THREADS")
    E2 = c.forward(x, w)
    dx2, dw2 = c.backward(x, w, gE)
    torch.cuda.synchronize()
    assert torch.equal(E0, E1) and torch.equal(E0, E2)
    assert torch.equal(dx0, dx2) and torch.equal(dw0, dw2)
    assert maxerr(dx1.cpu().numpy(), dx0.cpu().numpy()) <= 1e-6
    assert maxerr(dw1.cpu().numpy(), dw0.cpu().numpy()) <= 1e-5
