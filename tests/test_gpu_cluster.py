"""GPU parity of the thread-block-cluster backward (VQC_FORCE_PATH=cluster):
psi and lam of one sample spread over the shared memory of 2, 4 or 8 CTAs.

* random circuits with every gate kind at each state size that has a cluster
  backward schedule (complex64 14-16 qubits, complex128 and double-float 13-15),
  against the oracle: from the saved final state and recomputing it, with and
  without psi0; the HBM passes agree on the same batch; the one-call
  forward + backward; a batch larger than the resident clusters (each cluster
  takes several samples);
* the 16-qubit / 8-layer complex64 workload at its full batch (512 rows): dx
  and dw of every row against the batch-parallel oracle;
* a circuit whose accumulators do not fit beside the two slices falls back to
  the HBM passes.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc  # noqa: E402
from paper_2607_11985_gb300 import workloads as wl  # noqa: E402
from tests.test_gpu_hbm import cfg5_reference  # noqa: E402
from tests.test_gpu_parity import TOL, C, dev, devc, maxerr, report, run_bwd, run_fwd  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


CASES = [("c64", 14), ("c64", 15), ("c64", 16), ("c128", 13), ("c128", 14), ("c128", 15),
         ("c128df", 13), ("c128df", 15)]


@pytest.mark.parametrize("dtype,n", CASES)
def test_cluster_backward_random(monkeypatch, dtype, n):
    """dx and dw of a random circuit (every gate kind, constants, phases,
    folded CX / SWAP) against the oracle, from psi_final and recomputing, from
    |0...0> and from psi0; the HBM passes give the same gradients."""
    w_, psi0 = wl.small_random(7300 + n, n, 150, batch=5, dtype=dtype, with_psi0=True)
    c = C(w_.spec, dtype)
    # by default the cluster for 2-CTA clusters, else the HBM passes
    two_cta = (dtype, n) in (("c64", 14), ("c128", 13), ("c128df", 13))
    assert c.info(w_.batch)["bwd_path"] == (2 if two_cta else 1)
    monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
    info = c.info(w_.batch)
    assert info["bwd_path"] == 2
    assert info["bwd_threads_per_sample"] == 1 << (n - info["bwd_k"])
    tol = TOL[dtype]["grad"]
    for p0 in (None, psi0):
        dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=p0)
        E, st = run_fwd(c, w_, p0)
        dx, dw = run_bwd(c, w_, p0, psi_final=devc(st, dtype))
        dx2, dw2 = run_bwd(c, w_, p0)
        monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
        dx3, dw3 = run_bwd(c, w_, p0)
        monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
        errs = dict(dx=maxerr(dx, dx_ref), dw=maxerr(dw, dw_ref), dx_recompute=maxerr(dx2, dx_ref),
                    dw_recompute=maxerr(dw2, dw_ref), dx_hbm=maxerr(dx3, dx), dw_hbm=maxerr(dw3, dw))
        report("cluster_bwd_%s_n%d%s" % (dtype, n, "_psi0" if p0 is not None else ""), **errs)
        for k, v in errs.items():
            assert v <= tol, (k, v)


@pytest.mark.parametrize("dtype", ["c64", "c128"])
def test_cluster_forward_backward_and_many_samples(monkeypatch, dtype):
    """vqc_forward_backward with the cluster backward (the forward leaves the
    final states in the workspace), on a batch larger than the clusters that
    fit the GPU, against the oracle and the separate calls."""
    n = 15
    spec = wl.layered(n, 2, ("RX", "RY", "RZ"), "CX", ring_range=lambda l: 2 * l + 1)
    spec.add("CRZ", (n - 1, 2), [("w", 0)]).add("RZZ", (3, n - 3), [("x", 1)])
    rng = np.random.default_rng(2500 + n)
    B = 200
    w_ = wl.Workload("cluster_fb_n%d" % n, spec, B, wl._round(rng.uniform(-np.pi, np.pi, (B, n)), dtype),
                     wl._round(rng.uniform(-np.pi, np.pi, spec.num_w), dtype),
                     wl._round(rng.standard_normal((B, n)), dtype), dtype, 2500 + n)
    monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
    c = C(spec, dtype)
    assert c.info(B)["bwd_path"] == 2
    x, w, gE = dev(w_.x, dtype), dev(w_.w, dtype), dev(w_.gE, dtype)
    E, dx, dw = c.forward_backward(x, w, gE)
    torch.cuda.synchronize()
    E, dx, dw = E.cpu().numpy(), dx.cpu().numpy(), dw.cpu().numpy()
    dx2, dw2 = run_bwd(c, w_)
    tol = TOL[dtype]
    assert maxerr(dx, dx2) <= tol["grad"] and maxerr(dw, dw2) <= tol["grad"]
    rows = [0, 77, B - 1]
    E_ref = orc.forward(spec, w_.x[rows], w_.w)
    dx_ref, _ = orc.backward(spec, w_.x[rows], w_.w, w_.gE[rows])
    _, dw_ref = orc.backward_parallel(spec, w_.x, w_.w, w_.gE)
    errs = dict(E=maxerr(E[rows], E_ref), dx=maxerr(dx[rows], dx_ref), dw=maxerr(dw, dw_ref))
    report(w_.name + "_" + dtype, **errs)
    assert errs["E"] <= tol["E"] and errs["dx"] <= tol["grad"] and errs["dw"] <= tol["grad"]


def test_config5_cluster_backward_full_batch(monkeypatch):
    """The 16-qubit / 8-layer complex64 workload, all 512 rows, through the
    cluster backward (8-CTA clusters): dx and dw from the saved final states and
    recomputing them, against the oracle."""
    w_ = wl.config(5, dtype="c64")[0]
    c = C(w_.spec, "c64")
    monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
    assert c.info(w_.batch)["bwd_path"] == 2
    ref = cfg5_reference(w_)
    E, st = run_fwd(c, w_)
    dx, dw = run_bwd(c, w_, psi_final=devc(st, "c64"))
    del st
    dx2, dw2 = run_bwd(c, w_)
    errs = dict(dx=maxerr(dx, ref["dx"]), dw=maxerr(dw, ref["dw"]), dx_recompute=maxerr(dx2, ref["dx"]),
                dw_recompute=maxerr(dw2, ref["dw"]))
    report(w_.name + "_cluster", **errs)
    for k, v in errs.items():
        assert v <= TOL["c64"]["grad"], (k, v)


def test_cluster_backward_falls_back_when_accumulators_do_not_fit(monkeypatch):
    """A deep 14-qubit circuit (420 parametrised runs): the cluster backward's
    per-warp rho partials would not fit one CTA's shared memory next to psi and
    lam, so the backward takes the HBM passes, by default and when the cluster
    is asked for; its gradients still match the oracle."""
    n = 14
    spec = wl.layered(n, 30, ("RX", "RY"), "CX")
    rng = np.random.default_rng(3014)
    B = 2
    w_ = wl.Workload("deep_n14", spec, B, wl._round(rng.uniform(-np.pi, np.pi, (B, n)), "c64"),
                     wl._round(rng.uniform(-np.pi, np.pi, spec.num_w), "c64"),
                     wl._round(rng.standard_normal((B, n)), "c64"), "c64", 3014)
    c = C(spec, "c64")
    assert c.info(B)["bwd_path"] == 1
    monkeypatch.setenv("VQC_FORCE_PATH", "cluster")
    assert c.info(B)["bwd_path"] == 1
    dx, dw = run_bwd(c, w_)
    dx_ref, dw_ref = orc.backward(spec, w_.x, w_.w, w_.gE)
    assert maxerr(dx, dx_ref) <= TOL["c64"]["grad"] and maxerr(dw, dw_ref) <= TOL["c64"]["grad"]
