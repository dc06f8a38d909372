"""GPU parity on randomly drawn circuits, across execution paths.

Each case draws (from a fixed seed) a qubit count of 1-12, a gate count of
1-119, the precision, a batch of 1-6 and whether a psi0 is given, builds a
random circuit of the whole gate set, and runs the forward (E and final
state), the backward from the saved state and the one-call
forward+backward on:

* the default path choice;
* the HBM-tiled passes with 6-qubit tiles (VQC_FORCE_PATH=hbm), from 7 qubits;
* the resident sweep with the smallest register blocks (K = 1 below 3 qubits,
  else 2), so the stage cuts differ from the default ones;
* the same circuit in complex128 with double-float arithmetic (c128df) on the
  default path.

Every output is compared with the oracle element by element at the parity
tolerances.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc  # noqa: E402
from paper_2607_11985_gb300 import workloads as wl  # noqa: E402
from tests.test_gpu_parity import TOL, C, dev, devc, maxerr  # noqa: E402

pytestmark = pytest.mark.gpu

ENV = ("VQC_FORCE_PATH", "VQC_HBM_TILE_QUBITS", "VQC_FORCE_K_FWD", "VQC_FORCE_K_BWD")


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def draw(i):
    rng = np.random.default_rng(9100 + i)
    n = int(rng.integers(1, 13))
    G = int(rng.integers(1, 120))
    dtype = "c64" if rng.random() < 0.6 else "c128"
    seed = int(rng.integers(1 << 30))
    batch = int(rng.integers(1, 7))
    with_psi0 = bool(rng.random() < 0.4)
    return n, G, dtype, seed, batch, with_psi0


def cases():
    out = []
    for i in range(32):
        n = draw(i)[0]
        out.append((i, "default"))
        if n >= 7:
            out.append((i, "hbm"))
        out.append((i, "small_k"))
        out.append((i, "df"))
    return out


@pytest.mark.parametrize("i,mode", cases())
def test_random_circuit(monkeypatch, i, mode):
    n, G, dtype, seed, batch, with_psi0 = draw(i)
    if mode == "df":
        dtype = "c128df"
    for k in ENV:
        monkeypatch.delenv(k, raising=False)
    if mode == "hbm":
        monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
        monkeypatch.setenv("VQC_HBM_TILE_QUBITS", "6")
    elif mode == "small_k":
        k = "1" if n < 3 else "2"
        monkeypatch.setenv("VQC_FORCE_K_FWD", k)
        monkeypatch.setenv("VQC_FORCE_K_BWD", k)
    w_, psi0 = wl.small_random(seed, n, G, batch=batch, dtype=dtype, with_psi0=with_psi0)
    spec = w_.spec
    c = C(spec, dtype)
    if mode == "hbm":
        assert c.info(batch)["fwd_path"] == 1
    tol = TOL[dtype]
    E_ref, st_ref = orc.forward(spec, w_.x, w_.w, psi0=psi0, want_state=True)
    dx_ref, dw_ref = orc.backward(spec, w_.x, w_.w, w_.gE, psi0=psi0)

    x = dev(w_.x, dtype) if spec.num_x else None
    w = dev(w_.w, dtype) if spec.num_w else None
    gE = dev(w_.gE, dtype)
    p0 = devc(psi0, dtype) if psi0 is not None else None
    E, st = c.forward(x, w, psi0=p0, want_state=True)
    dx, dw = c.backward(x, w, gE, psi0=p0, psi_final=st)
    Ef, dxf, dwf = c.forward_backward(x, w, gE, psi0=p0)
    torch.cuda.synchronize()

    assert maxerr(E.cpu().numpy(), E_ref) <= tol["E"]
    assert maxerr(st.cpu().numpy(), st_ref) <= tol["state"]
    assert maxerr(Ef.cpu().numpy(), E_ref) <= tol["E"]
    for got_x, got_w in ((dx, dw), (dxf, dwf)):
        if spec.num_x:
            assert maxerr(got_x.cpu().numpy(), dx_ref) <= tol["grad"]
        if spec.num_w:
            assert maxerr(got_w.cpu().numpy(), dw_ref) <= tol["grad"]
