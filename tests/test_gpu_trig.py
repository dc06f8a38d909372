"""GPU test of the complex64 half-angle sin/cos over a wide angle range.

Complex64 table entries take sin and cos of each half-angle from a short FMA
chain (reduction by pi/2 in three parts, Taylor polynomials on [-pi/4, pi/4]);
beyond a half-angle of 65536 the reduction would no longer be exact and the
kernels call the library sincosf instead.  Closed forms pin both branches and
the boundary: on every qubit q, RY(a) then RX(b) with a = x[:, q] and b =
x[:, n + q], so that

    qubit state  RX(b) RY(a)|0> = (cb ca - i sb sa,  cb sa - i sb ca)
    <Z_q>        = cos a cos b
    dL/da        = -gE sin a cos b,   dL/db = -gE cos a sin b

with ca, sa = cos, sin(a/2) etc.  The backward also turns its gradient
accumulator through RX's full angle b with the same routine.  Angles are float32
values (as the engine sees them) from tiny to 3e7 in magnitude, both signs,
including values on either side of the switch; the closed forms are evaluated in
float64 from those float32 values.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2607_11985_gb300 import workloads as wl  # noqa: E402
from tests.test_gpu_parity import C, dev, maxerr, report  # noqa: E402

pytestmark = pytest.mark.gpu

N = 7
MAGNITUDES = [0.0, 1e-30, 1e-3, 0.3, 1.0, np.pi / 2, 2.5, np.pi, 7.0, 100.0, 500.0, 1e3, 3.1e4,
              65535.0, 131071.0, 131072.0, 131073.0, 1e5, 1.3e5, 2.6e5, 1e6, 1.2e7, 3e7]


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def angles(batch):
    rng = np.random.default_rng(4242)
    mags = np.asarray(MAGNITUDES, np.float64)
    x = np.empty((batch, 2 * N))
    for j in range(2 * N):
        m = mags[(np.arange(batch) * (j + 3) + j) % len(mags)]
        m = m * (1.0 + 1e-3 * rng.standard_normal(batch) * (m > 1e3))
        x[:, j] = np.where(rng.random(batch) < 0.5, -m, m)
    return wl._round(x, "c64")


def spec():
    s = wl.CircuitSpec(N, 2 * N, 0)
    for q in range(N):
        s.add("RY", (q,), [("x", q)]).add("RX", (q,), [("x", N + q)])
    return s


def closed_forms(x, gE):
    a, b = x[:, :N], x[:, N:]
    ca, sa, cb, sb = np.cos(a / 2), np.sin(a / 2), np.cos(b / 2), np.sin(b / 2)
    q0 = cb * ca - 1j * sb * sa          # amplitude of |0> on each qubit
    q1 = cb * sa - 1j * sb * ca          # amplitude of |1>
    B = x.shape[0]
    st = np.ones((B, 1), np.complex128)
    for q in range(N - 1, -1, -1):       # qubit q is bit q: kron(..., q1 part, q0 part)
        st = np.einsum("bi,bj->bij", st, np.stack([q0[:, q], q1[:, q]], 1)).reshape(B, -1)
    E = np.cos(a) * np.cos(b)
    dx = np.concatenate([-gE * np.sin(a) * np.cos(b), -gE * np.cos(a) * np.sin(b)], 1)
    return E, st, dx


@pytest.mark.parametrize("path", ["resident", "hbm_passes"])
def test_half_angle_trig_wide_range(monkeypatch, path):
    if path == "hbm_passes":
        monkeypatch.setenv("VQC_FORCE_PATH", "hbm")
        monkeypatch.setenv("VQC_HBM_TILE_QUBITS", "6")
    B = 3 * len(MAGNITUDES)
    x = angles(B)
    gE = wl._round(np.random.default_rng(7).standard_normal((B, N)), "c64")
    E_ref, st_ref, dx_ref = closed_forms(x, gE)
    c = C(spec(), "c64")
    info = c.info(B)
    assert info["fwd_path"] == (1 if path == "hbm_passes" else 0)
    xd, gd = dev(x, "c64"), dev(gE, "c64")
    E, st = c.forward(xd, None, want_state=True)
    dx, _ = c.backward(xd, None, gd, psi_final=st)
    Ef, dxf, _ = c.forward_backward(xd, None, gd)
    torch.cuda.synchronize()
    errs = dict(state=maxerr(st.cpu().numpy(), st_ref), E=maxerr(E.cpu().numpy(), E_ref),
                dx=maxerr(dx.cpu().numpy(), dx_ref), E_fused=maxerr(Ef.cpu().numpy(), E_ref),
                dx_fused=maxerr(dxf.cpu().numpy(), dx_ref))
    report("trig_" + path, **errs)
    # the amplitudes are products of the half-angle sin/cos: each within a few
    # float32 roundings of the float64 value on the whole range
    assert errs["state"] <= 1e-6
    assert errs["E"] <= 1e-4 and errs["E_fused"] <= 1e-4
    assert errs["dx"] <= 5e-4 and errs["dx_fused"] <= 5e-4
