"""vqc_stage_apply: one batch-shared 5-qubit stage on the tensor cores
(tcgen05, tf32 split into high and low parts, three products accumulated in
FP32) and on the FP32 units, against the oracle applying the same five gates.

The factors are U3 gates with random angles on qubits 0..4 (the oracle's own
gate matrices), the states random normalised complex64 rows; the oracle
applies the gates `repeats` times to the same states (psi0) in complex128.
Covered: one and several applications, in place, row counts below and above
one 128-row tile, and the tensor-core wait check afterwards.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc  # noqa: E402
from paper_2607_11985_gb300 import workloads as wl  # noqa: E402
from tests.test_gpu_parity import maxerr, report  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def case(seed, n, B):
    rng = np.random.default_rng(seed)
    th = rng.uniform(-np.pi, np.pi, (5, 3))
    factors = np.stack([orc.gate_matrix("U3", t) for t in th])
    z = rng.standard_normal((B, 1 << n)) + 1j * rng.standard_normal((B, 1 << n))
    z /= np.linalg.norm(z, axis=1, keepdims=True)
    return th, factors, z.astype(np.complex64)


def reference(th, n, psi0, repeats):
    spec = wl.CircuitSpec(n, 0, 0)
    for _ in range(repeats):
        for q in range(5):
            spec.add("U3", (q,), [("c", th[q, 0]), ("c", th[q, 1]), ("c", th[q, 2])])
    return orc.forward(spec, None, None, psi0=psi0.astype(np.complex128), want_state=True)[1]


@pytest.mark.parametrize("method", [0, 1])
@pytest.mark.parametrize("n,B,repeats", [(12, 24, 1), (12, 24, 3), (5, 3, 2), (6, 3, 1), (9, 5, 4)])
def test_stage_against_oracle(method, n, B, repeats):
    from paper_2607_11985_gb300 import binding as Bd
    th, factors, z = case(900 + 7 * n + B + repeats, n, B)
    ref = reference(th, n, z, repeats)
    src = torch.tensor(z, device="cuda")
    dst = torch.full_like(src, float("nan"))
    s = torch.cuda.current_stream().cuda_stream
    Bd.vqc_stage_apply(method, B, n, factors, src.data_ptr(), dst.data_ptr(), repeats, s)
    Bd.vqc_sync_check(s)
    err = maxerr(dst.cpu().numpy(), ref)
    report("stage_m%d_n%d_B%d_r%d" % (method, n, B, repeats), state=err)
    assert err <= 1e-5
    Bd.vqc_stage_apply(method, B, n, factors, src.data_ptr(), src.data_ptr(), repeats, s)   # in place
    Bd.vqc_sync_check(s)
    assert maxerr(src.cpu().numpy(), ref) <= 1e-5


def test_stage_argument_errors():
    from paper_2607_11985_gb300 import binding as Bd
    f = np.stack([np.eye(2)] * 5)
    x = torch.zeros(2, 1 << 6, dtype=torch.complex64, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    for call in (lambda: Bd.vqc_stage_apply(2, 2, 6, f, x.data_ptr(), x.data_ptr(), 1, s),
                 lambda: Bd.vqc_stage_apply(1, 2, 4, f, x.data_ptr(), x.data_ptr(), 1, s),
                 lambda: Bd.vqc_stage_apply(1, 2, 6, f, x.data_ptr() + 8, x.data_ptr(), 1, s),
                 lambda: Bd.vqc_stage_apply(0, 2, 6, f, x.data_ptr(), x.data_ptr(), 0, s)):
        with pytest.raises(Bd.VQCError) as e:
            call()
        assert e.value.status == 1
    Bd.vqc_sync_check(s)
