"""GPU: vqc_fma_peak, the measured arithmetic ceiling of the sweeps.

The packed-FP32 rate must lie near the unit-count figure (SMs x 128 lanes x 2
flops x clock: between a third of it, for a slow clock under load, and a
little above it); the FP64 rate must be positive and below the FP32 one; bad
arguments are rejected before anything runs.
"""
import ctypes

import pytest

torch = pytest.importorskip("torch")

from paper_2607_11985_gb300 import binding as B  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def cuda_ready():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def test_fma_rates_are_plausible():
    props = torch.cuda.get_device_properties(0)
    clock_mhz = 2070.0   # the part's maximum SM clock; the measured rate may run below it
    derived = props.multi_processor_count * 128 * 2 * clock_mhz * 1e6 / 1e12
    fp32 = B.vqc_fma_peak(0)
    fp64 = B.vqc_fma_peak(1)
    assert derived / 3 < fp32 < 1.1 * derived, (fp32, derived)
    assert 0 < fp64 < fp32, (fp64, fp32)


def test_fma_peak_argument_errors():
    out = ctypes.c_double(1.0)
    assert B.lib().vqc_fma_peak(7, ctypes.byref(out)) == 1   # VQC_ERR_INVALID_ARG
    assert B.lib().vqc_fma_peak(0, None) == 1   # VQC_ERR_INVALID_ARG
