"""Runs after the parity tests: with a library built with device-side checks (SC_BUILD_DEBUG=1 at
build time), no computed index, copy size or alignment failed during any of the
GPU tests before it."""
import pytest

pytestmark = pytest.mark.gpu


def test_no_device_check_failed_in_the_session():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2405_19261_gb300 import binding
    line = binding.debug_line()
    if line == -1:
        pytest.skip("the library was built without the device-side checks")
    assert line == 0, f"a device-side check failed at sc_verify.cu:{line}"
