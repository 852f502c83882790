import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a CUDA GPU (sm_103a) and the compiled CUDA library")


@pytest.fixture(scope="session")
def cuda_device():
    """The GPU tests run only when asked for (-m gpu); without a GPU they fail
    instead of skipping, so that a missing device is never mistaken for a pass."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test selected but torch.cuda.is_available() is False")
    return torch.device("cuda:0")


def pytest_terminal_summary(terminalreporter):
    """The largest share of bf16 weights more than 1 ulp from the oracle in
    any gated check (each one in the near-cancellation set the bar allows)."""
    try:
        import parity
    except Exception:
        return
    if parity.OBSERVED["checks"]:
        terminalreporter.write_line(
            f"bf16 weights beyond 1 ulp of the oracle: at most {parity.OBSERVED['frac_beyond_1ulp']:.3g} "
            f"of the elements in {parity.OBSERVED['checks']} checks (all where the step cancels the weight)")
