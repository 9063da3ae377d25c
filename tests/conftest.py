import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a CUDA GPU (sm_103a); run with -m gpu")
    config.addinivalue_line(
        "markers", "slow: full-size parity case (minutes)")


@pytest.fixture(scope="session")
def cuda_device():
    """The GPU the parity tests run on; a GPU test without one is an error,
    not a skip."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test collected on a machine without CUDA")
    return torch.device("cuda:0")


def pytest_collection_modifyitems(config, items):
    """Every GPU test runs under a wall-clock limit (pytest-timeout, where it
    is installed): a test that stops making progress ends its process instead
    of holding the GPU. The kernels' own waits are bounded well below it."""
    if not config.pluginmanager.hasplugin("timeout"):
        return
    for item in items:
        if item.get_closest_marker("gpu") is not None and item.get_closest_marker("timeout") is None:
            item.add_marker(pytest.mark.timeout(1200, method="thread"))


def pytest_terminal_summary(terminalreporter):
    """The worst parity figure of every buffer, per test that compared the
    CUDA path with the oracle: printed every run, so a drift shows before it
    crosses a bar. Floored metrics are asserted; ``*_raw_ulp_all`` (bf16
    code points over all elements), ``*_under_floor`` (elements under the
    floor) and ``*_norm`` (normwise) are reported beside them."""
    pu = sys.modules.get("parity_util")
    if pu is None or not getattr(pu, "WORST", None):
        return
    tr = terminalreporter
    tr.section("parity (worst over each test's comparisons)")
    for test, errs in sorted(pu.WORST.items()):
        cells = []
        for key in sorted(errs):
            v = errs[key]
            cells.append(f"{key}={v}" if isinstance(v, int) else f"{key}={v:.2e}")
        tr.write_line(f"{test.split('::', 1)[-1]}: " + " ".join(cells))
