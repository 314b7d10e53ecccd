import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) GPU and the built CUDA library")
    config.addinivalue_line("markers", "slow: full-size parity case")


import pytest  # noqa: E402

_REPORT = []


def report(line: str) -> None:
    """Adds a line to the parity report printed at the end of the run (counts
    of boundary rows and the like, shown without -s)."""
    _REPORT.append(line)


def pytest_terminal_summary(terminalreporter):
    if _REPORT:
        terminalreporter.write_sep("-", "parity report")
        for line in _REPORT:
            terminalreporter.write_line(line)


@pytest.fixture(scope="session")
def gpu_lib():
    """Builds (if stale) and loads the CUDA library; skips without a CUDA device."""
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_20791_gb300 import binding
    from paper_2607_20791_gb300.build import build
    return binding.load_library(build())
