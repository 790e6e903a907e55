import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs on the GB300 box)")


@pytest.fixture(scope="session")
def orc():
    import oracle
    oracle.build()
    return oracle


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """The bf16-mode distances the parity tests measured: per tensor kind,
    the largest entrywise error of the GPU against the exact oracle and of
    the oracle's own bf16-storage model against its exact mode."""
    mod = sys.modules.get("parity")
    stats = getattr(mod, "STATS", None) if mod else None
    if not stats:
        return
    terminalreporter.section("bf16 mode against the exact oracle (largest entrywise relative error)")
    for kind, (e_gpu, e_model) in sorted(stats.items()):
        terminalreporter.write_line(f"{kind:14s} GPU {e_gpu:.3g}   oracle bf16-storage model {e_model:.3g}")
