import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


@pytest.fixture(scope="session")
def cuda_lib():
    """The loaded C-ABI library; GPU tests fail loudly when it is missing."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test run without a CUDA device")
    from paper_2608_03276_gb300 import binding
    return binding.load()


def pytest_terminal_summary(terminalreporter):
    """Worst relative score error and near-tie kept-set differences of every
    parity test that compared scores with the oracle (tests/parity.py)."""
    from tests import parity
    tr = terminalreporter
    if parity.REPORTS:
        tr.section("method-level figures (reported)")
        for line in parity.REPORTS:
            tr.write_line(line)
    if not parity.STATS:
        return
    tr.section("parity margins (bar: rel err <= 2e-3; kept sets equal outside near-ties)")
    worst = 0.0
    for test, st in sorted(parity.STATS.items()):
        worst = max(worst, st["max_rel"])
        tr.write_line(f"{test}: max rel err {st['max_rel']:.2e} over {st['units']} "
                      f"(document, head) rows; {st['near_tie_diffs']} near-tie kept-set differences")
    tr.write_line(f"worst over all tests: {worst:.2e}")
