import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


@pytest.fixture(scope="session")
def oracle():
    from oracle import oracle as o
    o.lib()
    return o


def pytest_terminal_summary(terminalreporter):
    """Report what the parity protocol excused in this run: decisions that
    fell within the margin of their boundary, and prefixes (trees) excluded
    because such a decision went the other way on the GPU."""
    from tests.parity import SESSION
    if SESSION["calls"] == 0 and SESSION["trees"] == 0:
        return
    terminalreporter.write_line(
        "parity protocol: %d linear calls, %d prefixes, %d near-boundary decisions, "
        "%d paths with a flipped decision, %d prefixes checked conditionally, %d excluded; "
        "%d trees, %d trees excluded" % (
            SESSION["calls"], SESSION["prefixes"], SESSION["near_boundary_decisions"],
            SESSION["diverged_paths"], SESSION["conditional_prefixes"],
            SESSION["excluded_prefixes"], SESSION["trees"], SESSION["excluded_trees"]))
