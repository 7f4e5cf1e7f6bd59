import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
_TESTS = os.path.dirname(os.path.abspath(__file__))
if _TESTS not in sys.path:
    sys.path.insert(0, _TESTS)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: full-size workloads")


def pytest_collection_modifyitems(config, items):
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


@pytest.fixture(scope="session")
def aatc():
    """The built library's Python binding (builds libaatc.so in-tree if it is missing)."""
    from paper_2608_14191_gb300 import build as b
    b.build()
    import paper_2608_14191_gb300 as m
    m.load()
    return m


@pytest.fixture(scope="session")
def oracle_pool():
    """Spawned worker processes for the oracle side of the full-size parity checks (numpy only;
    spawn, so no worker inherits this process's CUDA state)."""
    import multiprocessing as mp
    n = max(1, min(16, len(os.sched_getaffinity(0))))
    pool = mp.get_context("spawn").Pool(n)
    try:
        yield pool
    finally:
        pool.close()
        pool.join()


def pytest_terminal_summary(terminalreporter):
    try:
        import harness
    except Exception:  # pragma: no cover
        return
    rows = harness.NearThreshold.rows
    if not rows:
        return
    terminalreporter.section("near-threshold codes (one level off, |h/Delta - (k + 1/2)| <= 1e-4 rel)")
    for name, (mis, tot, near) in sorted(rows.items()):
        terminalreporter.write_line(f"{name}: {mis} of {tot} codes ({mis / max(tot, 1):.2e}); "
                                    f"{near} codes near a threshold in the oracle")
