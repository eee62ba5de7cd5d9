import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")


def read_golden(name):
    """key/value or bare-value lines of a golden fixture, comments dropped."""
    out = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                out.append(line.split())
    return out


@pytest.fixture(scope="session")
def stlib():
    """The built library (compiled here with nvcc if missing or stale)."""
    import paper_2608_13667_gb300 as stpkg
    stpkg.build()
    return stpkg


@pytest.fixture(autouse=True)
def _release_device_memory(request):
    """Return pooled device memory between GPU tests (the full-size workloads
    each hold tens of GB)."""
    yield
    if request.node.get_closest_marker("gpu"):
        import gc
        gc.collect()
        try:
            import torch
            if torch.cuda.is_available():
                torch.cuda.empty_cache()
        except ImportError:
            pass


@pytest.fixture(scope="session")
def oracle_jobs():
    """A pool of float64-oracle worker processes (spawned), shared by the
    full-size parity tests."""
    from oracle_jobs import OracleJobs
    jobs = OracleJobs()
    yield jobs
    jobs.close()
