import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: full-size workloads")


def pytest_collection_modifyitems(config, items):
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA GPU in this environment")
    for it in items:
        if "gpu" in it.keywords:
            it.add_marker(skip)


@pytest.fixture(scope="session")
def ctx():
    import torch
    from paper_2607_21686_gb300 import build, pcs
    build.build()
    torch.cuda.set_device(0)
    c = pcs.Context(0)
    yield c
    c.close()


@pytest.fixture(scope="session")
def dev():
    import torch
    return torch.device("cuda:0")


@pytest.fixture(autouse=True)
def _device_errors_are_failures(request):
    """After every GPU test, errors recorded by kernels (an index out of
    range, a bounded wait that gave up) surface through pcs_sync."""
    yield
    for name in ("ctx", "ctx_reg"):
        if name in request.fixturenames:
            request.getfixturevalue(name).sync()
