import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: full-size parity cases")


@pytest.fixture(params=["chunks", "groups"])
def stream_kernel(request):
    """Runs a streaming-pass test (hard-threshold, Top-k or layer-wise Top-k)
    with each streaming kernel: the static-chunk
    kernel and the claimed-group look-back kernel (by default the library
    picks by size; small test inputs would reach only the first)."""
    import paper_2108_00951_gb300 as efs
    efs.ef_test_set_stream_kernel({"chunks": 1, "groups": 2}[request.param])
    try:
        yield request.param
    finally:
        efs.ef_test_set_stream_kernel(0)


@pytest.fixture(params=["chunks", "groups", "shallow"])
def ht_stream_kernel(request):
    """Runs a hard-threshold test with each of its streaming kernels: static
    chunks, claimed groups, and claimed groups with the shallower ring and
    larger pair buffers that dense calls use."""
    import paper_2108_00951_gb300 as efs
    efs.ef_test_set_stream_kernel({"chunks": 1, "groups": 2, "shallow": 3}[request.param])
    try:
        yield request.param
    finally:
        efs.ef_test_set_stream_kernel(0)
