"""GB300-native error-feedback gradient sparsification (arXiv:2108.00951).

The hot path of the paper's method — one error-feedback compression step per
worker (a = e + gamma g, hard-threshold or Top-k selection, ordered
compaction into (index, value) pairs, residual e <- a - C(a)) and the
worker-ordered sparse aggregation — runs in hand-written CUDA kernels for
sm_103a behind the C ABI of ``include/efsparse.h``. This package is the thin
Python binding of that library (torch supplies device memory and streams)
plus the seeded synthetic workloads used by the tests and the benchmark.
"""
from ._binding import (  # noqa: F401
    EF_ERR_BAD_INPUT,
    EF_ERR_CUDA,
    EF_ERR_INVALID_ARG,
    EF_ERR_NO_MEMORY,
    EF_ERR_TIMEOUT,
    EF_OK,
    TILE,
    EfError,
    ef_check_status,
    ef_hard_threshold,
    ef_scaled_round,
    ef_kernel_launches,
    ef_test_set_lookback_fault,
    ef_test_set_stream_kernel,
    ef_topk,
    ef_topk_layerwise,
    ef_workspace_release,
    library_path,
    int_aggregate,
    load_library,
    sparse_aggregate,
    sparse_aggregate_apply,
    status_string,
    tiles_for,
)
