"""Failure detection without faulting the GPU: bounded device waits that run
out latch EF_ERR_TIMEOUT and finish; malformed sparse input is skipped and
latched as EF_ERR_BAD_INPUT; in every case the context stays usable."""
import numpy as np
import pytest
import torch

import oracle
import paper_2108_00951_gb300 as efs

pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import gpu_util as gu  # noqa: E402


def _inputs(d):
    rng = np.random.default_rng(99)
    return (rng.standard_normal(d) * 1e-2).astype(np.float32), \
        (rng.standard_normal(d) * 1e-3).astype(np.float32)


def _healthy_call_matches_oracle(g, e):
    ri, rv, re_ = oracle.ef_hard_threshold(g, e, 0.1, 1e-3)
    gi, gv, ge = gu.ht(g, e, 0.1, 1e-3)
    gu.assert_bits(gi, ri, "idx")
    gu.assert_bits(gv, rv, "val")
    gu.assert_bits(ge, re_, "e'")
    assert efs.ef_check_status() == efs.EF_OK


@pytest.mark.usefixtures("stream_kernel")
@pytest.mark.parametrize("method", ["ht", "topk"])
def test_lookback_wait_runs_out_and_recovers(method):
    d = 40 * 4096 + 9
    g, e = _inputs(d)
    assert efs.ef_check_status() == efs.EF_OK
    efs.ef_test_set_lookback_fault(5, 2000)      # tile 5 never publishes; waits end after 2 ms
    try:
        if method == "ht":
            gu.ht(g, e, 0.1, 1e-3)
        else:
            gu.topk(g, e, 0.1, 1000)
        status = efs.ef_check_status()
    finally:
        efs.ef_test_set_lookback_fault(-1)
    assert status == efs.EF_ERR_TIMEOUT
    assert efs.ef_check_status() == efs.EF_OK     # cleared once reported
    _healthy_call_matches_oracle(g, e)


def test_aggregate_malformed_input_is_latched_not_faulting():
    d = 10_000
    good = np.array([1, 50, 9000], np.uint32)
    unsorted = np.array([9000, 5, 4097, 3], np.uint32)
    out_of_range = np.array([2, 9999, 10_000, 4_000_000_000], np.uint32)
    vals = [np.ones(3, np.float32), np.ones(4, np.float32), np.ones(4, np.float32)]
    out = gu.aggregate([good, unsorted, out_of_range], vals, d)
    assert np.all(np.isfinite(out))
    assert efs.ef_check_status() == efs.EF_ERR_BAD_INPUT
    assert efs.ef_check_status() == efs.EF_OK
    g, e = _inputs(5000)
    _healthy_call_matches_oracle(g, e)


def test_invalid_arguments_launch_nothing():
    before = efs.ef_kernel_launches()
    x = torch.zeros(100, device=gu.DEV)
    i = torch.zeros(100, dtype=torch.int32, device=gu.DEV)
    with pytest.raises(efs.EfError) as err:
        efs.ef_hard_threshold(x, x.clone(), 0.1, -1.0, i, x.clone(), i[:1])
    assert err.value.status == efs.EF_ERR_INVALID_ARG
    i101 = torch.zeros(101, dtype=torch.int32, device=gu.DEV)
    with pytest.raises(efs.EfError) as err:        # k > d
        efs.ef_topk(x, x.clone(), 0.1, 101, i101, torch.zeros(101, device=gu.DEV), i[:1])
    assert err.value.status == efs.EF_ERR_INVALID_ARG
    with pytest.raises(efs.EfError):       # output aliases the error memory
        efs.ef_hard_threshold(x, x, 0.1, 1e-3, i, x[:100], i[:1])
    assert efs.ef_kernel_launches() == before
