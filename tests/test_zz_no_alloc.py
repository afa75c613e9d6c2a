"""The allocation-free hard-threshold entry point (ef_hard_threshold_noalloc).

It exists for callers that must not allocate device memory (their memory is
owned by their own allocator or a framework pool, or they may never block in
cudaMalloc). It is called here through the C ABI with raw device pointers and
must reproduce ef_hard_threshold bit for bit, on two calls in a row (the
second starting from the first call's residuals, so the shared scratch is
reused). This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2108_00951_gb300 as efs

pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

vp = ctypes.c_void_p


def _entry():
    lib = efs.load_library()
    fn = lib.ef_hard_threshold_noalloc
    fn.argtypes = [vp, vp, ctypes.c_float, ctypes.c_float, ctypes.c_uint64, vp, vp, vp, vp, vp]
    fn.restype = ctypes.c_int
    return fn


def _bits(t):
    return t.cpu().numpy().view(np.uint32)


@pytest.mark.parametrize("d", [1, 4097, 3 * 4096 + 17, 1_000_003])
def test_noalloc_matches_ef_hard_threshold_twice(d):
    fn = _entry()
    dev = torch.device("cuda:0")
    gen = torch.Generator().manual_seed(d)
    e_ref = (torch.randn(d, generator=gen) * 1e-3).to(dev)
    e_new = e_ref.clone()
    stream = torch.cuda.current_stream()
    for call in range(2):
        g = (torch.randn(d, generator=gen) * 1e-2).to(dev)
        gamma, lam = 0.1, 1.5e-3
        idx_a = torch.full((d,), -1, dtype=torch.int32, device=dev)
        val_a = torch.zeros(d, device=dev)
        cnt_a = torch.zeros(1, dtype=torch.int32, device=dev)
        efs.ef_hard_threshold(g, e_ref, gamma, lam, idx_a, val_a, cnt_a)
        idx_b = torch.full((d,), -1, dtype=torch.int32, device=dev)
        val_b = torch.zeros(d, device=dev)
        cnt_b = torch.full((1,), 7, dtype=torch.int32, device=dev)
        status = torch.full((1,), 99, dtype=torch.int32, device=dev)
        rc = fn(vp(g.data_ptr()), vp(e_new.data_ptr()), gamma, lam, d, vp(idx_b.data_ptr()),
                vp(val_b.data_ptr()), vp(cnt_b.data_ptr()), vp(status.data_ptr()),
                vp(stream.cuda_stream))
        assert rc == efs.EF_OK
        torch.cuda.synchronize()
        assert int(status.item()) == 0, "device-side error bits %d" % int(status.item())
        c = int(cnt_a.item())
        assert int(cnt_b.item()) == c, (call, c, int(cnt_b.item()))
        assert np.array_equal(_bits(idx_a[:c]), _bits(idx_b[:c]))
        assert np.array_equal(_bits(val_a[:c]), _bits(val_b[:c]))
        assert np.array_equal(_bits(e_ref), _bits(e_new))


def test_noalloc_rejects_sizes_beyond_its_scratch():
    fn = _entry()
    # rejected by the size check before any pointer is touched or work launched
    rc = fn(vp(16), vp(32), 0.1, 1e-3, (1 << 28) + 1, vp(48), vp(64), vp(80), vp(0), vp(0))
    assert rc == efs.EF_ERR_INVALID_ARG
