"""The allocation-free hard-threshold entry point (ef_hard_threshold_noalloc).

It exists for callers that must not allocate device memory (their memory is
owned by their own allocator or a framework pool, or they may never block in
cudaMalloc). It is called here through the C ABI with raw device pointers and
must reproduce ef_hard_threshold and the CPU oracle bit for bit, on two calls
in a row (the second starting from the first call's residuals, so the shared
scratch is reused), at aligned and misaligned bases; it must allocate no
device memory once the library is loaded; its status word must report a
bounded wait that ran out; and its per-call tag must survive its wrap-around.
This file is collected last on purpose.
"""
import ctypes
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import oracle
import paper_2108_00951_gb300 as efs

pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import gpu_util as gu  # noqa: E402

vp = ctypes.c_void_p
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _entry():
    lib = efs.load_library()
    fn = lib.ef_hard_threshold_noalloc
    fn.argtypes = [vp, vp, ctypes.c_float, ctypes.c_float, ctypes.c_uint64, vp, vp, vp, vp, vp]
    fn.restype = ctypes.c_int
    return fn


def _bits(t):
    return t.cpu().numpy().view(np.uint32)


def _noalloc(fn, g, e, gamma, lam, idx, val, cnt, status, stream):
    return fn(vp(g.data_ptr()), vp(e.data_ptr()), gamma, lam, e.numel(), vp(idx.data_ptr()),
              vp(val.data_ptr()), vp(cnt.data_ptr()),
              vp(status.data_ptr() if status is not None else 0), vp(stream.cuda_stream))


def _offset_copy(x: torch.Tensor, offset: int) -> torch.Tensor:
    """A copy of x whose base lies `offset` floats past an allocation."""
    buf = torch.empty(x.numel() + offset, dtype=x.dtype, device=x.device)
    view = buf[offset:offset + x.numel()]
    view.copy_(x)
    return view


@pytest.mark.parametrize("offset", [0, 1])
@pytest.mark.parametrize("d", [1, 4097, 3 * 4096 + 17, 1_000_003])
def test_noalloc_matches_ef_hard_threshold_and_oracle_twice(d, offset):
    fn = _entry()
    dev = torch.device("cuda:0")
    gen = torch.Generator().manual_seed(d + offset)
    e0 = (torch.randn(d, generator=gen) * 1e-3)
    e_ref = e0.to(dev)                      # the regular entry's error memory
    e_new = _offset_copy(e0.to(dev), offset)  # the allocation-free entry's
    e_host = e0.numpy().copy()              # the oracle's
    stream = torch.cuda.current_stream()
    for call in range(2):
        g_host = (torch.randn(d, generator=gen) * 1e-2)
        g = g_host.to(dev)
        g_off = _offset_copy(g, offset)
        gamma, lam = 0.1, 1.5e-3
        idx_a = torch.full((d,), -1, dtype=torch.int32, device=dev)
        val_a = torch.zeros(d, device=dev)
        cnt_a = torch.zeros(1, dtype=torch.int32, device=dev)
        efs.ef_hard_threshold(g, e_ref, gamma, lam, idx_a, val_a, cnt_a)
        idx_b = torch.full((d,), -1, dtype=torch.int32, device=dev)
        val_b = torch.zeros(d, device=dev)
        cnt_b = torch.full((1,), 7, dtype=torch.int32, device=dev)
        status = torch.full((1,), 99, dtype=torch.int32, device=dev)
        rc = _noalloc(fn, g_off, e_new, gamma, lam, idx_b, val_b, cnt_b, status, stream)
        assert rc == efs.EF_OK
        torch.cuda.synchronize()
        assert int(status.item()) == 0, "device-side error bits %d" % int(status.item())
        ri, rv, e_host = oracle.ef_hard_threshold(g_host.numpy(), e_host, gamma, lam)
        c = int(cnt_b.item())
        assert c == ri.size == int(cnt_a.item()), (call, c, ri.size, int(cnt_a.item()))
        gu.assert_bits(_bits(idx_b[:c]), ri, "idx vs oracle")
        gu.assert_bits(val_b[:c].cpu().numpy(), rv, "val vs oracle")
        gu.assert_bits(e_new.cpu().numpy(), e_host, "e' vs oracle")
        assert np.array_equal(_bits(idx_a[:c]), _bits(idx_b[:c]))
        assert np.array_equal(_bits(val_a[:c]), _bits(val_b[:c]))
        assert np.array_equal(_bits(e_ref), _bits(e_new))


def test_noalloc_allocates_no_device_memory():
    fn = _entry()
    dev = torch.device("cuda:0")
    d = 1 << 20
    g = torch.randn(d, device=dev) * 1e-2
    e = torch.zeros(d, device=dev)
    idx = torch.empty(d, dtype=torch.int32, device=dev)
    val = torch.empty(d, device=dev)
    cnt = torch.zeros(1, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    # one call first: loading the library's device code (which holds the
    # fixed scratch) may itself take device memory, once
    assert _noalloc(fn, g, e, 0.1, 1e-3, idx, val, cnt, status,
                    torch.cuda.current_stream()) == efs.EF_OK
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    side = torch.cuda.Stream()   # a stream the library has never seen
    for _ in range(3):
        assert _noalloc(fn, g, e, 0.1, 1e-3, idx, val, cnt, status, side) == efs.EF_OK
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, (free0, free1)
    assert int(status.item()) == 0


def test_noalloc_status_reports_a_wait_that_ran_out():
    fn = _entry()
    dev = torch.device("cuda:0")
    d = 40 * 4096 + 3
    g = torch.randn(d, device=dev) * 1e-2
    e = torch.zeros(d, device=dev)
    idx = torch.empty(d, dtype=torch.int32, device=dev)
    val = torch.empty(d, device=dev)
    cnt = torch.zeros(1, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()
    assert efs.ef_check_status() == efs.EF_OK
    efs.ef_test_set_lookback_fault(5, 2000)   # tile 5 never publishes; waits end after ~2 ms
    try:
        assert _noalloc(fn, g, e, 0.1, 1e-3, idx, val, cnt, status, stream) == efs.EF_OK
        torch.cuda.synchronize()
    finally:
        efs.ef_test_set_lookback_fault(-1)
    assert int(status.item()) & 1, "the timeout bit is not set: %d" % int(status.item())
    assert efs.ef_check_status() == efs.EF_OK   # the regular entries' status is not touched
    # a healthy call afterwards: status 0 and the regular entry's bits
    g2 = torch.randn(d, device=dev) * 1e-2
    e_a = torch.randn(d, device=dev) * 1e-3
    e_b = e_a.clone()
    idx_a = torch.empty(d, dtype=torch.int32, device=dev)
    val_a = torch.empty(d, device=dev)
    cnt_a = torch.zeros(1, dtype=torch.int32, device=dev)
    efs.ef_hard_threshold(g2, e_a, 0.1, 1e-3, idx_a, val_a, cnt_a)
    assert _noalloc(fn, g2, e_b, 0.1, 1e-3, idx, val, cnt, status, stream) == efs.EF_OK
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    c = int(cnt_a.item())
    assert int(cnt.item()) == c
    assert np.array_equal(_bits(idx_a[:c]), _bits(idx[:c]))
    assert np.array_equal(_bits(val_a[:c]), _bits(val[:c]))
    assert np.array_equal(_bits(e_a), _bits(e_b))


_WRAP_SCRIPT = r"""
import sys
sys.path.insert(0, %(root)r)
sys.path.insert(0, %(tests)r)
import ctypes
import numpy as np
import torch
import paper_2108_00951_gb300 as efs
import test_zz_no_alloc as t
fn = t._entry()
dev = torch.device("cuda:0")
d = 9 * 4096 + 5
gen = torch.Generator().manual_seed(11)
e_a = (torch.randn(d, generator=gen) * 1e-3).to(dev)
e_b = e_a.clone()
stream = torch.cuda.current_stream()
for call in range(4):      # tags 2^30-2, 2^30-1, then the wrap: 1, 2
    g = (torch.randn(d, generator=gen) * 1e-2).to(dev)
    out = [torch.empty(d, dtype=torch.int32, device=dev), torch.empty(d, device=dev),
           torch.zeros(1, dtype=torch.int32, device=dev)]
    ref = [torch.empty(d, dtype=torch.int32, device=dev), torch.empty(d, device=dev),
           torch.zeros(1, dtype=torch.int32, device=dev)]
    status = torch.full((1,), 9, dtype=torch.int32, device=dev)
    efs.ef_hard_threshold(g, e_a, 0.1, 1.5e-3, *ref)
    assert t._noalloc(fn, g, e_b, 0.1, 1.5e-3, *out, status, stream) == efs.EF_OK
    torch.cuda.synchronize()
    assert int(status.item()) == 0, (call, int(status.item()))
    c = int(ref[2].item())
    assert int(out[2].item()) == c, (call, c, int(out[2].item()))
    assert np.array_equal(t._bits(ref[0][:c]), t._bits(out[0][:c])), call
    assert np.array_equal(t._bits(ref[1][:c]), t._bits(out[1][:c])), call
    assert np.array_equal(t._bits(e_a), t._bits(e_b)), call
print("wrap ok")
"""


def test_noalloc_tag_wraps_around():
    # a fresh process whose first call starts the per-call tag three short of
    # its wrap (the testing aid EF_NOALLOC_FIRST_EPOCH), so four calls cross it
    env = dict(os.environ, EF_NOALLOC_FIRST_EPOCH=str((1 << 30) - 3))
    script = _WRAP_SCRIPT % {"root": ROOT, "tests": os.path.join(ROOT, "tests")}
    r = subprocess.run([sys.executable, "-c", script], env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0 and "wrap ok" in r.stdout, r.stdout + r.stderr


def test_noalloc_rejects_sizes_beyond_its_scratch():
    fn = _entry()
    # rejected by the size check before any pointer is touched or work launched
    rc = fn(vp(16), vp(32), 0.1, 1e-3, (1 << 28) + 1, vp(48), vp(64), vp(80), vp(0), vp(0))
    assert rc == efs.EF_ERR_INVALID_ARG
