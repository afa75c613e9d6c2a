"""Parity at the full sizes of the benchmark workloads, through the same
library calls the benchmark times.

Hard-threshold: every output of two workers over two EF iterations is
compared bit for bit with the oracle, and so is their aggregate; the
ResNet-50-sized vector at each of its three thresholds. The aggregate of all
16 ResNet-50 workers' messages is compared with the oracle's over two
iterations. Top-k: the ResNet-18- and ResNet-50-sized cases (the latter at
both Top-k fractions, 0.1 % and 1 %) are compared with the oracle over two
iterations; the larger ones are checked at iteration 0 against properties
that fix the Top-k result uniquely at any size: exactly k ascending indices,
values equal to the oracle's a at those indices, residual equal to a with
those coordinates zeroed, and every selected composite key (|a| bits, then
lower index) greater than every unselected one.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2108_00951_gb300 as efs
from paper_2108_00951_gb300 import workloads

pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import gpu_util as gu  # noqa: E402

DEV = gu.DEV


def _bf16_bits(g):
    return g.view(torch.int16).cpu().numpy().view(np.uint16)


def _host(g):
    return _bf16_bits(g) if g.dtype == torch.bfloat16 else g.cpu().numpy()


def _lambda(w, which=0):
    if w.density is not None:
        return workloads.density_lambda(w, workloads.gradient(w, 0, 0, device=DEV), w.density)
    return w.lambdas[which]


@pytest.mark.parametrize("name,dtype,which", [
    ("resnet18", torch.float32, 0), ("lstm", torch.float32, 0), ("resnet50", torch.float32, 0),
    ("resnet50", torch.float32, 1), ("resnet50", torch.float32, 2), ("vgg16", torch.float32, 0),
    ("vgg16", torch.bfloat16, 0)])
def test_full_size_hard_threshold(name, dtype, which):
    w = workloads.BY_NAME[name]
    lam = _lambda(w, which)
    workers = (0, w.n - 1)
    e_gpu = {i: torch.zeros(w.d, device=DEV) for i in workers}
    e_ref = {i: np.zeros(w.d, np.float32) for i in workers}
    idx = {i: torch.empty(w.d, dtype=torch.int32, device=DEV) for i in workers}
    val = {i: torch.empty(w.d, dtype=torch.float32, device=DEV) for i in workers}
    cnt = torch.empty(len(workers), dtype=torch.int32, device=DEV)
    for t in range(2):
        refs = []
        for slot, i in enumerate(workers):
            g = workloads.gradient(w, i, t, device=DEV, dtype=dtype)
            efs.ef_hard_threshold(g, e_gpu[i], w.gamma, lam, idx[i], val[i], cnt[slot:slot + 1])
            ri, rv, e_ref[i] = oracle.ef_hard_threshold(_host(g), e_ref[i], w.gamma, lam)
            c = int(cnt[slot].item())
            assert c == ri.size, (name, t, i, c, ri.size)
            assert 0 < c < w.d
            gu.assert_bits(idx[i][:c].cpu().numpy().view(np.uint32), ri, "idx")
            gu.assert_bits(val[i][:c].cpu().numpy(), rv, "val")
            gu.assert_bits(e_gpu[i].cpu().numpy(), e_ref[i], "e'")
            refs.append((ri, rv))
        dense = torch.empty(w.d, device=DEV)
        efs.sparse_aggregate([idx[i] for i in workers], [val[i] for i in workers], cnt, w.d, dense)
        gu.assert_bits(dense.cpu().numpy(),
                       oracle.sparse_aggregate([r[0] for r in refs], [r[1] for r in refs], w.d),
                       "aggregate")
    assert efs.ef_check_status() == efs.EF_OK


def _check_topk_properties(a, k, gi, gv, ge):
    d = a.size
    assert gi.size == k
    assert np.all(gi[1:] > gi[:-1]) and (k == 0 or gi[-1] < d)
    gu.assert_bits(gv, a[gi], "values")
    want = a.copy()
    want[gi] = 0.0
    gu.assert_bits(ge, want, "residual")
    key = ((a.view(np.uint32) & np.uint32(0x7fffffff)).astype(np.uint64) << np.uint64(32)) | \
        (~np.arange(d, dtype=np.uint32)).astype(np.uint64)
    sel = np.zeros(d, bool)
    sel[gi] = True
    if 0 < k < d:
        assert key[sel].min() > key[~sel].max()


def test_full_size_aggregate_all_workers():
    # all 16 ResNet-50-sized workers at the densest threshold (1e-4), two EF
    # iterations: every worker's message against the oracle, then the
    # aggregate of the 16 messages (with and without their tile indexes)
    w = workloads.BY_NAME["resnet50"]
    lam = w.lambdas[0]
    e_gpu = [torch.zeros(w.d, device=DEV) for _ in range(w.n)]
    e_ref = [np.zeros(w.d, np.float32) for _ in range(w.n)]
    idx = [torch.empty(w.d, dtype=torch.int32, device=DEV) for _ in range(w.n)]
    val = [torch.empty(w.d, dtype=torch.float32, device=DEV) for _ in range(w.n)]
    tiles = [torch.empty(efs.tiles_for(w.d), dtype=torch.int32, device=DEV) for _ in range(w.n)]
    cnt = torch.empty(w.n, dtype=torch.int32, device=DEV)
    for t in range(2):
        refs = []
        for i in range(w.n):
            g = workloads.gradient(w, i, t, device=DEV)
            efs.ef_hard_threshold(g, e_gpu[i], w.gamma, lam, idx[i], val[i], cnt[i:i + 1],
                                  tiles_out=tiles[i])
            ri, rv, e_ref[i] = oracle.ef_hard_threshold(g.cpu().numpy(), e_ref[i], w.gamma, lam)
            c = int(cnt[i].item())
            assert c == ri.size, (t, i, c, ri.size)
            gu.assert_bits(idx[i][:c].cpu().numpy().view(np.uint32), ri, "idx")
            gu.assert_bits(val[i][:c].cpu().numpy(), rv, "val")
            gu.assert_bits(e_gpu[i].cpu().numpy(), e_ref[i], "e'")
            refs.append((ri, rv))
        want = oracle.sparse_aggregate([r[0] for r in refs], [r[1] for r in refs], w.d)
        dense = torch.empty(w.d, device=DEV)
        efs.sparse_aggregate(idx, val, cnt, w.d, dense)
        gu.assert_bits(dense.cpu().numpy(), want, "aggregate")
        dense.fill_(float("nan"))
        efs.sparse_aggregate(idx, val, cnt, w.d, dense, tiles=tiles)
        gu.assert_bits(dense.cpu().numpy(), want, "aggregate with tile indexes")
    assert efs.ef_check_status() == efs.EF_OK


@pytest.mark.parametrize("name,which", [("resnet18", 0), ("lstm", 0), ("resnet50", 0),
                                        ("resnet50", 1), ("vgg16", 0)])
def test_full_size_topk(name, which):
    w = workloads.BY_NAME[name]
    k = w.topk_values()[which]
    idx = torch.empty(k, dtype=torch.int32, device=DEV)
    val = torch.empty(k, dtype=torch.float32, device=DEV)
    cnt = torch.empty(1, dtype=torch.int32, device=DEV)
    e_gpu = torch.zeros(w.d, device=DEV)
    e_ref = np.zeros(w.d, np.float32)
    compare_oracle = name in ("resnet18", "resnet50")
    iterations = 2 if compare_oracle else 1
    for t in range(iterations):
        g = workloads.gradient(w, 0, t, device=DEV)
        g_host = g.cpu().numpy()
        e_before = e_ref
        efs.ef_topk(g, e_gpu, w.gamma, k, idx, val, cnt)
        assert int(cnt.item()) == k
        gi = idx.cpu().numpy().view(np.uint32)
        gv = val.cpu().numpy()
        ge = e_gpu.cpu().numpy()
        # the oracle's accumulator: hard-threshold at lambda = inf sends no
        # finite coordinate, so its residual is a itself
        _, _, a = oracle.ef_hard_threshold(g_host, e_before, w.gamma, float("inf"))
        assert np.all(np.isfinite(a))
        _check_topk_properties(a, k, gi, gv, ge)
        if compare_oracle:
            ri, rv, e_ref = oracle.ef_topk(g_host, e_before, w.gamma, k)
            gu.assert_bits(gi, ri, "idx")
            gu.assert_bits(gv, rv, "val")
            gu.assert_bits(ge, e_ref, "e'")
    assert efs.ef_check_status() == efs.EF_OK
