"""GPU parity of the fused exchange-and-update step (sparse_aggregate_apply)
against the CPU oracle, bit for bit: Algorithm 1's x <- x - mean, and the
Appendix's EF SGD with momentum by gradient compression
(m <- fmaf(mu, m, Delta'), x <- fmaf(-lr, Delta' + m, x)).

Cases: 1..16 workers, ragged sizes across several 4096-coordinate tiles,
empty and dense lists, misaligned x and m, NaN and infinities in the state,
a multi-iteration EF-SGD loop whose messages come from the library's own
compression, and the ResNet-18-sized workload.
"""
import zlib

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


def _rng(*key):
    return np.random.default_rng(zlib.crc32(repr(key).encode()))


def _lists(n, d, density, seed):
    rng = _rng("upd", n, d, seed)
    idx, val = [], []
    for _ in range(n):
        i = np.nonzero(rng.random(d) < density)[0].astype(np.uint32)
        idx.append(i)
        val.append(rng.standard_normal(i.size).astype(np.float32))
    return idx, val


def _apply(idx, val, d, alpha, x, m=None, mu=0.0, lr=0.0, off=0):
    idx_t = [gu.to_dev(np.asarray(i, np.uint32).view(np.int32)) if len(i) else
             torch.zeros(1, dtype=torch.int32, device=DEV) for i in idx]
    val_t = [gu.to_dev(np.asarray(v, np.float32)) if len(v) else
             torch.zeros(1, dtype=torch.float32, device=DEV) for v in val]
    counts = torch.tensor([len(i) for i in idx], dtype=torch.int32, device=DEV)
    xd = gu.to_dev(x, off)
    md = None if m is None else gu.to_dev(m, off)
    efs.sparse_aggregate_apply(idx_t, val_t, counts, d, alpha, xd, md, mu, lr)
    torch.cuda.synchronize()
    return xd.cpu().numpy(), None if md is None else md.cpu().numpy()


def _check(idx, val, d, alpha, x, m=None, mu=0.0, lr=0.0, off=0, what=""):
    gx, gm = _apply(idx, val, d, alpha, x, m, mu, lr, off)
    rx, rm = oracle.sparse_aggregate_apply(idx, val, d, alpha, x, m, mu, lr)
    gu.assert_bits(gx, rx, what + " x")
    if m is not None:
        gu.assert_bits(gm, rm, what + " m")
    assert efs.ef_check_status() == efs.EF_OK


@pytest.mark.parametrize("momentum", [False, True])
@pytest.mark.parametrize("n", [1, 4, 8, 16])
@pytest.mark.parametrize("d", [5, 4096, 4097, 100_003])
def test_apply_random(d, n, momentum):
    rng = _rng("state", d, n)
    for density in (0.001, 0.05, 1.0):
        idx, val = _lists(n, d, density, 1)
        x = rng.standard_normal(d).astype(np.float32)
        m = (rng.standard_normal(d) * 0.1).astype(np.float32) if momentum else None
        _check(idx, val, d, 1.0 / n, x, m, 0.9, 0.05, what="n=%d d=%d rho=%g" % (n, d, density))


@pytest.mark.parametrize("off", [1, 3])
def test_apply_misaligned_state(off):
    d = 3 * 4096 + 77
    idx, val = _lists(5, d, 0.02, 2)
    rng = _rng("mis", off)
    x = rng.standard_normal(d).astype(np.float32)
    m = rng.standard_normal(d).astype(np.float32)
    _check(idx, val, d, 0.2, x, m, 0.5, 0.1, off=off, what="momentum off=%d" % off)
    _check(idx, val, d, 0.2, x, None, off=off, what="sgd off=%d" % off)


def test_apply_special_values():
    d = 4096 + 9
    idx = [np.array([0, 1, 2, 3, 4, 4100], np.uint32)] * 2
    val = [np.array([np.inf, -np.inf, np.nan, 1e38, -0.0, 2.0], np.float32),
           np.array([1.0, np.inf, 0.0, 1e38, -0.0, -2.0], np.float32)]
    x = np.zeros(d, np.float32)
    x[5] = np.nan
    x[6] = np.inf
    m = np.zeros(d, np.float32)
    m[7] = -np.inf
    _check(idx, val, d, 0.5, x, m, 0.9, 0.1, what="special momentum")
    _check(idx, val, d, 0.5, x, None, what="special sgd")


def test_apply_empty_lists_and_zero_scale():
    d = 10_000
    idx, val = _lists(4, d, 0.01, 3)
    idx[1], val[1] = idx[1][:0], val[1][:0]
    x = np.linspace(-1, 1, d).astype(np.float32)
    m = np.linspace(1, -1, d).astype(np.float32)
    _check(idx, val, d, 0.0, x, m, 0.9, 0.1, what="alpha 0")
    _check(idx, val, d, 0.25, x, m, 0.0, 0.0, what="mu 0 lr 0")


def test_ef_sgd_loop_with_library_messages():
    """Ten EF-SGD iterations of four workers: hard-threshold messages from the
    library, then the momentum update; every state bit-equal to the oracle's."""
    w = workloads.BY_NAME["lr"]
    d, n, lam = w.d, w.n, w.lambdas[0]
    e_gpu = [torch.zeros(d, device=DEV) for _ in range(n)]
    e_ref = [np.zeros(d, np.float32) for _ in range(n)]
    x_gpu, m_gpu = torch.zeros(d, device=DEV), torch.zeros(d, device=DEV)
    x_ref, m_ref = np.zeros(d, np.float32), np.zeros(d, np.float32)
    idx = [torch.empty(d, dtype=torch.int32, device=DEV) for _ in range(n)]
    val = [torch.empty(d, dtype=torch.float32, device=DEV) for _ in range(n)]
    counts = torch.empty(n, dtype=torch.int32, device=DEV)
    for t in range(w.T):
        ri_all, rv_all = [], []
        for i in range(n):
            g = workloads.gradient(w, i, t)
            efs.ef_hard_threshold(g.to(DEV), e_gpu[i], 1.0, lam, idx[i], val[i], counts[i:i + 1])
            ri, rv, e_ref[i] = oracle.ef_hard_threshold(g.numpy(), e_ref[i], 1.0, lam)
            ri_all.append(ri)
            rv_all.append(rv)
        efs.sparse_aggregate_apply(idx, val, counts, d, 1.0 / n, x_gpu, m_gpu, 0.9, w.gamma)
        x_ref, m_ref = oracle.sparse_aggregate_apply(ri_all, rv_all, d, 1.0 / n, x_ref, m_ref,
                                                     0.9, w.gamma)
        gu.assert_bits(x_gpu.cpu().numpy(), x_ref, "x t=%d" % t)
        gu.assert_bits(m_gpu.cpu().numpy(), m_ref, "m t=%d" % t)
    assert efs.ef_check_status() == efs.EF_OK


def test_full_size_resnet18_update():
    w = workloads.BY_NAME["resnet18"]
    d, n = w.d, w.n
    lam = workloads.density_lambda(w, workloads.gradient(w, 0, 0, device=DEV), w.density)
    idx = [torch.empty(d, dtype=torch.int32, device=DEV) for _ in range(n)]
    val = [torch.empty(d, dtype=torch.float32, device=DEV) for _ in range(n)]
    counts = torch.empty(n, dtype=torch.int32, device=DEV)
    for i in range(n):
        e = torch.zeros(d, device=DEV)
        efs.ef_hard_threshold(workloads.gradient(w, i, 0, device=DEV), e, w.gamma, lam, idx[i],
                              val[i], counts[i:i + 1])
    c = counts.cpu().numpy()
    ri = [idx[i][:c[i]].cpu().numpy().view(np.uint32) for i in range(n)]
    rv = [val[i][:c[i]].cpu().numpy() for i in range(n)]
    rng = _rng("r18")
    x = rng.standard_normal(d).astype(np.float32)
    m = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    xd, md = gu.to_dev(x), gu.to_dev(m)
    efs.sparse_aggregate_apply(idx, val, counts, d, 1.0 / n, xd, md, 0.9, 0.1)
    rx, rm = oracle.sparse_aggregate_apply(ri, rv, d, 1.0 / n, x, m, 0.9, 0.1)
    gu.assert_bits(xd.cpu().numpy(), rx, "x")
    gu.assert_bits(md.cpu().numpy(), rm, "m")
    assert efs.ef_check_status() == efs.EF_OK
