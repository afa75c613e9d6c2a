"""Distributed EF-SGD on l2-regularised logistic regression (the paper's convex
experiments, eq. 7) through the library, on a seeded synthetic problem.

The loop's states agree with the oracle's bit for bit at every step when both
sides see the same gradients (compression, residuals, the model after the
fused update), and its error norms with the oracle's fp64 norms; the
hard-threshold error obeys the absolute-compressor bound ||e||^2 <= d lambda^2
at every step; the matched-volume tuning meets its target.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2108_00951_gb300 as efs
from paper_2108_00951_gb300 import ef_sgd

pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import gpu_util as gu  # noqa: E402

DEV = gu.DEV


@pytest.fixture(scope="module")
def tiny():
    return ef_sgd.make_problem("tiny", device=DEV)


@pytest.mark.parametrize("compressor,param", [("ht", 2e-3), ("topk", 3)])
def test_loop_matches_oracle_step_by_step(tiny, compressor, param):
    n, d, T = 4, tiny.d, 40
    gen = torch.Generator().manual_seed(5)
    x = torch.zeros(d, device=DEV)
    e = torch.zeros(n, d, device=DEV)
    idx = [torch.empty(d, dtype=torch.int32, device=DEV) for _ in range(n)]
    val = [torch.empty(d, dtype=torch.float32, device=DEV) for _ in range(n)]
    counts = torch.empty(n, dtype=torch.int32, device=DEV)
    err = torch.empty(n, dtype=torch.float64, device=DEV)
    x_ref = np.zeros(d, np.float32)
    e_ref = [np.zeros(d, np.float32) for _ in range(n)]
    for t in range(T):
        rows = torch.randint(0, tiny.N, (n,), generator=gen).to(DEV)
        g = ef_sgd.local_gradients(tiny, x, rows)
        g_host = g.cpu().numpy()
        ri_all, rv_all = [], []
        for w in range(n):
            if compressor == "ht":
                efs.ef_hard_threshold(g[w], e[w], tiny.gamma, param, idx[w], val[w],
                                      counts[w:w + 1], err_sq_out=err[w:w + 1])
                ri, rv, e_ref[w] = oracle.ef_hard_threshold(g_host[w], e_ref[w], tiny.gamma, param)
            else:
                efs.ef_topk(g[w], e[w], tiny.gamma, int(param), idx[w], val[w], counts[w:w + 1],
                            err_sq_out=err[w:w + 1])
                ri, rv, e_ref[w] = oracle.ef_topk(g_host[w], e_ref[w], tiny.gamma, int(param))
            ri_all.append(ri)
            rv_all.append(rv)
        efs.sparse_aggregate_apply(idx, val, counts, d, 1.0 / n, x)
        x_ref, _ = oracle.sparse_aggregate_apply(ri_all, rv_all, d, 1.0 / n, x_ref)
        c = counts.cpu().numpy()
        for w in range(n):
            gu.assert_bits(idx[w][:c[w]].cpu().numpy().view(np.uint32), ri_all[w], "idx t=%d" % t)
            gu.assert_bits(val[w][:c[w]].cpu().numpy(), rv_all[w], "val t=%d" % t)
            gu.assert_bits(e[w].cpu().numpy(), e_ref[w], "e t=%d w=%d" % (t, w))
            want = oracle.error_norm_sq(e_ref[w])
            assert abs(float(err[w]) - want) <= 1e-6 * want + 1e-300
        gu.assert_bits(x.cpu().numpy(), x_ref, "x t=%d" % t)
    assert efs.ef_check_status() == efs.EF_OK


def test_hard_threshold_error_bound_every_step(tiny):
    # absolute compressor: every residual coordinate is below lambda in
    # magnitude, so each worker's ||e||^2 <= d lambda^2 (Sec. 5); summed over n
    n, lam = 8, 5e-3
    hist = ef_sgd.run(tiny, n, 100, "ht", lam)
    assert max(hist["err_sq"]) <= n * tiny.d * lam * lam
    assert hist["subopt"][-1] < hist["subopt"][0]


def test_matched_volume(tiny):
    n, T = 8, 100
    topk = ef_sgd.run(tiny, n, T, "topk", 1, record_every=T)
    lam = ef_sgd.match_volume(tiny, n, T, topk["sent"][-1])
    ht = ef_sgd.run(tiny, n, T, "ht", lam, record_every=T)
    assert abs(ht["sent"][-1] - topk["sent"][-1]) <= 0.15 * topk["sent"][-1]
