"""GPU parity of error feedback with scaled integer rounding (an absolute
compressor, Sec. 5) and of the exact integer exchange of its messages,
against the oracle: messages, residuals, counts and dense sums bit for bit,
the error norm within 1e-6. Ragged sizes, several scales, bf16 gradients,
misaligned arrays (scalar path), values that do not fit an int32 message,
and a multi-iteration EF loop with the residual carried over.
"""
import zlib

import numpy as np
import pytest
import torch

import oracle
import paper_2108_00951_gb300 as efs

pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import gpu_util as gu  # noqa: E402

DEV = gu.DEV


def _rng(*key):
    return np.random.default_rng(zlib.crc32(repr(key).encode()))


def _round(g, e, gamma, m, off=0):
    d = e.size
    gd, ed = gu.g_device(g, off), gu.to_dev(e, off)
    qbuf = torch.empty(d + off, dtype=torch.int32, device=DEV)
    q = qbuf[off:]
    unsent = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    err = torch.empty(1, dtype=torch.float64, device=DEV)
    efs.ef_scaled_round(gd, ed, gamma, m, q, unsent, err_sq_out=err)
    torch.cuda.synchronize()
    return q.cpu().numpy(), ed.cpu().numpy(), int(unsent.item()), float(err.item())


def _check(g, e, gamma, m, what, off=0):
    gq, ge, gu_, gerr = _round(g, e, gamma, m, off)
    rq, re_, ru = oracle.ef_scaled_round(g, e, gamma, m)
    gu.assert_bits(gq.view(np.uint32), rq.view(np.uint32), what + " q")
    gu.assert_bits(ge, re_, what + " e'")
    assert gu_ == ru, (what, gu_, ru)
    want = oracle.error_norm_sq(re_)
    if np.isfinite(want):
        assert abs(gerr - want) <= 1e-6 * want + 1e-300, (what, gerr, want)
    assert efs.ef_check_status() == efs.EF_OK
    return rq, re_


@pytest.mark.parametrize("d", [1, 3, 4, 4097, 100_003])
@pytest.mark.parametrize("m", [-4, 0, 10, 23])
def test_scaled_round_random(d, m):
    rng = _rng("round", d, m)
    g = (rng.standard_normal(d) * 5.0).astype(np.float32)
    e = (rng.standard_normal(d) * 0.1).astype(np.float32)
    _check(g, e, 0.1, m, "d=%d m=%d" % (d, m))


@pytest.mark.parametrize("off", [1, 2])
def test_scaled_round_misaligned_and_bf16(off):
    d = 3 * 4096 + 5
    rng = _rng("mis", off)
    g = (rng.standard_normal(d)).astype(np.float32)
    e = (rng.standard_normal(d) * 0.01).astype(np.float32)
    _check(g, e, 0.5, 8, "misaligned off=%d" % off, off=off)
    gb = torch.from_numpy(g).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    _check(gb, e, 0.5, 8, "bf16 off=%d" % off, off=off)
    _check(gb, e, 0.5, 8, "bf16 aligned")


def test_scaled_round_values_that_do_not_fit():
    d = 4096 + 11
    rng = _rng("big")
    e = (rng.standard_normal(d) * 1e3).astype(np.float32)
    e[::97] = np.float32(2.0 ** 31)
    e[5] = np.inf
    e[6] = -np.inf
    e[7] = np.nan
    e[8] = np.float32(-(2.0 ** 31))
    e[9] = np.float32(2.0 ** 31 - 128)
    g = np.zeros(d, np.float32)
    _check(g, e, 1.0, 0, "no-fit m=0")
    _check(g, e, 1.0, 4, "no-fit m=4")


def test_scaled_round_ef_loop():
    """Ten EF iterations with the residual carried: states stay bit-equal."""
    d, m = 50_001, 12
    e_gpu = torch.zeros(d, device=DEV)
    e_ref = np.zeros(d, np.float32)
    q = torch.empty(d, dtype=torch.int32, device=DEV)
    unsent = torch.empty(1, dtype=torch.int32, device=DEV)
    for t in range(10):
        g = (_rng("loop", t).standard_normal(d) * 1e-3).astype(np.float32)
        efs.ef_scaled_round(gu.to_dev(g), e_gpu, 0.1, m, q, unsent)
        rq, e_ref, _ = oracle.ef_scaled_round(g, e_ref, 0.1, m)
        gu.assert_bits(q.cpu().numpy().view(np.uint32), rq.view(np.uint32), "q t=%d" % t)
        gu.assert_bits(e_gpu.cpu().numpy(), e_ref, "e t=%d" % t)
    assert efs.ef_check_status() == efs.EF_OK


@pytest.mark.parametrize("n", [1, 3, 8, 16])
@pytest.mark.parametrize("d", [5, 4096, 100_003])
@pytest.mark.parametrize("off", [0, 1])
def test_int_aggregate(n, d, off):
    rng = _rng("iagg", n, d)
    qs = [rng.integers(-(2 ** 31) + 1, 2 ** 31 - 1, d, dtype=np.int64).astype(np.int32)
          for _ in range(n)]
    qd = [gu.to_dev(q, off) for q in qs]
    buf = torch.full((d + off,), float("nan"), device=DEV)
    dense = buf[off:]
    for m in (-3, 0, 20):
        efs.int_aggregate(qd, d, m, dense)
        torch.cuda.synchronize()
        gu.assert_bits(dense.cpu().numpy(), oracle.int_aggregate(qs, d, m), "n=%d m=%d" % (n, m))
    assert efs.ef_check_status() == efs.EF_OK
