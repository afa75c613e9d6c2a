"""The optional per-step error norm ||e_{t+1}||^2 (the total error's term)
against the oracle's fp64 sum of the oracle's own residual.

Tolerance, derived from the arithmetic (every partial sum of nonnegative fp32
squares sees at most 13 roundings, then fp64): relative 1e-6. Every route of
every step is reached: the hard-threshold stream and its look-back fallback
for misaligned inputs; entire-vector Top-k with a short candidate list, a list
beyond shared memory, the full-array mode, k = 0 and k = d, misaligned
inputs; layer-wise Top-k over every kind of segment, teams, selection from e,
a cut-off list and misaligned inputs. Requesting the norm leaves every other
output bit-identical, and the norm itself is reproducible bit for bit.
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
REL = 1e-6


def _rng(*key):
    return np.random.default_rng(zlib.crc32(repr(key).encode()))


def _inputs(d, seed):
    rng = _rng("err", d, seed)
    return ((rng.standard_normal(d) * 1e-2).astype(np.float32),
            (rng.standard_normal(d) * 1e-3).astype(np.float32))


def _run(kind, g, e, gamma, arg, off=0):
    """One step through the binding with err_sq_out; returns (idx, val, e', err)."""
    d = e.size
    gd, ed = gu.g_device(g, off), gu.to_dev(e, off)
    if kind == "ht":
        cap = max(d, 1)
    elif kind == "topk":
        cap = max(int(arg), 1)
    else:
        cap = max(int(np.sum(np.asarray(arg[1], np.uint64))), 1)
    idx = torch.full((cap,), -1, dtype=torch.int32, device=DEV)
    val = torch.empty(cap, dtype=torch.float32, device=DEV)
    cnt = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    err = torch.full((1,), float("nan"), dtype=torch.float64, device=DEV)
    if kind == "ht":
        efs.ef_hard_threshold(gd, ed, gamma, arg, idx, val, cnt, err_sq_out=err)
    elif kind == "topk":
        efs.ef_topk(gd, ed, gamma, int(arg), idx, val, cnt, err_sq_out=err)
    else:
        efs.ef_topk_layerwise(gd, ed, gamma, arg[0], arg[1], idx, val, cnt, err_sq_out=err)
    torch.cuda.synchronize()
    c = int(cnt.item())
    return (idx[:c].cpu().numpy().view(np.uint32), val[:c].cpu().numpy(), ed.cpu().numpy(),
            float(err.item()))


def _ref(kind, g, e, gamma, arg):
    if kind == "ht":
        return oracle.ef_hard_threshold(g, e, gamma, arg)
    if kind == "topk":
        return oracle.ef_topk(g, e, gamma, int(arg))
    return oracle.ef_topk_layerwise(g, e, gamma, arg[0], arg[1])


def _check(kind, g, e, gamma, arg, what, off=0):
    ri, rv, re_ = _ref(kind, g, e, gamma, arg)
    gi, gv, ge, gerr = _run(kind, g, e, gamma, arg, off)
    gu.assert_bits(gi, ri, what + " idx")
    gu.assert_bits(gv, rv, what + " val")
    gu.assert_bits(ge, re_, what + " e'")
    want = oracle.error_norm_sq(re_)
    assert abs(gerr - want) <= REL * want + 1e-300, (what, gerr, want)
    again = _run(kind, g, e, gamma, arg, off)[3]
    assert np.float64(again).view(np.uint64) == np.float64(gerr).view(np.uint64), what
    assert efs.ef_check_status() == efs.EF_OK, what
    return gerr, want


@pytest.mark.usefixtures("ht_stream_kernel")
@pytest.mark.parametrize("d", [1, 4097, 3 * 4096 + 17, 300_001])
@pytest.mark.parametrize("off", [0, 1])
def test_ht_error_norm(d, off):
    g, e = _inputs(d, 1)
    for lam in (0.0, 1.5e-3, 1.0):
        _check("ht", g, e, 0.1, lam, "ht d=%d off=%d lam=%g" % (d, off, lam), off=off)


@pytest.mark.usefixtures("ht_stream_kernel")
def test_ht_error_norm_bf16():
    d = 100_003
    g, e = _inputs(d, 2)
    gb = torch.from_numpy(g).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    _check("ht", gb, e, 0.1, 1e-3, "ht bf16")


@pytest.mark.parametrize("d,k", [(100_003, 1000),      # short candidate list
                                 (1_000_000, 60_000),  # list beyond shared memory
                                 (300_000, 150_000),   # full-array mode
                                 (50_000, 0), (50_000, 50_000), (7, 3)])
@pytest.mark.usefixtures("stream_kernel")
def test_topk_error_norm(d, k):
    g, e = _inputs(d, 3)
    _check("topk", g, e, 0.1, k, "topk d=%d k=%d" % (d, k))


def test_topk_error_norm_misaligned():
    g, e = _inputs(200_001, 4)
    _check("topk", g, e, 0.1, 2000, "topk misaligned", off=1)


KINDS_SIZES = [0, 5, 64, 4097, 49152, 49153, 100_003, 3 * 4096 + 17, 1, 200_000, 7, 65_536]
KINDS_K = [0, 5, 3, 40, 491, 1, 1000, 0, 1, 2000, 6, 65_535]


@pytest.mark.usefixtures("stream_kernel")
@pytest.mark.parametrize("case", ["kinds", "team", "from_e", "cut_off", "misaligned"])
def test_layerwise_error_norm(case):
    if case in ("kinds", "misaligned"):
        sizes, ks = KINDS_SIZES, KINDS_K
    elif case == "team":
        sizes, ks = [400_000, 70_000], [60_000, 700]
    elif case == "from_e":
        sizes, ks = [1_500_000, 1_500_003], [750_000, 10]
    else:
        sizes, ks = [1_000_000] * 5 + [4099], [150_000] * 5 + [17]
    g, e = _inputs(sum(sizes), 5)
    ends = np.cumsum(np.asarray(sizes, dtype=np.uint64)).astype(np.uint64)
    _check("lw", g, e, 0.1, (ends, ks), "layer-wise " + case,
           off=1 if case == "misaligned" else 0)


def test_error_norm_full_size_resnet18():
    w = workloads.BY_NAME["resnet18"]
    g = workloads.gradient(w, 0, 0, device=DEV).cpu().numpy()
    e = (np.random.default_rng(7).standard_normal(w.d) * 1e-4).astype(np.float32)
    lam = workloads.density_lambda(w, torch.from_numpy(g), w.density)
    ends = np.asarray(workloads.segment_ends(w), dtype=np.uint64)
    ks = workloads.layerwise_k(w, 1e-3)
    _check("ht", g, e, w.gamma, lam, "resnet18 ht")
    _check("topk", g, e, w.gamma, w.topk_values()[0], "resnet18 topk")
    _check("lw", g, e, w.gamma, (ends, ks), "resnet18 layer-wise")


@pytest.mark.usefixtures("stream_kernel")
@pytest.mark.parametrize("kind", ["ht", "topk"])
def test_error_norm_reproducible_over_calls(kind):
    # calls that return the norm use equal chunks and the sampled Top-k bound
    # (the norm's summation order follows them), so identical inputs give the
    # same bits however many calls of the size ran before on the stream
    d = 4 * 2**20 + 3
    g, e = _inputs(d, 9)
    g[: d // 5] *= 20.0   # a dense region: balanced chunks would differ from equal ones
    arg = 1.5e-3 if kind == "ht" else 20_000
    bits = set()
    for _ in range(4):
        bits.add(np.float64(_run(kind, g, e, 0.1, arg)[3]).view(np.uint64).item())
        # calls without the norm in between (they may balance and use the bound)
        if kind == "ht":
            gu.ht(g, e, 0.1, arg)
        else:
            gu.topk(g, e, 0.1, arg)
    assert len(bits) == 1
    assert efs.ef_check_status() == efs.EF_OK
