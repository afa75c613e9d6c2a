"""GPU parity: the CUDA path against the CPU oracle, bit for bit.

Masks, indices, counts, sent values and residuals must match exactly (same
single fma, same tie rule); the aggregate must match exactly (same worker
order). Small cases span several 4096-coordinate tiles with ragged tails;
full-size cases use the benchmark's workloads and launch configuration.
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

RAGGED = [1, 3, 4, 5, 127, 4095, 4096, 4097, 3 * 4096 + 17, 100_003]


def _rng(*key):
    return np.random.default_rng(zlib.crc32(repr(key).encode()))


def _inputs(d, seed, gscale=1e-2, escale=1e-3, bf16=False):
    rng = _rng("in", d, seed)
    g = (rng.standard_normal(d) * gscale).astype(np.float32)
    e = (rng.standard_normal(d) * escale).astype(np.float32)
    if bf16:
        g = torch.from_numpy(g).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    return g, e


def _check_same(gpu, ref, what):
    gi, gv, ge = gpu
    ri, rv, re_ = ref
    gu.assert_bits(gi, ri, what + " idx")
    gu.assert_bits(gv, rv, what + " val")
    gu.assert_bits(ge, re_, what + " e'")


# ------------------------------------------------------------ hard-threshold
@pytest.mark.usefixtures("ht_stream_kernel")
@pytest.mark.parametrize("bf16", [False, True])
@pytest.mark.parametrize("d", RAGGED)
def test_ht_random(d, bf16):
    g, e = _inputs(d, 1, bf16=bf16)
    for lam in (0.0, 1e-3, 2e-3, 1.0):
        _check_same(gu.ht(g, e, 0.1, lam), oracle.ef_hard_threshold(g, e, 0.1, lam),
                    "d=%d lam=%g" % (d, lam))


@pytest.mark.parametrize("offs", [(1, 0), (0, 1), (1, 1), (3, 2), (2, 0)])
@pytest.mark.parametrize("bf16", [False, True])
def test_ht_misaligned_bases(offs, bf16):
    d = 2 * 4096 + 333
    g, e = _inputs(d, 2, bf16=bf16)
    _check_same(gu.ht(g, e, 0.1, 1.5e-3, g_off=offs[0], e_off=offs[1]),
                oracle.ef_hard_threshold(g, e, 0.1, 1.5e-3), "offsets %s" % (offs,))


@pytest.mark.usefixtures("ht_stream_kernel")
def test_ht_adversarial_values():
    d = 3 * 4096 + 5
    rng = _rng("adv")
    lam = np.float32(0.25)
    pool = np.array([lam, -lam, np.nextafter(lam, np.float32(0)), 0.0, -0.0, np.nan, np.inf,
                     -np.inf, np.finfo(np.float32).smallest_subnormal,
                     -np.finfo(np.float32).tiny, 1e30, -3.0], dtype=np.float32)
    e = pool[rng.integers(0, len(pool), d)]
    g = np.zeros(d, np.float32)
    g[rng.integers(0, d, 500)] = -0.0
    for gamma, lam_ in ((1.0, float(lam)), (0.5, 0.0), (1.0, float("inf"))):
        _check_same(gu.ht(g, e, gamma, lam_), oracle.ef_hard_threshold(g, e, gamma, lam_),
                    "adversarial lam=%g" % lam_)


@pytest.mark.usefixtures("ht_stream_kernel")
def test_ht_fma_sensitive_values():
    # e = -round(gamma*g): a is the product's rounding error, which only a
    # single-rounding fma preserves
    d = 50_000
    rng = _rng("fma")
    g = (rng.standard_normal(d) * np.exp2(rng.integers(-10, 10, d))).astype(np.float32)
    gamma = np.float32(0.1)
    e = -(gamma * g)
    _check_same(gu.ht(g, e, float(gamma), 0.0), oracle.ef_hard_threshold(g, e, float(gamma), 0.0),
                "fma")


@pytest.mark.usefixtures("ht_stream_kernel")
def test_ht_all_and_nothing_sent():
    d = 5 * 4096 + 1
    g, e = _inputs(d, 3)
    i, v, en = gu.ht(g, e, 0.1, 0.0)            # every non-zero a is sent
    assert i.size == d
    _check_same((i, v, en), oracle.ef_hard_threshold(g, e, 0.1, 0.0), "all")
    i, v, en = gu.ht(g, e, 0.1, 1e9)            # nothing is sent
    assert i.size == 0
    _check_same((i, v, en), oracle.ef_hard_threshold(g, e, 0.1, 1e9), "none")


def test_ht_zero_length():
    cnt = torch.full((1,), 7, dtype=torch.int32, device=gu.DEV)
    z = torch.empty(0, device=gu.DEV)
    zi = torch.empty(0, dtype=torch.int32, device=gu.DEV)
    efs.ef_hard_threshold(z, z.clone(), 0.1, 1e-3, zi, z.clone(), cnt)
    assert int(cnt.item()) == 0


@pytest.mark.usefixtures("ht_stream_kernel")
@pytest.mark.parametrize("off", [0, 1])
def test_ht_concurrent_streams(off):
    # calls on different streams use different workspaces and may overlap
    # (off = 1: misaligned bases, the look-back kernel and its tile dispenser)
    d = 300_000
    g1, e1 = _inputs(d, 4)
    g2, e2 = _inputs(d, 5)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    outs = []
    for (g, e), s in (((g1, e1), s1), ((g2, e2), s2)):
        gd, ed = gu.to_dev(g, off), gu.to_dev(e, off)
        idx = torch.empty(d, dtype=torch.int32, device=gu.DEV)
        val = torch.empty(d, dtype=torch.float32, device=gu.DEV)
        cnt = torch.empty(1, dtype=torch.int32, device=gu.DEV)
        torch.cuda.synchronize()
        for _ in range(3):
            with torch.cuda.stream(s):  # the reset of e is ordered before the call
                ed.copy_(torch.from_numpy(e))
                efs.ef_hard_threshold(gd, ed, 0.1, 1e-3, idx, val, cnt)
        outs.append((idx, val, cnt, ed))
    torch.cuda.synchronize()
    for (idx, val, cnt, ed), (g, e) in zip(outs, ((g1, e1), (g2, e2))):
        c = int(cnt.item())
        _check_same((idx[:c].cpu().numpy().view(np.uint32), val[:c].cpu().numpy(),
                     ed.cpu().numpy()), oracle.ef_hard_threshold(g, e, 0.1, 1e-3), "stream")


@pytest.mark.usefixtures("stream_kernel")
@pytest.mark.parametrize("kind", ["topk", "topk_layerwise"])
def test_topk_concurrent_streams(kind):
    # Top-k calls on different streams (their own workspaces) may overlap on
    # the device; their grid-wide barriers need every CTA resident, which the
    # cooperative launches guarantee whatever the other stream runs
    d, k = 2 * 2**20 + 333, 4000
    seg_end = [d // 3, d // 2, d]
    seg_k = [1500, 1000, 1500]
    ins = [_inputs(d, 40), _inputs(d, 41), _inputs(d, 42)]
    streams = [torch.cuda.Stream() for _ in ins]
    outs = []
    for (g, e), s in zip(ins, streams):
        gd, ed = gu.to_dev(g), gu.to_dev(e)
        idx = torch.empty(k, dtype=torch.int32, device=gu.DEV)
        val = torch.empty(k, dtype=torch.float32, device=gu.DEV)
        cnt = torch.empty(1, dtype=torch.int32, device=gu.DEV)
        outs.append((gd, ed, idx, val, cnt))
    torch.cuda.synchronize()
    for rep in range(3):
        for (g, e), s, (gd, ed, idx, val, cnt) in zip(ins, streams, outs):
            with torch.cuda.stream(s):
                ed.copy_(torch.from_numpy(e).to(gu.DEV, non_blocking=True))
                if kind == "topk":
                    efs.ef_topk(gd, ed, 0.1, k, idx, val, cnt)
                else:
                    efs.ef_topk_layerwise(gd, ed, 0.1, seg_end, seg_k, idx, val, cnt)
    torch.cuda.synchronize()
    for (g, e), (gd, ed, idx, val, cnt) in zip(ins, outs):
        want = (oracle.ef_topk(g, e, 0.1, k) if kind == "topk"
                else oracle.ef_topk_layerwise(g, e, 0.1, seg_end, seg_k))
        _check_same((idx.cpu().numpy().view(np.uint32), val.cpu().numpy(), ed.cpu().numpy()),
                    want, kind + " concurrent")
    assert efs.ef_check_status() == efs.EF_OK


def test_ht_lookback_dispenser_back_to_back():
    # the look-back kernel (misaligned bases) takes its tile ids from a
    # per-stream dispenser that the last CTA to finish leaves at zero: launches
    # of different tile counts in a row on one stream, each equal to the oracle
    for r, d in enumerate([5 * 4096 + 3, 1, 4096, 700_001, 3 * 4096 + 17, 2 * 4096]):
        g, e = _inputs(d, 30 + r)
        _check_same(gu.ht(g, e, 0.1, 1.5e-3, g_off=1, e_off=1),
                    oracle.ef_hard_threshold(g, e, 0.1, 1.5e-3), "back to back d=%d" % d)
    assert efs.ef_check_status() == efs.EF_OK


def test_ht_balanced_chunks_over_calls():
    # each streaming call computes the next call's chunk boundaries from the
    # previous call's chunk totals; a dense quarter moves them. Calls of one
    # size in a row (the boundaries in use), a call of another size and a bf16
    # call between them (the boundaries dropped and rebuilt): every call equal
    # to the oracle
    d1, d2 = 5 * 2**20 + 77, 3 * 2**20 + 4099
    rng = np.random.default_rng(17)
    e_gpu = {d1: gu.to_dev(np.zeros(d1, np.float32)), d2: gu.to_dev(np.zeros(d2, np.float32))}
    e_ref = {d1: np.zeros(d1, np.float32), d2: np.zeros(d2, np.float32)}
    for r, (d, bf16) in enumerate([(d1, False)] * 4 + [(d2, False), (d1, False), (d1, True),
                                                         (d1, False), (d1, False)]):
        g = (rng.standard_normal(d) * 1e-2).astype(np.float32)
        g[: d // 4] *= 30.0 if r % 2 else 1.0          # the dense region comes and goes
        g[d // 2: d // 2 + d // 8] *= 10.0
        if bf16:
            g = (g.view(np.uint32) >> 16).astype(np.uint16)
        gd = gu.g_device(g)
        idx = torch.full((d,), -1, dtype=torch.int32, device=gu.DEV)
        val = torch.empty(d, dtype=torch.float32, device=gu.DEV)
        cnt = torch.zeros(1, dtype=torch.int32, device=gu.DEV)
        efs.ef_hard_threshold(gd, e_gpu[d], 0.1, 2e-3, idx, val, cnt)
        ri, rv, e_ref[d] = oracle.ef_hard_threshold(g, e_ref[d], 0.1, 2e-3)
        c = int(cnt.item())
        assert c == ri.size, (r, c, ri.size)
        gu.assert_bits(idx[:c].cpu().numpy().view(np.uint32), ri, "idx call %d" % r)
        gu.assert_bits(val[:c].cpu().numpy(), rv, "val call %d" % r)
        gu.assert_bits(e_gpu[d].cpu().numpy(), e_ref[d], "e' call %d" % r)
    assert efs.ef_check_status() == efs.EF_OK


def test_ht_ring_depth_follows_the_density_over_calls():
    # from 4096 tiles on, the claimed-group kernel picks its ring depth from
    # the density its earlier calls on this stream left in a hint word: sparse
    # and dense calls in a row on one EF residual (the dense ones switch the
    # next calls to the shallower ring, the sparse ones back), each equal to
    # the oracle, the residual carried from call to call on both sides
    d = 4096 * 4096 + 1237
    rng = np.random.default_rng(29)
    e_gpu, e_ref = gu.to_dev(np.zeros(d, np.float32)), np.zeros(d, np.float32)
    idx = torch.empty(d, dtype=torch.int32, device=gu.DEV)
    val = torch.empty(d, dtype=torch.float32, device=gu.DEV)
    cnt = torch.zeros(1, dtype=torch.int32, device=gu.DEV)
    for r, lam in enumerate([3e-3, 5e-4, 5e-4, 3e-3, 3e-3, 3e-2, 5e-4]):
        g = (rng.standard_normal(d) * 1e-2).astype(np.float32)
        efs.ef_hard_threshold(gu.g_device(g), e_gpu, 0.1, lam, idx, val, cnt)
        ri, rv, e_ref = oracle.ef_hard_threshold(g, e_ref, 0.1, lam)
        c = int(cnt.item())
        assert c == ri.size, (r, c, ri.size)
        gu.assert_bits(idx[:c].cpu().numpy().view(np.uint32), ri, "idx call %d" % r)
        gu.assert_bits(val[:c].cpu().numpy(), rv, "val call %d" % r)
        gu.assert_bits(e_gpu.cpu().numpy(), e_ref, "e' call %d" % r)
    assert efs.ef_check_status() == efs.EF_OK


# ---------------------------------------------------------------------- Top-k
# ------------------------------------------- on-chip staging and its spill
# The streaming compaction keeps each compute warp's first pairs of its CTA's
# chunk in shared memory (768 per warp for the hard-threshold op, 512 for the
# Top-k candidate op) and spills the rest to global slots. At this size every
# CTA owns several tiles, so dense chunks spill and sparse ones do not.
SPILL_D = 3 * 2**20 + 4099


@pytest.mark.usefixtures("ht_stream_kernel")
@pytest.mark.parametrize("bf16", [False, True])
def test_ht_spill_everything_sent(bf16):
    g, e = _inputs(SPILL_D, 21, bf16=bf16)
    _check_same(gu.ht(g, e, 0.1, 0.0), oracle.ef_hard_threshold(g, e, 0.1, 0.0), "all sent")


@pytest.mark.usefixtures("ht_stream_kernel")
def test_ht_spill_mixed_density():
    g, e = _inputs(SPILL_D, 22)
    g[: SPILL_D // 4] *= 1000.0  # a dense quarter (~96 % sent), the rest sends nothing
    i, v, en = gu.ht(g, e, 0.1, 0.05)
    assert i.size > 0.9 * (SPILL_D // 4) and i.max() < SPILL_D // 4
    _check_same((i, v, en), oracle.ef_hard_threshold(g, e, 0.1, 0.05), "mixed")


@pytest.mark.usefixtures("ht_stream_kernel")
@pytest.mark.parametrize("out_off", [(1, 0), (2, 3), (3, 1)])
def test_ht_misaligned_outputs(out_off):
    # the pairs are written with 16-byte stores matched to each output's own
    # alignment; dense (several buffer pieces per CTA) and sparse chunks
    g, e = _inputs(SPILL_D, 24)
    g[: SPILL_D // 3] *= 1000.0
    _check_same(gu.ht(g, e, 0.1, 0.05, out_off=out_off), oracle.ef_hard_threshold(g, e, 0.1, 0.05),
                "outputs offset %s" % (out_off,))
    d = 4096 + 77
    g, e = _inputs(d, 25)
    _check_same(gu.ht(g, e, 0.1, 1e-3, out_off=out_off), oracle.ef_hard_threshold(g, e, 0.1, 1e-3),
                "small, outputs offset %s" % (out_off,))


@pytest.mark.usefixtures("stream_kernel")
@pytest.mark.parametrize("region,k", [(SPILL_D // 50, 20_000), (SPILL_D // 5, SPILL_D // 16)])
def test_topk_spill_concentrated_candidates(region, k):
    # all candidates in the first `region` coordinates: the few CTAs there
    # stage more than their warps' on-chip share (short and long lists)
    g, e = _inputs(SPILL_D, 23)
    g[:region] *= 1000.0
    _check_same(gu.topk(g, e, 0.1, k), oracle.ef_topk(g, e, 0.1, k),
                "region=%d k=%d" % (region, k))


@pytest.mark.usefixtures("stream_kernel")
@pytest.mark.parametrize("d", RAGGED)
def test_topk_random(d):
    g, e = _inputs(d, 11)
    for k in sorted({0, 1, max(1, d // 100), d // 2, d}):
        _check_same(gu.topk(g, e, 0.1, k), oracle.ef_topk(g, e, 0.1, k), "d=%d k=%d" % (d, k))


def test_topk_bf16_and_misaligned():
    d = 3 * 4096 + 77
    g, e = _inputs(d, 12, bf16=True)
    for offs in ((0, 0), (1, 1), (3, 0), (0, 2)):
        _check_same(gu.topk(g, e, 0.1, 500, g_off=offs[0], e_off=offs[1]),
                    oracle.ef_topk(g, e, 0.1, 500), "offs %s" % (offs,))


@pytest.mark.usefixtures("stream_kernel")
def test_topk_heavy_ties():
    d = 200_003
    rng = _rng("ties")
    pool = np.array([0.0, -0.0, 0.5, -0.5, 0.25, 1.0, -1.0, 2.0], np.float32)
    e = pool[rng.integers(0, len(pool), d)]
    g = np.zeros(d, np.float32)
    for k in (1, 7, 1000, 25_000, 100_000, 199_999):
        _check_same(gu.topk(g, e, 1.0, k), oracle.ef_topk(g, e, 1.0, k), "ties k=%d" % k)


@pytest.mark.usefixtures("stream_kernel")
def test_topk_mostly_zero_like_lstm_embedding():
    # ~62% exact zeros; k beyond the non-zeros forces the choice into the zero bucket
    d = 400_000
    rng = _rng("zeros")
    g = (rng.standard_t(3, d) * 1e-3).astype(np.float32)
    g[rng.random(d) < 0.62] = 0.0
    e = np.zeros(d, np.float32)
    nz = int(np.count_nonzero(g))
    for k in (d // 100, nz - 1, nz, nz + 1, nz + 5000):
        _check_same(gu.topk(g, e, 0.1, k), oracle.ef_topk(g, e, 0.1, k), "zeros k=%d" % k)


@pytest.mark.usefixtures("stream_kernel")
def test_topk_all_equal_magnitude_large():
    # all keys tie in the magnitude bits: the index digits decide, through
    # full-array refine passes (the bucket exceeds the candidate buffer)
    d = 3_000_017
    e = np.full(d, 0.75, np.float32)
    e[1::3] = -0.75
    g = np.zeros(d, np.float32)
    for k in (1, 1_000_000, 2_500_000):
        gi, gv, ge = gu.topk(g, e, 1.0, k)
        assert gi.size == k and np.array_equal(gi, np.arange(k, dtype=np.uint32))
        gu.assert_bits(gv, e[:k], "vals")
        want = e.copy()
        want[:k] = 0.0
        gu.assert_bits(ge, want, "e'")


@pytest.mark.usefixtures("stream_kernel")
def test_topk_nan_inf():
    d = 9000
    g, e = _inputs(d, 13)
    e[[5, 4097, 8000]] = [np.nan, np.inf, -np.inf]
    for k in (1, 2, 3, 10):
        _check_same(gu.topk(g, e, 0.1, k), oracle.ef_topk(g, e, 0.1, k), "nan k=%d" % k)


@pytest.mark.usefixtures("stream_kernel")
def test_topk_calls_in_a_row_with_jumping_scales():
    # calls of one (k, d) on one stream whose scales jump by 100x between
    # calls, and a call with another k between them (the per-call state and
    # the sampled bound start afresh each time): every call equal to the oracle
    d, k = 3 * 2**20 + 517, 3000
    rng = np.random.default_rng(23)
    e_gpu = gu.to_dev(np.zeros(d, np.float32))
    e_ref = np.zeros(d, np.float32)
    for r, (scale, kk) in enumerate([(1.0, k), (1.0, k), (100.0, k), (1.0, k), (0.01, k),
                                     (0.01, k), (1.0, k + 1), (1.0, k), (1.0, k)]):
        g = (rng.standard_normal(d) * 1e-2 * scale).astype(np.float32)
        gd = gu.to_dev(g)
        idx = torch.full((kk,), -1, dtype=torch.int32, device=gu.DEV)
        val = torch.empty(kk, dtype=torch.float32, device=gu.DEV)
        cnt = torch.zeros(1, dtype=torch.int32, device=gu.DEV)
        efs.ef_topk(gd, e_gpu, 0.1, kk, idx, val, cnt)
        ri, rv, e_ref = oracle.ef_topk(g, e_ref, 0.1, kk)
        assert int(cnt.item()) == kk
        gu.assert_bits(idx.cpu().numpy().view(np.uint32), ri, "idx call %d" % r)
        gu.assert_bits(val.cpu().numpy(), rv, "val call %d" % r)
        gu.assert_bits(e_gpu.cpu().numpy(), e_ref, "e' call %d" % r)
    assert efs.ef_check_status() == efs.EF_OK


# ---------------------------------------------------------------- aggregation
def _sparse_lists(n, d, density, seed, integer=False):
    rng = _rng("agg", n, d, seed)
    idx, val = [], []
    for _ in range(n):
        m = rng.random(d) < density
        i = np.nonzero(m)[0].astype(np.uint32)
        v = (rng.integers(-9, 9, i.size) if integer else rng.standard_normal(i.size)).astype(np.float32)
        idx.append(i)
        val.append(v)
    return idx, val


@pytest.mark.parametrize("n", [1, 2, 4, 8, 16])
@pytest.mark.parametrize("d", [5, 4096, 4097, 100_003])
def test_aggregate_random(n, d):
    for density in (0.001, 0.05, 1.0):
        idx, val = _sparse_lists(n, d, density, 1)
        gu.assert_bits(gu.aggregate(idx, val, d), oracle.sparse_aggregate(idx, val, d),
                       "n=%d d=%d rho=%g" % (n, d, density))


def test_aggregate_order_and_signed_zero():
    big = np.float32(2.0 ** 24)
    idx = [np.array([3, 4100], np.uint32)] * 3
    val = [np.array([big, -0.0], np.float32), np.array([1.0, -0.0], np.float32),
           np.array([-big, -0.0], np.float32)]
    out = gu.aggregate(idx, val, 5000)
    gu.assert_bits(out, oracle.sparse_aggregate(idx, val, 5000), "order")
    assert out[3] == 0.0 and gu.bits(out[4100:4101])[0] == 0   # +0.0


def test_aggregate_empty_lists_and_misaligned_output():
    d = 20_001
    idx, val = _sparse_lists(6, d, 0.01, 2)
    idx[2], val[2] = idx[2][:0], val[2][:0]
    idx[5], val[5] = idx[5][:0], val[5][:0]
    for off in (0, 1, 3):
        gu.assert_bits(gu.aggregate(idx, val, d, dense_off=off),
                       oracle.sparse_aggregate(idx, val, d), "off=%d" % off)


def test_aggregate_tile_boundary_layouts():
    # lists with long runs of empty tiles, lists inside one tile, a list that
    # ends in the first tile, one that starts in the last, the last coordinate,
    # entries on tile boundaries: every per-tile offset pattern of the lists
    d = 300 * 4096 + 123
    rng = np.random.default_rng(31)
    lists = [
        np.array([0, 4095, 4096, 8191, 8192], np.uint32),
        np.array([d - 1], np.uint32),
        np.array([7], np.uint32),
        np.sort(rng.choice(np.arange(150 * 4096, 151 * 4096), 900, replace=False)).astype(np.uint32),
        np.array([5, 250 * 4096, d - 2], np.uint32),
        np.arange(299 * 4096, d, 3, dtype=np.uint32),
        np.zeros(0, np.uint32),
        np.sort(rng.choice(d, 20_000, replace=False)).astype(np.uint32),
    ]
    vals = [rng.standard_normal(len(x)).astype(np.float32) for x in lists]
    gu.assert_bits(gu.aggregate(lists, vals, d), oracle.sparse_aggregate(lists, vals, d),
                   "tile layouts")
    assert efs.ef_check_status() == efs.EF_OK


@pytest.mark.parametrize("n", [33, 100])
def test_aggregate_many_workers(n):
    # more workers than one stage takes (32 runs): the runs of a tile are
    # staged in several groups, in worker order
    d = 3 * 4096 + 7
    for density in (0.01, 0.4):
        idx, val = _sparse_lists(n, d, density, 5)
        gu.assert_bits(gu.aggregate(idx, val, d), oracle.sparse_aggregate(idx, val, d),
                       "n=%d rho=%g" % (n, density))


@pytest.mark.parametrize("offs", [(1, 0), (0, 3), (2, 2)])
def test_aggregate_misaligned_lists(offs):
    # lists that are not 16-byte aligned take the 4-byte staging path; one
    # such list is enough
    d = 5 * 4096 + 11
    idx, val = _sparse_lists(6, d, 0.2, 6)
    idx_t = [gu.to_dev(i.view(np.int32), offs[0] if w == 3 else 0) for w, i in enumerate(idx)]
    val_t = [gu.to_dev(v, offs[1] if w == 3 else 0) for w, v in enumerate(val)]
    counts = torch.tensor([len(i) for i in idx], dtype=torch.int32, device=gu.DEV)
    dense = torch.full((d,), float("nan"), device=gu.DEV)
    efs.sparse_aggregate(idx_t, val_t, counts, d, dense)
    torch.cuda.synchronize()
    gu.assert_bits(dense.cpu().numpy(), oracle.sparse_aggregate(idx, val, d), "offs %s" % (offs,))
    assert efs.ef_check_status() == efs.EF_OK


def test_aggregate_runs_across_stages():
    # runs longer than a stage (1024 staged elements), runs that start and
    # end at every residue modulo 4, and a tile whose pairs are all in one
    # warp's coordinates
    d = 8 * 4096
    rng = np.random.default_rng(41)
    lists = []
    for w in range(7):
        start = 4096 + w            # every start residue
        lists.append(np.arange(start, 3 * 4096 - w, 1 + (w % 3), dtype=np.uint32))
    lists.append(np.arange(5 * 4096 + 600, 5 * 4096 + 1000, dtype=np.uint32))
    lists.append(np.sort(rng.choice(d, 9000, replace=False)).astype(np.uint32))
    vals = [rng.standard_normal(len(x)).astype(np.float32) for x in lists]
    gu.assert_bits(gu.aggregate(lists, vals, d), oracle.sparse_aggregate(lists, vals, d),
                   "long runs")
    assert efs.ef_check_status() == efs.EF_OK


# ------------------------------------------------------- multi-iteration EF
@pytest.mark.parametrize("method", ["ht", "topk"])
def test_lr_workload_all_iterations(method):
    """Configuration 0 (d = 100,000, n = 4, T = 10): every worker, every
    iteration, and the aggregate of every iteration, each side on its own state."""
    w = workloads.BY_NAME["lr"]
    e_ref = [np.zeros(w.d, np.float32) for _ in range(w.n)]
    e_gpu = [gu.to_dev(np.zeros(w.d, np.float32)) for _ in range(w.n)]
    k, lam = w.topk_k[0], w.lambdas[0]
    for t in range(w.T):
        gi_all, gv_all, ri_all, rv_all = [], [], [], []
        for i in range(w.n):
            g = workloads.gradient(w, i, t)
            idx = torch.empty(w.d, dtype=torch.int32, device=gu.DEV)
            val = torch.empty(w.d, dtype=torch.float32, device=gu.DEV)
            cnt = torch.empty(1, dtype=torch.int32, device=gu.DEV)
            if method == "ht":
                efs.ef_hard_threshold(g.to(gu.DEV), e_gpu[i], w.gamma, lam, idx, val, cnt)
                ri, rv, e_ref[i] = oracle.ef_hard_threshold(g.numpy(), e_ref[i], w.gamma, lam)
            else:
                efs.ef_topk(g.to(gu.DEV), e_gpu[i], w.gamma, k, idx, val, cnt)
                ri, rv, e_ref[i] = oracle.ef_topk(g.numpy(), e_ref[i], w.gamma, k)
            c = int(cnt.item())
            gu.assert_bits(idx[:c].cpu().numpy().view(np.uint32), ri, "t=%d i=%d idx" % (t, i))
            gu.assert_bits(val[:c].cpu().numpy(), rv, "val")
            gu.assert_bits(e_gpu[i].cpu().numpy(), e_ref[i], "e'")
            gi_all.append(idx[:c])
            gv_all.append(val[:c])
            ri_all.append(ri)
            rv_all.append(rv)
        counts = torch.tensor([len(r) for r in ri_all], dtype=torch.int32, device=gu.DEV)
        dense = torch.empty(w.d, dtype=torch.float32, device=gu.DEV)
        efs.sparse_aggregate(gi_all, gv_all, counts, w.d, dense)
        gu.assert_bits(dense.cpu().numpy(), oracle.sparse_aggregate(ri_all, rv_all, w.d),
                       "aggregate t=%d" % t)
    assert efs.ef_check_status() == efs.EF_OK
