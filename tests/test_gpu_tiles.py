"""The tile index of a message (uint32[ceil(d / 4096) + 1]: the pairs below
each multiple of 4096, then the count): written by ef_hard_threshold_tiled
(streaming path, and the look-back path for misaligned inputs), consumed by
the tiled aggregation entries, which must give the same results as the
searching ones. The expected tile index is the definition evaluated on the
oracle's index list (np.searchsorted); the sums are the oracle's."""
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
SIZES = [1, 4095, 4096, 4097, 3 * 4096 + 17, 100_003, 3 * 2**20 + 4099]


def _rng(*key):
    return np.random.default_rng(zlib.crc32(repr(key).encode()))


def _inputs(d, seed, bf16=False):
    rng = _rng("tiles", d, seed)
    g = (rng.standard_normal(d) * 1e-2).astype(np.float32)
    e = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    if d > 50_000:  # a dense region and an empty one
        g[: d // 5] *= 30.0
        g[d // 2: d // 2 + d // 5] = 0.0
    if bf16:
        g = torch.from_numpy(g).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    return g, e


def _tile_index(idx, d):
    bounds = np.arange(efs.tiles_for(d) - 1, dtype=np.uint64) * efs.TILE
    t = np.searchsorted(idx.astype(np.uint64), bounds, side="left").astype(np.uint32)
    return np.concatenate([t, np.array([idx.size], np.uint32)])


def _ht_tiled(g, e, gamma, lam, g_off=0, e_off=0):
    d = e.size
    gd, ed = gu.g_device(g, g_off), gu.to_dev(e, e_off)
    idx = torch.full((max(d, 1),), -1, dtype=torch.int32, device=DEV)
    val = torch.empty(max(d, 1), dtype=torch.float32, device=DEV)
    cnt = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    tiles = torch.full((efs.tiles_for(d),), -7, dtype=torch.int32, device=DEV)
    efs.ef_hard_threshold(gd, ed, gamma, lam, idx, val, cnt, tiles_out=tiles)
    torch.cuda.synchronize()
    c = int(cnt.item())
    return (idx[:c].cpu().numpy().view(np.uint32), val[:c].cpu().numpy(), ed.cpu().numpy(),
            tiles.cpu().numpy().view(np.uint32))


@pytest.mark.usefixtures("ht_stream_kernel")
@pytest.mark.parametrize("bf16", [False, True])
@pytest.mark.parametrize("d", SIZES)
def test_hard_threshold_writes_the_tile_index(d, bf16):
    g, e = _inputs(d, 1, bf16)
    for lam in (0.0, 1.5e-3, 1.0):
        ri, rv, re_ = oracle.ef_hard_threshold(g, e, 0.1, lam)
        gi, gv, ge, gt = _ht_tiled(g, e, 0.1, lam)
        gu.assert_bits(gi, ri, "idx")
        gu.assert_bits(gv, rv, "val")
        gu.assert_bits(ge, re_, "e'")
        gu.assert_bits(gt, _tile_index(ri, d), "tile index d=%d lam=%g" % (d, lam))
    assert efs.ef_check_status() == efs.EF_OK


@pytest.mark.usefixtures("ht_stream_kernel")
@pytest.mark.parametrize("offs", [(0, 0), (1, 0)])
def test_tile_index_with_the_error_norm(offs):
    # both optional outputs of ef_hard_threshold_tiled at once, on the
    # streaming and on the misaligned path; the norm within the relative
    # 1e-6 of the error-norm tests, the other outputs bit-exact
    d = 3 * 2**20 + 4099
    g, e = _inputs(d, 3)
    ri, rv, re_ = oracle.ef_hard_threshold(g, e, 0.1, 1.5e-3)
    gd, ed = gu.g_device(g, offs[0]), gu.to_dev(e, offs[1])
    idx = torch.empty(d, dtype=torch.int32, device=DEV)
    val = torch.empty(d, dtype=torch.float32, device=DEV)
    cnt = torch.empty(1, dtype=torch.int32, device=DEV)
    tiles = torch.empty(efs.tiles_for(d), dtype=torch.int32, device=DEV)
    err = torch.full((1,), float("nan"), dtype=torch.float64, device=DEV)
    efs.ef_hard_threshold(gd, ed, 0.1, 1.5e-3, idx, val, cnt, err_sq_out=err, tiles_out=tiles)
    c = int(cnt.item())
    gu.assert_bits(idx[:c].cpu().numpy().view(np.uint32), ri, "idx")
    gu.assert_bits(val[:c].cpu().numpy(), rv, "val")
    gu.assert_bits(ed.cpu().numpy(), re_, "e'")
    gu.assert_bits(tiles.cpu().numpy().view(np.uint32), _tile_index(ri, d), "tile index")
    want = oracle.error_norm_sq(re_)
    assert abs(float(err.item()) - want) <= 1e-6 * want
    assert efs.ef_check_status() == efs.EF_OK


@pytest.mark.parametrize("offs", [(1, 0), (0, 3)])
def test_tile_index_on_the_misaligned_path(offs):
    d = 5 * 4096 + 999
    g, e = _inputs(d, 2)
    ri, rv, re_ = oracle.ef_hard_threshold(g, e, 0.1, 1.5e-3)
    gi, gv, ge, gt = _ht_tiled(g, e, 0.1, 1.5e-3, g_off=offs[0], e_off=offs[1])
    gu.assert_bits(gi, ri, "idx")
    gu.assert_bits(ge, re_, "e'")
    gu.assert_bits(gt, _tile_index(ri, d), "tile index")


def test_tile_index_of_an_empty_vector():
    gd, ed = gu.to_dev(np.zeros(1, np.float32))[:0], gu.to_dev(np.zeros(1, np.float32))[:0]
    idx = torch.zeros(1, dtype=torch.int32, device=DEV)
    val = torch.zeros(1, dtype=torch.float32, device=DEV)
    cnt = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    tiles = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    efs.ef_hard_threshold(gd, ed, 0.1, 1e-3, idx, val, cnt, tiles_out=tiles)
    assert int(cnt.item()) == 0 and int(tiles.item()) == 0


@pytest.mark.usefixtures("stream_kernel")
@pytest.mark.parametrize("d", [4097, 100_003, 3 * 2**20 + 4099])
def test_tiled_aggregation_matches(d):
    n = 8
    idx_l, val_l, tiles_l, ri_l, rv_l = [], [], [], [], []
    cap = efs.tiles_for(d)
    for i in range(n):
        g, e = _inputs(d, 10 + i)
        ri, rv, _ = oracle.ef_hard_threshold(g, e, 0.1, 1.5e-3)
        gi, gv, _, gt = _ht_tiled(g, e, 0.1, 1.5e-3)
        gu.assert_bits(gt, _tile_index(ri, d), "tile index")
        idx_l.append(gu.to_dev(gi.view(np.int32)) if gi.size
                     else torch.zeros(1, dtype=torch.int32, device=DEV))
        val_l.append(gu.to_dev(gv) if gv.size else torch.zeros(1, device=DEV))
        tiles_l.append(gu.to_dev(gt.view(np.int32)))
        ri_l.append(ri)
        rv_l.append(rv)
    assert all(t.numel() == cap for t in tiles_l)
    counts = torch.tensor([x.size for x in ri_l], dtype=torch.int32, device=DEV)
    want = oracle.sparse_aggregate(ri_l, rv_l, d)
    dense = torch.full((d,), float("nan"), device=DEV)
    efs.sparse_aggregate(idx_l, val_l, counts, d, dense, tiles=tiles_l)
    gu.assert_bits(dense.cpu().numpy(), want, "tiled sum")
    rng = _rng("x", d)
    x0 = rng.standard_normal(d).astype(np.float32)
    m0 = rng.standard_normal(d).astype(np.float32)
    xw, mw = oracle.sparse_aggregate_apply(ri_l, rv_l, d, 0.125, x0, m0, 0.9, 0.1)
    x, m = gu.to_dev(x0), gu.to_dev(m0)
    efs.sparse_aggregate_apply(idx_l, val_l, counts, d, 0.125, x, m, 0.9, 0.1, tiles=tiles_l)
    gu.assert_bits(x.cpu().numpy(), xw, "tiled update x")
    gu.assert_bits(m.cpu().numpy(), mw, "tiled update m")
    assert efs.ef_check_status() == efs.EF_OK


def test_wrong_tile_index_stays_in_bounds():
    d = 5 * 4096 + 1
    lists = [np.array([3, 4100, 9000, 20000], np.uint32)]
    vals = [np.ones(4, np.float32)]
    idx = [gu.to_dev(lists[0].view(np.int32))]
    val = [gu.to_dev(vals[0])]
    counts = torch.tensor([4], dtype=torch.int32, device=DEV)
    t = efs.tiles_for(d)
    bad = [np.full(t, 0, np.uint32), np.full(t, 4_000_000_000, np.uint32),
           np.array([0, 3, 1, 4, 2, 4, 4][:t], np.uint32)]
    # clamped to the list: nothing read (all 0, all past the count), or pairs
    # read for tiles they do not belong to (skipped, latched)
    for b, latched in zip(bad, (False, False, True)):
        dense = torch.full((d,), float("nan"), device=DEV)
        efs.sparse_aggregate(idx, val, counts, d, dense, tiles=[gu.to_dev(b.view(np.int32))])
        out = dense.cpu().numpy()
        assert np.all(np.isfinite(out))
        st = efs.ef_check_status()
        assert st == (efs.EF_ERR_BAD_INPUT if latched else efs.EF_OK)
    # a correct index after the wrong ones
    good = _tile_index(lists[0], d)
    dense = torch.empty(d, device=DEV)
    efs.sparse_aggregate(idx, val, counts, d, dense, tiles=[gu.to_dev(good.view(np.int32))])
    gu.assert_bits(dense.cpu().numpy(), oracle.sparse_aggregate(lists, vals, d), "after")
    assert efs.ef_check_status() == efs.EF_OK
