"""GPU parity of layer-wise Top-k: the CUDA path against the CPU oracle, bit
for bit (indices, sent values, residuals).

The cases reach every selection route of the kernels: segments that send
nothing, that send everything, that fit one CTA's shared memory whole, that
are sampled and selected from a short candidate list, from a candidate list
too long for shared memory, from e itself (the sampled bound would admit too
many candidates), and segments whose candidates were cut off at the list's
capacity; plus ties, zeros, NaN and infinities, bf16 gradients, misaligned
bases, several EF iterations on one workspace, a changing segment table, and
calls interleaved with entire-vector Top-k. At the benchmark's full sizes the
ResNet-18 table is compared with the oracle over two iterations; the others
are checked against properties that fix the per-segment Top-k uniquely.
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


def _ends(sizes):
    return np.cumsum(np.asarray(sizes, dtype=np.uint64)).astype(np.uint64)


def _inputs(d, seed, bf16=False):
    rng = _rng("lw", d, seed)
    g = (rng.standard_normal(d) * 1e-2).astype(np.float32)
    e = (rng.standard_normal(d) * 1e-3).astype(np.float32)
    if bf16:
        g = torch.from_numpy(g).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    return g, e


def _check(g, e, gamma, sizes, ks, what, g_off=0, e_off=0):
    ends = _ends(sizes)
    ref = oracle.ef_topk_layerwise(g, e, gamma, ends, ks)
    got = gu.topk_layerwise(g, e, gamma, ends, ks, g_off=g_off, e_off=e_off)
    gu.assert_bits(got[0], ref[0], what + " idx")
    gu.assert_bits(got[1], ref[1], what + " val")
    gu.assert_bits(got[2], ref[2], what + " e'")
    assert efs.ef_check_status() == efs.EF_OK, what
    return ref


# sizes and budgets that reach each kind of segment: empty, nothing sent,
# everything sent, selected from e whole (<= 4096), sampled at every aligned
# group (<= 65536), sampled sparsely (> 65536), at unaligned boundaries
KINDS_SIZES = [0, 5, 64, 4097, 49152, 49153, 100_003, 3 * 4096 + 17, 1, 200_000, 7, 65_536,
               4096, 65_537, 2]
KINDS_K = [0, 5, 3, 40, 491, 1, 1000, 0, 1, 2000, 6, 65_535, 4095, 66, 1]


@pytest.mark.usefixtures("stream_kernel")
@pytest.mark.parametrize("bf16", [False, True])
def test_layerwise_every_kind(bf16):
    g, e = _inputs(sum(KINDS_SIZES), 1, bf16=bf16)
    _check(g, e, 0.1, KINDS_SIZES, KINDS_K, "kinds bf16=%s" % bf16)


@pytest.mark.parametrize("offs", [(1, 0), (0, 1), (3, 2)])
def test_layerwise_misaligned_bases(offs):
    g, e = _inputs(sum(KINDS_SIZES), 2)
    _check(g, e, 0.1, KINDS_SIZES, KINDS_K, "offsets %s" % (offs,), g_off=offs[0], e_off=offs[1])


@pytest.mark.usefixtures("stream_kernel")
def test_layerwise_single_segment_is_entire_vector_topk():
    d, k = 300_001, 3000
    g, e = _inputs(d, 3)
    ref = _check(g, e, 0.1, [d], [k], "one segment")
    ti, tv, te = oracle.ef_topk(g, e, 0.1, k)
    gu.assert_bits(ref[0], ti, "idx vs entire")
    gu.assert_bits(ref[2], te, "e' vs entire")


@pytest.mark.usefixtures("stream_kernel")
def test_layerwise_candidates_beyond_shared_memory():
    # one sampled segment whose candidate list exceeds a CTA's shared memory
    sizes, ks = [400_000, 70_000], [60_000, 700]
    g, e = _inputs(sum(sizes), 4)
    _check(g, e, 0.1, sizes, ks, "long candidate list")


@pytest.mark.usefixtures("stream_kernel")
def test_layerwise_long_list_from_ties_one_cta():
    # a modest k whose cut falls inside a block of 100,000 equal magnitudes:
    # the candidates far exceed shared memory but the segment is not given a
    # team, so one CTA selects from the list in global memory
    rng = _rng("tieblock")
    n = 200_000
    e = (rng.standard_normal(n + 5000) * 1e-3).astype(np.float32)
    e[:10_000] = (1.0 + np.arange(10_000, dtype=np.float32) * 1e-4)[rng.permutation(10_000)]
    block = rng.permutation(np.arange(10_000, n))[:100_000]
    e[block] = np.where(rng.random(100_000) < 0.5, 0.5, -0.5).astype(np.float32)
    g = np.zeros(n + 5000, np.float32)
    _check(g, e, 1.0, [n, 5000], [15_000, 5], "tie block")


@pytest.mark.usefixtures("stream_kernel")
def test_layerwise_bound_admits_too_many():
    # half of a large segment: the candidates would not fit, so the segment
    # is selected from e itself
    sizes, ks = [1_500_000, 1_500_003], [750_000, 10]
    g, e = _inputs(sum(sizes), 5)
    _check(g, e, 0.1, sizes, ks, "selection from e")


@pytest.mark.usefixtures("stream_kernel")
def test_layerwise_candidate_list_cut_off():
    # the segments' candidates together overflow the list's capacity: the
    # segments whose candidates were cut off are selected from e
    sizes = [1_000_000] * 5 + [4099]
    ks = [150_000] * 5 + [17]
    g, e = _inputs(sum(sizes), 6)
    _check(g, e, 0.1, sizes, ks, "cut-off list")


@pytest.mark.usefixtures("stream_kernel")
def test_layerwise_ties_zeros_nan_inf():
    rng = _rng("ties")
    sizes = [60_000, 30_000, 120_000, 9, 50_000]
    d = sum(sizes)
    pool = np.array([0.5, -0.5, 0.25, 0.0, -0.0, 1.0, -1.0], np.float32)
    e = pool[rng.integers(0, len(pool), d)]
    g = np.zeros(d, np.float32)
    # segment 1 all zero but a few; segment 3 NaN and infinities
    lo1 = sizes[0]
    e[lo1:lo1 + sizes[1]] = 0.0
    e[lo1 + rng.integers(0, sizes[1], 10)] = 2.0
    lo3 = sum(sizes[:3])
    e[lo3:lo3 + 9] = np.array([np.nan, 1, np.inf, -np.inf, 0, np.nan, -2, 3, 0], np.float32)
    lo4 = sum(sizes[:4])
    e[lo4 + rng.integers(0, sizes[4], 50)] = np.nan
    ks = [7_000, 100, 30_000, 4, 60]
    _check(g, e, 1.0, sizes, ks, "ties")


@pytest.mark.usefixtures("stream_kernel")
def test_layerwise_iterations_table_change_and_interleaving():
    sizes_a = [70_000, 1_000, 200_003, 4_096, 55_555]
    sizes_b = [100_000, 230_654]  # same d, another table
    d = sum(sizes_a)
    assert d == sum(sizes_b)
    ks_a = [70, 1, 2000, 40, 555]
    ks_b = [1000, 2306]
    rng = _rng("iters")
    e_gpu = torch.zeros(d, device=DEV)
    e_ref = np.zeros(d, np.float32)
    idx = torch.empty(d, dtype=torch.int32, device=DEV)
    val = torch.empty(d, dtype=torch.float32, device=DEV)
    cnt = torch.empty(1, dtype=torch.int32, device=DEV)
    plan = ["a", "a", "a", "b", "topk", "a", "b", "b"]
    for t, which in enumerate(plan):
        g = (rng.standard_normal(d) * 1e-2).astype(np.float32)
        gd = gu.to_dev(g)
        if which == "topk":
            k = 4321
            efs.ef_topk(gd, e_gpu, 0.1, k, idx, val, cnt)
            ri, rv, e_ref = oracle.ef_topk(g, e_ref, 0.1, k)
        else:
            sizes, ks = (sizes_a, ks_a) if which == "a" else (sizes_b, ks_b)
            efs.ef_topk_layerwise(gd, e_gpu, 0.1, _ends(sizes), ks, idx, val, cnt)
            ri, rv, e_ref = oracle.ef_topk_layerwise(g, e_ref, 0.1, _ends(sizes), ks)
        torch.cuda.synchronize()
        c = int(cnt.item())
        assert c == ri.size, (t, which)
        gu.assert_bits(idx[:c].cpu().numpy().view(np.uint32), ri, "iter %d idx" % t)
        gu.assert_bits(val[:c].cpu().numpy(), rv, "iter %d val" % t)
        gu.assert_bits(e_gpu.cpu().numpy(), e_ref, "iter %d e'" % t)
    assert efs.ef_check_status() == efs.EF_OK


def test_layerwise_zero_length_and_nothing_sent():
    cnt = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    empty = torch.empty(0, device=DEV)
    efs.ef_topk_layerwise(empty, empty, 0.1, [0], [0], torch.empty(1, dtype=torch.int32,
                                                                   device=DEV),
                          torch.empty(1, device=DEV), cnt)
    torch.cuda.synchronize()
    assert int(cnt.item()) == 0
    g, e = _inputs(10_000, 7)
    _check(g, e, 0.1, [4_000, 6_000], [0, 0], "nothing sent")


# ------------------------------------------------------------ full sizes
def _check_layerwise_properties(a, ends, ks, gi, gv, ge):
    d = a.size
    assert gi.size == int(np.sum(ks))
    assert np.all(gi[1:] > gi[:-1]) and (gi.size == 0 or gi[-1] < d)
    gu.assert_bits(gv, a[gi], "values")
    want = a.copy()
    want[gi] = 0.0
    gu.assert_bits(ge, want, "residual")
    starts = np.concatenate([[0], ends[:-1]]).astype(np.int64)
    per_seg = np.diff(np.searchsorted(gi, np.concatenate([[0], ends]).astype(np.int64)))
    assert np.array_equal(per_seg, np.asarray(ks, dtype=np.int64)), "per-segment counts"
    key = ((a.view(np.uint32) & np.uint32(0x7fffffff)).astype(np.uint64) << np.uint64(32)) | \
        (~np.arange(d, dtype=np.uint32)).astype(np.uint64)
    sel = np.zeros(d, bool)
    sel[gi] = True
    nonempty = starts < ends.astype(np.int64)
    st = starts[nonempty]
    min_sel = np.minimum.reduceat(np.where(sel, key, np.uint64(2 ** 64 - 1)), st)
    max_uns = np.maximum.reduceat(np.where(sel, np.uint64(0), key), st)
    k_ne = np.asarray(ks, dtype=np.int64)[nonempty]
    n_ne = (ends.astype(np.int64) - starts)[nonempty]
    partial = (k_ne > 0) & (k_ne < n_ne)
    assert np.all(min_sel[partial] > max_uns[partial]), "per-segment order"


@pytest.mark.parametrize("name,frac,dtype", [("resnet18", 1e-3, torch.float32),
                                             ("lstm", 1e-2, torch.float32),
                                             ("resnet50", 1e-3, torch.float32),
                                             ("resnet50", 1e-2, torch.float32),
                                             ("vgg16", 1e-4, torch.float32),
                                             ("vgg16", 1e-4, torch.bfloat16)])
def test_full_size_layerwise(name, frac, dtype):
    w = workloads.BY_NAME[name]
    ends = np.asarray(workloads.segment_ends(w), dtype=np.uint64)
    ks = workloads.layerwise_k(w, frac)
    total = sum(ks)
    idx = torch.empty(total, dtype=torch.int32, device=DEV)
    val = torch.empty(total, dtype=torch.float32, device=DEV)
    cnt = torch.empty(1, dtype=torch.int32, device=DEV)
    e_gpu = torch.zeros(w.d, device=DEV)
    e_ref = np.zeros(w.d, np.float32)
    iterations = 2 if name == "resnet18" else 1
    for t in range(iterations):
        g = workloads.gradient(w, 0, t, device=DEV, dtype=dtype)
        g_host = g.view(torch.int16).cpu().numpy().view(np.uint16) \
            if dtype == torch.bfloat16 else g.cpu().numpy()
        e_before = e_ref
        efs.ef_topk_layerwise(g, e_gpu, w.gamma, ends, ks, idx, val, cnt)
        assert int(cnt.item()) == total
        gi = idx.cpu().numpy().view(np.uint32)
        gv = val.cpu().numpy()
        ge = e_gpu.cpu().numpy()
        _, _, a = oracle.ef_hard_threshold(g_host, e_before, w.gamma, float("inf"))
        _check_layerwise_properties(a, ends, ks, gi, gv, ge)
        if name == "resnet18":
            ri, rv, e_ref = oracle.ef_topk_layerwise(g_host, e_before, w.gamma, ends, ks)
            gu.assert_bits(gi, ri, "idx")
            gu.assert_bits(gv, rv, "val")
            gu.assert_bits(ge, e_ref, "e'")
        else:
            e_ref = ge
    assert efs.ef_check_status() == efs.EF_OK
