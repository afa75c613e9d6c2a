"""The largest sizes the API admits: indices past 2^31 (hard-threshold and
Top-k at d = 2^31 + 4099) and the aggregate at d = 2^32 - 1, the API's
maximum. The oracle cannot run at these sizes in seconds, so the results are
checked exactly against plain PyTorch computations of the same definitions,
a chunk of the vector at a time, on the device:

  a = RN(gamma * g) (e starts at zero, so fmaf(gamma, g, e) = RN(gamma * g)),
  hard-threshold: the sent set is {j : |a_j| >= lambda, a_j != 0} in order,
  the values are a at those indices, the residual is a with them zeroed;
  Top-k: k ascending indices, values a at them, residual zero there, and no
  unsent magnitude above the smallest sent one (equal magnitudes: the sent
  ones have the lower indices).
"""
import numpy as np
import pytest
import torch

import paper_2108_00951_gb300 as efs

pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

DEV = torch.device("cuda:0")
D_BIG = 2**31 + 4099
CHUNK = 2**28
GAMMA = 0.1


def _need(gib):
    free, _ = torch.cuda.mem_get_info()
    if free < gib * 2**30:
        pytest.skip("needs %d GiB of free device memory" % gib)


def _gradient(d, seed):
    gen = torch.Generator(device=DEV).manual_seed(seed)
    return torch.randn(d, generator=gen, device=DEV, dtype=torch.float32).to(torch.bfloat16)


def _u32(t):
    return t.to(torch.int64) & 0xFFFFFFFF


def _a(g, s, t):
    return g[s:t].float() * GAMMA


def test_hard_threshold_indices_past_2_31():
    _need(70)
    d = D_BIG
    g = _gradient(d, 7)
    e = torch.zeros(d, device=DEV)
    idx = torch.empty(d, dtype=torch.int32, device=DEV)
    val = torch.empty(d, dtype=torch.float32, device=DEV)
    cnt = torch.zeros(1, dtype=torch.int32, device=DEV)
    lam = 0.37  # |N(0,1)| * 0.1 >= 0.37: about 2e-4 of the coordinates
    efs.ef_hard_threshold(g, e, GAMMA, lam, idx, val, cnt)
    assert efs.ef_check_status() == efs.EF_OK
    c = int(_u32(cnt)[0])
    pos = 0
    for s in range(0, d, CHUNK):
        t = min(d, s + CHUNK)
        a = _a(g, s, t)
        mask = (a.abs() >= lam) & (a != 0)
        nz = torch.nonzero(mask).flatten() + s
        m = nz.numel()
        assert pos + m <= c
        assert torch.equal(_u32(idx[pos:pos + m]), nz), "indices in [%d, %d)" % (s, t)
        assert torch.equal(val[pos:pos + m], a[mask]), "values in [%d, %d)" % (s, t)
        assert torch.equal(e[s:t], torch.where(mask, torch.zeros_like(a), a)), "residual"
        pos += m
    assert pos == c and c > 2**17
    assert int(_u32(idx[c - 1:c])[0]) >= 2**31  # indices past 2^31 were sent


def test_topk_indices_past_2_31():
    _need(70)
    d, k = D_BIG, 4096
    g = _gradient(d, 8)
    # plant the largest magnitudes past 2^31, with ties across the 2^31 line
    big = torch.tensor([9.0, -9.0, 8.0, 9.0], dtype=torch.bfloat16, device=DEV)
    where = torch.tensor([5, 2**31 - 1, 2**31 + 17, d - 1], device=DEV)
    g[where] = big
    e = torch.zeros(d, device=DEV)
    idx = torch.empty(k, dtype=torch.int32, device=DEV)
    val = torch.empty(k, dtype=torch.float32, device=DEV)
    cnt = torch.zeros(1, dtype=torch.int32, device=DEV)
    efs.ef_topk(g, e, GAMMA, k, idx, val, cnt)
    assert efs.ef_check_status() == efs.EF_OK
    assert int(cnt[0]) == k
    gi = _u32(idx)
    assert bool((gi[1:] > gi[:-1]).all()) and int(gi[-1]) < d
    assert set(where.tolist()) <= set(gi.tolist())
    # values and residual at the sent indices
    a_at = g[gi].float() * GAMMA
    assert torch.equal(val, a_at)
    assert bool((e[gi] == 0).all())
    m = float(val.abs().min())
    top_sent_at_m = int(gi[val.abs() == m].max())
    for s in range(0, d, CHUNK):
        t = min(d, s + CHUNK)
        a = _a(g, s, t)
        sent = torch.zeros(t - s, dtype=torch.bool, device=DEV)
        inside = (gi >= s) & (gi < t)
        sent[gi[inside] - s] = True
        assert torch.equal(e[s:t], torch.where(sent, torch.zeros_like(a), a)), "residual"
        rest = a.abs()[~sent]
        assert float(rest.max()) <= m
        tied = torch.nonzero((a.abs() == m) & ~sent).flatten() + s
        assert tied.numel() == 0 or int(tied.min()) > top_sent_at_m


def test_aggregate_at_the_maximum_d():
    _need(24)
    d = 2**32 - 1
    lists = [np.array([0, 5, 4095, 4096], np.uint64),
             np.array([2**31 - 1, 2**31, 2**31 + 1, 2**32 - 3], np.uint64),
             np.array([5, 2**31, 2**32 - 3, 2**32 - 2], np.uint64)]
    rng = np.random.default_rng(5)
    vals = [rng.standard_normal(len(x)).astype(np.float32) for x in lists]
    idx_t = [torch.from_numpy(x.astype(np.uint32).view(np.int32)).to(DEV) for x in lists]
    val_t = [torch.from_numpy(v).to(DEV) for v in vals]
    counts = torch.tensor([len(x) for x in lists], dtype=torch.int32, device=DEV)
    dense = torch.full((d,), float("nan"), dtype=torch.float32, device=DEV)
    efs.sparse_aggregate(idx_t, val_t, counts, d, dense)
    assert efs.ef_check_status() == efs.EF_OK
    expect = {}
    for x, v in zip(lists, vals):  # worker order, from +0.0
        for j, y in zip(x.tolist(), v.tolist()):
            expect[j] = np.float32(expect.get(j, np.float32(0.0)) + np.float32(y))
    nonzero = 0
    for s in range(0, d, CHUNK):
        t = min(d, s + CHUNK)
        nonzero += int(torch.count_nonzero(dense[s:t]))
        assert not bool(torch.isnan(dense[s:t]).any())
    assert nonzero == len(expect)
    got = dense[torch.tensor(sorted(expect), device=DEV)].cpu().numpy()
    want = np.array([expect[j] for j in sorted(expect)], np.float32)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
