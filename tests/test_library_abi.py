"""The C-ABI library builds, loads and exports every declared entry point;
host-side argument checks reject bad calls before any CUDA work (no GPU)."""
import ctypes
import os
import re

import pytest

import paper_2108_00951_gb300 as efs
from paper_2108_00951_gb300 import build

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                      "include", "efsparse.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return re.findall(r"^(?:ef_status|const char\s*\*|uint64_t|void)\s+(\w+)\s*\(", text, re.M)


def test_header_declares_the_boundary():
    names = set(declared_functions())
    for required in ("ef_hard_threshold", "ef_hard_threshold_bf16", "ef_topk", "ef_topk_bf16",
                     "sparse_aggregate", "ef_check_status", "ef_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol():
    lib = ctypes.CDLL(build.build())
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_status_strings():
    for code, name in [(0, "EF_OK"), (1, "EF_ERR_INVALID_ARG"), (2, "EF_ERR_CUDA"),
                       (3, "EF_ERR_TIMEOUT"), (4, "EF_ERR_BAD_INPUT"), (5, "EF_ERR_NO_MEMORY")]:
        assert efs.status_string(code) == name


# Host-side checks run before any CUDA call, so they work without a GPU. The
# pointers below are fake, 16-byte aligned, non-overlapping addresses; they
# are never dereferenced because every call is rejected first.
G, E, IDX, VAL, CNT = 0x10000000, 0x20000000, 0x30000000, 0x40000000, 0x50000000
vp = ctypes.c_void_p


def _ht(g=G, e=E, gamma=0.1, lam=1e-3, d=1000, idx=IDX, val=VAL, cnt=CNT, bf16=False):
    lib = efs.load_library()
    fn = lib.ef_hard_threshold_bf16 if bf16 else lib.ef_hard_threshold
    return fn(vp(g), vp(e), ctypes.c_float(gamma), ctypes.c_float(lam), d, vp(idx), vp(val),
              vp(cnt), vp(0))


def _topk(g=G, e=E, gamma=0.1, k=10, d=1000, idx=IDX, val=VAL, cnt=CNT):
    lib = efs.load_library()
    return lib.ef_topk(vp(g), vp(e), ctypes.c_float(gamma), k, d, vp(idx), vp(val), vp(cnt),
                       vp(0))


@pytest.mark.parametrize("kwargs", [
    dict(cnt=0), dict(g=0), dict(e=0), dict(idx=0), dict(val=0),
    dict(lam=-1e-3), dict(lam=float("nan")), dict(gamma=float("inf")), dict(gamma=float("nan")),
    dict(d=2 ** 32), dict(e=E + 2), dict(g=G + 1), dict(idx=IDX + 1), dict(cnt=CNT + 2),
    dict(idx=E + 64), dict(val=G), dict(val=IDX + 100), dict(cnt=VAL + 8), dict(e=G + 400),
])
def test_hard_threshold_rejects(kwargs):
    assert _ht(**kwargs) == efs.EF_ERR_INVALID_ARG


def test_hard_threshold_bf16_alignment_rule():
    assert _ht(g=G + 1, bf16=True) == efs.EF_ERR_INVALID_ARG      # bf16 needs 2-byte alignment


@pytest.mark.parametrize("kwargs", [
    dict(k=1001), dict(d=2 ** 32, k=1), dict(cnt=0), dict(g=0), dict(idx=0),
    dict(gamma=float("nan")), dict(val=E), dict(e=E + 1),
])
def test_topk_rejects(kwargs):
    assert _topk(**kwargs) == efs.EF_ERR_INVALID_ARG


def _layerwise(g=G, e=E, gamma=0.1, ends=(600, 1000), ks=(6, 4), d=1000, idx=IDX, val=VAL,
               cnt=CNT, n_seg=None):
    import numpy as np
    lib = efs.load_library()
    ends_a = np.ascontiguousarray(ends, dtype=np.uint64)
    ks_a = np.ascontiguousarray(ks, dtype=np.uint64)
    n = len(ends) if n_seg is None else n_seg
    return lib.ef_topk_layerwise(vp(g), vp(e), ctypes.c_float(gamma), ctypes.c_uint32(n),
                                 vp(ends_a.ctypes.data if ends_a.size else 0),
                                 vp(ks_a.ctypes.data if ks_a.size else 0), d, vp(idx), vp(val),
                                 vp(cnt), vp(0))


@pytest.mark.parametrize("kwargs", [
    dict(n_seg=0), dict(ends=(600, 999)), dict(ends=(600, 1001)), dict(ends=(700, 600, 1000),
                                                                        ks=(1, 0, 1)),
    dict(ks=(601, 4)), dict(ks=(6, 401)), dict(d=2 ** 32, ends=(600, 2 ** 32)), dict(cnt=0),
    dict(g=0), dict(idx=0), dict(gamma=float("inf")), dict(e=E + 2), dict(val=E),
    dict(idx=VAL - 20),  # 10 pairs overlap val
])
def test_topk_layerwise_rejects(kwargs):
    assert _layerwise(**kwargs) == efs.EF_ERR_INVALID_ARG


def test_aggregate_rejects():
    lib = efs.load_library()
    arr = (vp * 1)(vp(IDX))
    varr = (vp * 1)(vp(VAL))
    assert lib.sparse_aggregate(0, arr, varr, vp(CNT), 100, vp(G), vp(0)) == efs.EF_ERR_INVALID_ARG
    assert lib.sparse_aggregate(257, arr, varr, vp(CNT), 100, vp(G), vp(0)) == efs.EF_ERR_INVALID_ARG
    assert lib.sparse_aggregate(1, arr, varr, vp(0), 100, vp(G), vp(0)) == efs.EF_ERR_INVALID_ARG
    assert lib.sparse_aggregate(1, arr, varr, vp(CNT), 100, vp(0), vp(0)) == efs.EF_ERR_INVALID_ARG
    assert lib.sparse_aggregate(1, arr, varr, vp(CNT), 2 ** 32, vp(G), vp(0)) == efs.EF_ERR_INVALID_ARG
    bad = (vp * 1)(vp(0))
    assert lib.sparse_aggregate(1, bad, varr, vp(CNT), 100, vp(G), vp(0)) == efs.EF_ERR_INVALID_ARG
    assert lib.sparse_aggregate(1, arr, varr, vp(CNT), 100, vp(G + 1), vp(0)) == efs.EF_ERR_INVALID_ARG


def test_aggregate_apply_rejects():
    lib = efs.load_library()
    arr = (vp * 1)(vp(IDX))
    varr = (vp * 1)(vp(VAL))
    f = ctypes.c_float

    def call(n=1, cnt=CNT, d=100, alpha=0.5, x=G, m=E, mu=0.9, lr=0.1):
        return lib.sparse_aggregate_apply(n, arr, varr, vp(cnt), d, f(alpha), vp(x), vp(m), f(mu),
                                          f(lr), vp(0))
    for kwargs in (dict(n=0), dict(n=257), dict(cnt=0), dict(d=2 ** 32), dict(x=0),
                   dict(x=G + 2), dict(m=E + 1), dict(m=G + 200), dict(alpha=float("nan")),
                   dict(mu=float("inf")), dict(lr=float("nan"))):
        assert call(**kwargs) == efs.EF_ERR_INVALID_ARG, kwargs


TILES = 0x60000000


def _ht_tiled(tiles=TILES, d=1000, err=0, **kw):
    lib = efs.load_library()
    a = dict(g=G, e=E, idx=IDX, val=VAL, cnt=CNT)
    a.update(kw)
    return lib.ef_hard_threshold_tiled(vp(a["g"]), 0, vp(a["e"]), ctypes.c_float(0.1),
                                       ctypes.c_float(1e-3), d, vp(a["idx"]), vp(a["val"]),
                                       vp(a["cnt"]), vp(tiles), vp(err), vp(0))


@pytest.mark.parametrize("kwargs", [
    dict(tiles=0), dict(tiles=TILES + 2),
    dict(tiles=IDX + 3996),   # the index's 2 words overlap the last index entry
    dict(tiles=CNT - 4),      # its second word is the count
    dict(tiles=E + 100), dict(tiles=G),
    dict(err=TILES + 4),      # the error norm inside the index
    dict(cnt=0), dict(g=G + 1),
])
def test_hard_threshold_tiled_rejects(kwargs):
    assert _ht_tiled(**kwargs) == efs.EF_ERR_INVALID_ARG


def test_aggregate_tiled_rejects():
    lib = efs.load_library()
    arr = (vp * 1)(vp(IDX))
    varr = (vp * 1)(vp(VAL))
    tarr = (vp * 1)(vp(TILES))
    f = ctypes.c_float
    assert lib.sparse_aggregate_tiled(1, arr, varr, None, vp(CNT), 100, vp(G),
                                      vp(0)) == efs.EF_ERR_INVALID_ARG
    for t in (0, TILES + 2):
        bad = (vp * 1)(vp(t))
        assert lib.sparse_aggregate_tiled(1, arr, varr, bad, vp(CNT), 100, vp(G),
                                          vp(0)) == efs.EF_ERR_INVALID_ARG
        assert lib.sparse_aggregate_apply_tiled(1, arr, varr, bad, vp(CNT), 100, f(0.5), vp(G),
                                                vp(E), f(0.9), f(0.1),
                                                vp(0)) == efs.EF_ERR_INVALID_ARG
    assert lib.sparse_aggregate_tiled(0, arr, varr, tarr, vp(CNT), 100, vp(G),
                                      vp(0)) == efs.EF_ERR_INVALID_ARG
    assert lib.sparse_aggregate_apply_tiled(1, arr, varr, None, vp(CNT), 100, f(0.5), vp(G), vp(E),
                                            f(0.9), f(0.1), vp(0)) == efs.EF_ERR_INVALID_ARG
    assert lib.sparse_aggregate_apply_tiled(1, arr, varr, tarr, vp(CNT), 100, f(0.5), vp(0), vp(E),
                                            f(0.9), f(0.1), vp(0)) == efs.EF_ERR_INVALID_ARG


def test_binding_fails_loudly_on_cpu_tensors():
    torch = pytest.importorskip("torch")
    x = torch.zeros(8)
    i = torch.zeros(8, dtype=torch.int32)
    with pytest.raises(TypeError):
        efs.ef_hard_threshold(x, x.clone(), 0.1, 1e-3, i, x.clone(), i[:1])


ST = 0x60000000


def _noalloc(g=G, e=E, gamma=0.1, lam=1e-3, d=1000, idx=IDX, val=VAL, cnt=CNT, status=ST):
    lib = efs.load_library()
    fn = lib.ef_hard_threshold_noalloc
    fn.argtypes = [vp, vp, ctypes.c_float, ctypes.c_float, ctypes.c_uint64, vp, vp, vp, vp, vp]
    fn.restype = ctypes.c_int
    return fn(vp(g), vp(e), gamma, lam, d, vp(idx), vp(val), vp(cnt), vp(status), vp(0))


@pytest.mark.parametrize("kwargs", [
    dict(d=(1 << 28) + 1), dict(cnt=0), dict(g=0), dict(e=0), dict(idx=0), dict(val=0),
    dict(lam=-1.0), dict(gamma=float("nan")), dict(e=E + 2), dict(status=ST + 2),
    dict(idx=E + 64), dict(cnt=VAL + 8),
    # the status word may not overlap any other buffer
    dict(status=G), dict(status=E + 400), dict(status=IDX + 3996), dict(status=VAL),
    dict(status=CNT), dict(d=0, status=CNT),
])
def test_noalloc_rejects(kwargs):
    assert _noalloc(**kwargs) == efs.EF_ERR_INVALID_ARG
