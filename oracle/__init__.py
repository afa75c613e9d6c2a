"""CPU oracle for the error-feedback sparsification step (arXiv:2108.00951).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / reference leg of ``bench.py`` may use this package; the
product library never does. The arithmetic lives in ``oracle.c`` (plain C,
single thread); this module only compiles it with gcc and marshals numpy
arrays through ctypes.

Functions (each follows Algorithm 1 of the paper; see oracle.c for the
passage behind every line):

* ``ef_hard_threshold(g, e, gamma, lam)`` — hard-threshold sparsifier
  S_lambda = {j : |a_j| >= lambda} (Sec. 1, Sec. 4.2).
* ``ef_topk(g, e, gamma, k)`` — Top-k sparsifier (Lemma 1, Lemma 2).
* ``ef_topk_layerwise(g, e, gamma, seg_end, seg_k)`` — Top-k invoked on each
  layer's tensor separately (Appendix, layer-wise sparsification).
* ``sparse_aggregate(idx_list, val_list, d)`` — worker-ordered sum of the
  decompressed vectors (Algorithm 1, exchange step).
* ``error_norm_sq(e)`` — ||e||^2 in fp64, the per-step term of the total error.
* ``ef_scaled_round(g, e, gamma, m)``, ``int_aggregate(q_list, d, m)`` — scaled
  integer rounding under EF (an absolute compressor, Sec. 5) and the exact
  integer exchange of its messages.
* ``sparse_aggregate_apply(idx_list, val_list, d, alpha, x, m, mu, lr)`` —
  that sum scaled by alpha, applied as Algorithm 1's model update, or as the
  momentum update of the Appendix's gradient-compression EF SGD.

Each compression function returns ``(idx, val, e_new)`` and leaves its inputs
untouched; ``g`` may be float32 or bfloat16 bit patterns (uint16).
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIBDIR = os.path.join(_HERE, "lib")
_LIB = os.path.join(_LIBDIR, "liboracle.so")
_CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into oracle/lib/liboracle.so with gcc; return the path."""
    os.makedirs(_LIBDIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp%d" % os.getpid()
        subprocess.run(["gcc", *_CFLAGS, "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            u32p = ctypes.POINTER(ctypes.c_uint32)
            f32p = ctypes.POINTER(ctypes.c_float)
            u16p = ctypes.POINTER(ctypes.c_uint16)
            for name, gp in (("oracle_ef_hard_threshold", f32p),
                             ("oracle_ef_hard_threshold_bf16", u16p)):
                fn = getattr(lib, name)
                fn.argtypes = [gp, f32p, ctypes.c_float, ctypes.c_float, ctypes.c_uint64,
                               u32p, f32p, u32p]
                fn.restype = ctypes.c_int
            for name, gp in (("oracle_ef_topk", f32p), ("oracle_ef_topk_bf16", u16p)):
                fn = getattr(lib, name)
                fn.argtypes = [gp, f32p, ctypes.c_float, ctypes.c_uint64, ctypes.c_uint64,
                               u32p, f32p, u32p]
                fn.restype = ctypes.c_int
            u64p = ctypes.POINTER(ctypes.c_uint64)
            for name, gp in (("oracle_ef_topk_layerwise", f32p),
                             ("oracle_ef_topk_layerwise_bf16", u16p)):
                fn = getattr(lib, name)
                fn.argtypes = [gp, f32p, ctypes.c_float, ctypes.c_uint32, u64p, u64p,
                               ctypes.c_uint64, u32p, f32p, u32p]
                fn.restype = ctypes.c_int
            lib.oracle_sparse_aggregate.argtypes = [
                ctypes.c_uint32, ctypes.POINTER(u32p), ctypes.POINTER(f32p), u32p,
                ctypes.c_uint64, f32p]
            lib.oracle_sparse_aggregate.restype = ctypes.c_int
            lib.oracle_sparse_aggregate_apply.argtypes = [
                ctypes.c_uint32, ctypes.POINTER(u32p), ctypes.POINTER(f32p), u32p,
                ctypes.c_uint64, ctypes.c_float, f32p, f32p, ctypes.c_float, ctypes.c_float]
            lib.oracle_sparse_aggregate_apply.restype = ctypes.c_int
            lib.oracle_error_norm_sq.argtypes = [f32p, ctypes.c_uint64]
            lib.oracle_error_norm_sq.restype = ctypes.c_double
            i32p = ctypes.POINTER(ctypes.c_int32)
            for name, gp in (("oracle_ef_scaled_round", f32p),
                             ("oracle_ef_scaled_round_bf16", ctypes.POINTER(ctypes.c_uint16))):
                fn = getattr(lib, name)
                fn.argtypes = [gp, f32p, ctypes.c_float, ctypes.c_int, ctypes.c_uint64, i32p, u32p]
                fn.restype = ctypes.c_int
            lib.oracle_int_aggregate.argtypes = [ctypes.c_uint32, ctypes.POINTER(i32p),
                                                 ctypes.c_uint64, ctypes.c_int, f32p]
            lib.oracle_int_aggregate.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(arr: np.ndarray, ctype):
    return arr.ctypes.data_as(ctypes.POINTER(ctype))


def _gradient(g: np.ndarray):
    g = np.ascontiguousarray(g)
    if g.dtype == np.float32:
        return g, ctypes.c_float, False
    if g.dtype == np.uint16:
        return g, ctypes.c_uint16, True
    raise TypeError("g must be float32 or uint16 (bfloat16 bit patterns)")


def ef_hard_threshold(g: np.ndarray, e: np.ndarray, gamma: float, lam: float):
    """One EF step with the hard-threshold sparsifier; returns (idx, val, e_new)."""
    lib = _load()
    g, gctype, is_bf16 = _gradient(g)
    e_new = np.array(e, dtype=np.float32, copy=True)
    d = e_new.size
    assert g.size == d
    idx = np.empty(max(d, 1), np.uint32)
    val = np.empty(max(d, 1), np.float32)
    cnt = np.zeros(1, np.uint32)
    fn = lib.oracle_ef_hard_threshold_bf16 if is_bf16 else lib.oracle_ef_hard_threshold
    rc = fn(_ptr(g, gctype), _ptr(e_new, ctypes.c_float), ctypes.c_float(gamma),
            ctypes.c_float(lam), d, _ptr(idx, ctypes.c_uint32), _ptr(val, ctypes.c_float),
            _ptr(cnt, ctypes.c_uint32))
    if rc != 0:
        raise RuntimeError("oracle_ef_hard_threshold failed (%d)" % rc)
    c = int(cnt[0])
    return idx[:c].copy(), val[:c].copy(), e_new


def ef_topk(g: np.ndarray, e: np.ndarray, gamma: float, k: int):
    """One EF step with the Top-k sparsifier; returns (idx, val, e_new)."""
    lib = _load()
    g, gctype, is_bf16 = _gradient(g)
    e_new = np.array(e, dtype=np.float32, copy=True)
    d = e_new.size
    assert g.size == d
    if not 0 <= k <= d:
        raise ValueError("need 0 <= k <= d")
    idx = np.empty(max(k, 1), np.uint32)
    val = np.empty(max(k, 1), np.float32)
    cnt = np.zeros(1, np.uint32)
    fn = lib.oracle_ef_topk_bf16 if is_bf16 else lib.oracle_ef_topk
    rc = fn(_ptr(g, gctype), _ptr(e_new, ctypes.c_float), ctypes.c_float(gamma), k, d,
            _ptr(idx, ctypes.c_uint32), _ptr(val, ctypes.c_float), _ptr(cnt, ctypes.c_uint32))
    if rc != 0:
        raise RuntimeError("oracle_ef_topk failed (%d)" % rc)
    c = int(cnt[0])
    return idx[:c].copy(), val[:c].copy(), e_new


def ef_topk_layerwise(g: np.ndarray, e: np.ndarray, gamma: float, seg_end, seg_k):
    """One EF step with layer-wise Top-k: segment s = [seg_end[s-1], seg_end[s])
    sends its seg_k[s] largest-magnitude coordinates; returns (idx, val, e_new)."""
    lib = _load()
    g, gctype, is_bf16 = _gradient(g)
    e_new = np.array(e, dtype=np.float32, copy=True)
    d = e_new.size
    assert g.size == d
    ends = np.ascontiguousarray(seg_end, dtype=np.uint64)
    ks = np.ascontiguousarray(seg_k, dtype=np.uint64)
    n_seg = ends.size
    if n_seg < 1 or ks.size != n_seg:
        raise ValueError("need one k per segment and at least one segment")
    total = int(ks.sum())
    idx = np.empty(max(total, 1), np.uint32)
    val = np.empty(max(total, 1), np.float32)
    cnt = np.zeros(1, np.uint32)
    fn = lib.oracle_ef_topk_layerwise_bf16 if is_bf16 else lib.oracle_ef_topk_layerwise
    rc = fn(_ptr(g, gctype), _ptr(e_new, ctypes.c_float), ctypes.c_float(gamma), n_seg,
            _ptr(ends, ctypes.c_uint64), _ptr(ks, ctypes.c_uint64), d,
            _ptr(idx, ctypes.c_uint32), _ptr(val, ctypes.c_float), _ptr(cnt, ctypes.c_uint32))
    if rc != 0:
        raise ValueError("oracle_ef_topk_layerwise rejected the segment table (%d)" % rc)
    c = int(cnt[0])
    return idx[:c].copy(), val[:c].copy(), e_new


def _lists(idx_list, val_list):
    n = len(idx_list)
    assert n == len(val_list) and n >= 1
    idx_arrs = [np.ascontiguousarray(x, dtype=np.uint32) for x in idx_list]
    val_arrs = [np.ascontiguousarray(v, dtype=np.float32) for v in val_list]
    # keep zero-length lists addressable
    idx_arrs = [a if a.size else np.zeros(1, np.uint32) for a in idx_arrs]
    val_arrs = [v if v.size else np.zeros(1, np.float32) for v in val_arrs]
    counts = np.array([len(x) for x in idx_list], dtype=np.uint32)
    for i in range(n):
        assert len(val_list[i]) == counts[i]
    u32p = ctypes.POINTER(ctypes.c_uint32)
    f32p = ctypes.POINTER(ctypes.c_float)
    idx_ptrs = (u32p * n)(*[_ptr(a, ctypes.c_uint32) for a in idx_arrs])
    val_ptrs = (f32p * n)(*[_ptr(v, ctypes.c_float) for v in val_arrs])
    return n, idx_arrs, val_arrs, counts, idx_ptrs, val_ptrs


def sparse_aggregate_apply(idx_list, val_list, d: int, alpha: float, x, m=None, mu: float = 0.0,
                           lr: float = 0.0):
    """Model update from the worker-ordered sum s of n sparse vectors:
    Delta' = alpha * s; without ``m``: x <- x - Delta'; with ``m``:
    m <- fmaf(mu, m, Delta'), x <- fmaf(-lr, Delta' + m, x). Returns
    (x_new, m_new or None); the inputs are left untouched."""
    lib = _load()
    n, idx_arrs, val_arrs, counts, idx_ptrs, val_ptrs = _lists(idx_list, val_list)
    x_new = np.array(x, dtype=np.float32, copy=True).reshape(-1)
    assert x_new.size == d
    m_new = None if m is None else np.array(m, dtype=np.float32, copy=True).reshape(-1)
    if m_new is not None:
        assert m_new.size == d
    f32p = ctypes.POINTER(ctypes.c_float)
    xb = x_new if d else np.zeros(1, np.float32)
    mb = None if m_new is None else (m_new if d else np.zeros(1, np.float32))
    rc = lib.oracle_sparse_aggregate_apply(
        n, idx_ptrs, val_ptrs, _ptr(counts, ctypes.c_uint32), d, ctypes.c_float(alpha),
        _ptr(xb, ctypes.c_float), ctypes.cast(None, f32p) if mb is None else _ptr(mb, ctypes.c_float),
        ctypes.c_float(mu), ctypes.c_float(lr))
    if rc != 0:
        raise RuntimeError("oracle_sparse_aggregate_apply: index out of range")
    return x_new, m_new


def ef_scaled_round(g: np.ndarray, e: np.ndarray, gamma: float, m: int):
    """One EF step with scaled integer rounding: q = RNE(a 2^m) (int32),
    C(a) = q 2^-m, e' = a - C(a); coordinates that do not fit are kept in e.
    Returns (q, e_new, unsent)."""
    lib = _load()
    g, gctype, is_bf16 = _gradient(g)
    e_new = np.array(e, dtype=np.float32, copy=True)
    d = e_new.size
    q = np.empty(max(d, 1), np.int32)
    unsent = np.zeros(1, np.uint32)
    fn = lib.oracle_ef_scaled_round_bf16 if is_bf16 else lib.oracle_ef_scaled_round
    fn(_ptr(g, gctype), _ptr(e_new, ctypes.c_float), ctypes.c_float(gamma), int(m), d,
       _ptr(q, ctypes.c_int32), _ptr(unsent, ctypes.c_uint32))
    return q[:d].copy(), e_new, int(unsent[0])


def int_aggregate(q_list, d: int, m: int) -> np.ndarray:
    """Exact integer sum of n dense messages, decompressed as RN(S) 2^-m."""
    lib = _load()
    n = len(q_list)
    arrs = [np.ascontiguousarray(q, dtype=np.int32) for q in q_list]
    arrs = [a if a.size else np.zeros(1, np.int32) for a in arrs]
    i32p = ctypes.POINTER(ctypes.c_int32)
    ptrs = (i32p * n)(*[_ptr(a, ctypes.c_int32) for a in arrs])
    dense = np.empty(max(d, 1), np.float32)
    lib.oracle_int_aggregate(n, ptrs, d, int(m), _ptr(dense, ctypes.c_float))
    return dense[:d].copy()


def error_norm_sq(e) -> float:
    """||e||^2 = sum_j e_j^2 in fp64, index order: the per-step error norm whose
    sum over iterations is the paper's total error."""
    lib = _load()
    e = np.ascontiguousarray(e, dtype=np.float32).reshape(-1)
    buf = e if e.size else np.zeros(1, np.float32)
    return float(lib.oracle_error_norm_sq(_ptr(buf, ctypes.c_float), e.size))


def sparse_aggregate(idx_list, val_list, d: int) -> np.ndarray:
    """Worker-ordered fp32 sum of n sparse vectors into a dense float32[d]."""
    lib = _load()
    n = len(idx_list)
    assert n == len(val_list) and n >= 1
    idx_arrs = [np.ascontiguousarray(x, dtype=np.uint32) for x in idx_list]
    val_arrs = [np.ascontiguousarray(v, dtype=np.float32) for v in val_list]
    # keep zero-length lists addressable
    idx_arrs = [a if a.size else np.zeros(1, np.uint32) for a in idx_arrs]
    val_arrs = [v if v.size else np.zeros(1, np.float32) for v in val_arrs]
    counts = np.array([len(x) for x in idx_list], dtype=np.uint32)
    for i in range(n):
        assert len(val_list[i]) == counts[i]
    u32p = ctypes.POINTER(ctypes.c_uint32)
    f32p = ctypes.POINTER(ctypes.c_float)
    idx_ptrs = (u32p * n)(*[_ptr(a, ctypes.c_uint32) for a in idx_arrs])
    val_ptrs = (f32p * n)(*[_ptr(v, ctypes.c_float) for v in val_arrs])
    dense = np.empty(max(d, 1), np.float32)
    rc = lib.oracle_sparse_aggregate(n, idx_ptrs, val_ptrs, _ptr(counts, ctypes.c_uint32), d,
                                     _ptr(dense, ctypes.c_float))
    if rc != 0:
        raise RuntimeError("oracle_sparse_aggregate: index out of range")
    return dense[:d].copy()
