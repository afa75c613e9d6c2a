"""ctypes binding of libefsparse.so — argument marshalling only.

Every function here has the name of the C entry point it calls (declared in
``include/efsparse.h``), takes torch CUDA tensors, checks their dtype, device,
shape and contiguity, and passes raw device pointers and the current CUDA
stream across the C ABI. All computation happens in the library's kernels;
there is no fallback: if the library cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np
import torch

from . import build as _build

EF_OK = 0
EF_ERR_INVALID_ARG = 1
EF_ERR_CUDA = 2
EF_ERR_TIMEOUT = 3
EF_ERR_BAD_INPUT = 4
EF_ERR_NO_MEMORY = 5


class EfError(RuntimeError):
    """A non-OK ef_status returned by the library."""

    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__("%s: %s" % (where, status_string(status)))


_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIBPATH


def load_library(build_if_missing: bool = True):
    """Load libefsparse.so (building it in-tree first if it is missing)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIBPATH
        if not os.path.exists(path) or not _build.up_to_date():
            if not build_if_missing:
                raise RuntimeError("libefsparse.so is not built: run __graft_entry__.build()")
            _build.build()
        lib = ctypes.CDLL(path)
        vp, u64, f32, u32 = ctypes.c_void_p, ctypes.c_uint64, ctypes.c_float, ctypes.c_uint32
        sig = {
            "ef_hard_threshold": [vp, vp, f32, f32, u64, vp, vp, vp, vp],
            "ef_hard_threshold_bf16": [vp, vp, f32, f32, u64, vp, vp, vp, vp],
            "ef_topk": [vp, vp, f32, u64, u64, vp, vp, vp, vp],
            "ef_topk_bf16": [vp, vp, f32, u64, u64, vp, vp, vp, vp],
            "ef_topk_layerwise": [vp, vp, f32, u32, vp, vp, u64, vp, vp, vp, vp],
            "ef_topk_layerwise_bf16": [vp, vp, f32, u32, vp, vp, u64, vp, vp, vp, vp],
            "ef_hard_threshold_ex": [vp, ctypes.c_int, vp, f32, f32, u64, vp, vp, vp, vp, vp],
            "ef_topk_ex": [vp, ctypes.c_int, vp, f32, u64, u64, vp, vp, vp, vp, vp],
            "ef_topk_layerwise_ex": [vp, ctypes.c_int, vp, f32, u32, vp, vp, u64, vp, vp, vp, vp,
                                     vp],
            "ef_scaled_round_ex": [vp, ctypes.c_int, vp, f32, ctypes.c_int32, u64, vp, vp, vp,
                                   vp],
            "int_aggregate": [u32, ctypes.POINTER(vp), u64, ctypes.c_int32, vp, vp],
            "sparse_aggregate": [u32, ctypes.POINTER(vp), ctypes.POINTER(vp), vp, u64, vp, vp],
            "sparse_aggregate_apply": [u32, ctypes.POINTER(vp), ctypes.POINTER(vp), vp, u64, f32,
                                       vp, vp, f32, f32, vp],
            "ef_hard_threshold_tiled": [vp, ctypes.c_int, vp, f32, f32, u64, vp, vp, vp, vp, vp,
                                        vp],
            "sparse_aggregate_tiled": [u32, ctypes.POINTER(vp), ctypes.POINTER(vp),
                                       ctypes.POINTER(vp), vp, u64, vp, vp],
            "sparse_aggregate_apply_tiled": [u32, ctypes.POINTER(vp), ctypes.POINTER(vp),
                                             ctypes.POINTER(vp), vp, u64, f32, vp, vp, f32, f32,
                                             vp],
            "ef_check_status": [vp],
            "ef_workspace_release": [],
        }
        for name, args in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        lib.ef_status_string.argtypes = [ctypes.c_int]
        lib.ef_status_string.restype = ctypes.c_char_p
        lib.ef_kernel_launches.argtypes = []
        lib.ef_kernel_launches.restype = ctypes.c_uint64
        lib.ef_test_set_lookback_fault.argtypes = [ctypes.c_int64, ctypes.c_uint32]
        lib.ef_test_set_lookback_fault.restype = None
        lib.ef_test_set_stream_kernel.argtypes = [ctypes.c_int]
        lib.ef_test_set_stream_kernel.restype = None
        _lib = lib
        return lib


def status_string(status: int) -> str:
    return load_library().ef_status_string(int(status)).decode()


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(status: int, where: str):
    if status != EF_OK:
        raise EfError(status, where)


def _dev(t: torch.Tensor, name: str, dtype, numel=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError("%s must be a CUDA tensor" % name)
    if t.dtype != dtype:
        raise TypeError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if numel is not None and t.numel() < numel:
        raise ValueError("%s holds %d elements, needs %d" % (name, t.numel(), numel))
    return ctypes.c_void_p(t.data_ptr() if t.numel() else 0)


def _gradient(g: torch.Tensor):
    if g.dtype == torch.float32:
        return False
    if g.dtype == torch.bfloat16:
        return True
    raise TypeError("g must be float32 or bfloat16")


def _err(err_sq_out):
    if err_sq_out is None:
        return ctypes.c_void_p(0)
    return _dev(err_sq_out, "err_sq_out", torch.float64, 1)


TILE = 4096  # coordinates per tile of a message's tile index


def tiles_for(d: int) -> int:
    """Length of a message's tile index for dimension d: ceil(d / TILE) + 1."""
    return (int(d) + TILE - 1) // TILE + 1


def ef_hard_threshold(g, e, gamma, lam, idx_out, val_out, count_out, stream=None,
                      err_sq_out=None, tiles_out=None):
    """EF accumulate + hard-threshold + compaction (``ef_hard_threshold[_bf16]``;
    ``ef_hard_threshold_ex`` when ``err_sq_out`` is given,
    ``ef_hard_threshold_tiled`` when ``tiles_out`` is given).

    ``g`` float32 or bfloat16 [d]; ``e`` float32 [d], updated in place;
    ``idx_out`` int32 [>= d] (uint32 bit patterns), ``val_out`` float32 [>= d],
    ``count_out`` int32 [>= 1]; ``err_sq_out`` optional float64 [>= 1]:
    ||e'||^2 of the step; ``tiles_out`` optional int32 [>= tiles_for(d)]: the
    message's tile index (pairs below each multiple of TILE, then the count).
    """
    lib = load_library()
    bf16 = _gradient(g)
    d = e.numel()
    if g.numel() != d:
        raise ValueError("g and e differ in length")
    head = (_dev(g, "g", g.dtype), _dev(e, "e", torch.float32), ctypes.c_float(gamma),
            ctypes.c_float(lam), d, _dev(idx_out, "idx_out", torch.int32, d),
            _dev(val_out, "val_out", torch.float32, d),
            _dev(count_out, "count_out", torch.int32, 1))
    if tiles_out is not None:
        _check(lib.ef_hard_threshold_tiled(
            head[0], int(bf16), *head[1:], _dev(tiles_out, "tiles_out", torch.int32, tiles_for(d)),
            ctypes.c_void_p(0) if err_sq_out is None else _err(err_sq_out), _stream(stream)),
            "ef_hard_threshold_tiled")
        return
    if err_sq_out is not None:
        _check(lib.ef_hard_threshold_ex(head[0], int(bf16), *head[1:], _err(err_sq_out),
                                        _stream(stream)), "ef_hard_threshold_ex")
        return
    fn = lib.ef_hard_threshold_bf16 if bf16 else lib.ef_hard_threshold
    _check(fn(*head, _stream(stream)), "ef_hard_threshold")


def ef_topk(g, e, gamma, k, idx_out, val_out, count_out, stream=None, err_sq_out=None):
    """EF accumulate + Top-k + compaction (``ef_topk[_bf16]``, ``ef_topk_ex`` with
    ``err_sq_out``); exactly k pairs."""
    lib = load_library()
    bf16 = _gradient(g)
    d = e.numel()
    if g.numel() != d:
        raise ValueError("g and e differ in length")
    head = (_dev(g, "g", g.dtype), _dev(e, "e", torch.float32), ctypes.c_float(gamma), int(k),
            d, _dev(idx_out, "idx_out", torch.int32, k),
            _dev(val_out, "val_out", torch.float32, k),
            _dev(count_out, "count_out", torch.int32, 1))
    if err_sq_out is not None:
        _check(lib.ef_topk_ex(head[0], int(bf16), *head[1:], _err(err_sq_out), _stream(stream)),
               "ef_topk_ex")
        return
    fn = lib.ef_topk_bf16 if bf16 else lib.ef_topk
    _check(fn(*head, _stream(stream)), "ef_topk")


def ef_topk_layerwise(g, e, gamma, seg_end, seg_k, idx_out, val_out, count_out, stream=None,
                      err_sq_out=None):
    """EF accumulate + layer-wise Top-k + compaction (``ef_topk_layerwise[_bf16]``).

    ``seg_end``/``seg_k``: sequences of n_seg integers (host side): segment s
    is ``[seg_end[s-1], seg_end[s])`` and sends its ``seg_k[s]`` largest
    coordinates; exactly ``sum(seg_k)`` pairs are written.
    """
    lib = load_library()
    bf16 = _gradient(g)
    d = e.numel()
    if g.numel() != d:
        raise ValueError("g and e differ in length")
    ends = np.ascontiguousarray(seg_end, dtype=np.uint64)
    ks = np.ascontiguousarray(seg_k, dtype=np.uint64)
    if ends.ndim != 1 or ks.shape != ends.shape:
        raise ValueError("seg_end and seg_k must be 1-D of one length")
    total = int(ks.sum()) if ks.size else 0
    head = (_dev(g, "g", g.dtype), _dev(e, "e", torch.float32), ctypes.c_float(gamma),
            ctypes.c_uint32(ends.size), ctypes.c_void_p(ends.ctypes.data),
            ctypes.c_void_p(ks.ctypes.data), d, _dev(idx_out, "idx_out", torch.int32, total),
            _dev(val_out, "val_out", torch.float32, total),
            _dev(count_out, "count_out", torch.int32, 1))
    if err_sq_out is not None:
        _check(lib.ef_topk_layerwise_ex(head[0], int(bf16), *head[1:], _err(err_sq_out),
                                        _stream(stream)), "ef_topk_layerwise_ex")
        return
    fn = lib.ef_topk_layerwise_bf16 if bf16 else lib.ef_topk_layerwise
    _check(fn(*head, _stream(stream)), "ef_topk_layerwise")


def _tile_array(tiles, n, d):
    if len(tiles) != n:
        raise ValueError("one tile index per list")
    return (ctypes.c_void_p * max(n, 1))(*[_dev(t, "tiles", torch.int32, tiles_for(d))
                                           for t in tiles])


def sparse_aggregate(idx_list, val_list, counts, d, dense_out, stream=None, tiles=None):
    """Worker-ordered sum of n sparse vectors into ``dense_out`` (float32 [d]).

    ``idx_list``/``val_list``: n int32 / float32 CUDA tensors; ``counts``: int32
    CUDA tensor of n pair counts; ``tiles`` optional: the n lists' tile indexes
    (``sparse_aggregate_tiled``).
    """
    lib = load_library()
    n = len(idx_list)
    if n != len(val_list):
        raise ValueError("idx_list and val_list differ in length")
    idx_arr = (ctypes.c_void_p * max(n, 1))(*[_dev(t, "idx", torch.int32) for t in idx_list])
    val_arr = (ctypes.c_void_p * max(n, 1))(*[_dev(t, "val", torch.float32) for t in val_list])
    cnt = _dev(counts, "counts", torch.int32, n)
    out = _dev(dense_out, "dense_out", torch.float32, d)
    if tiles is not None:
        _check(lib.sparse_aggregate_tiled(n, idx_arr, val_arr, _tile_array(tiles, n, d), cnt,
                                          int(d), out, _stream(stream)), "sparse_aggregate_tiled")
        return
    _check(lib.sparse_aggregate(n, idx_arr, val_arr, cnt, int(d), out, _stream(stream)),
           "sparse_aggregate")


def sparse_aggregate_apply(idx_list, val_list, counts, d, alpha, x, m=None, momentum=0.0, lr=0.0,
                           stream=None, tiles=None):
    """Worker-ordered sum of n sparse vectors, scaled by ``alpha``, applied to
    the model ``x`` (float32 [d], in place): ``x -= Delta'`` without ``m``;
    with ``m`` (float32 [d], in place) ``m = fmaf(momentum, m, Delta')`` and
    ``x = fmaf(-lr, Delta' + m, x)``. ``tiles`` optional: the lists' tile
    indexes (``sparse_aggregate_apply_tiled``)."""
    lib = load_library()
    n = len(idx_list)
    if n != len(val_list):
        raise ValueError("idx_list and val_list differ in length")
    idx_arr = (ctypes.c_void_p * max(n, 1))(*[_dev(t, "idx", torch.int32) for t in idx_list])
    val_arr = (ctypes.c_void_p * max(n, 1))(*[_dev(t, "val", torch.float32) for t in val_list])
    m_ptr = ctypes.c_void_p(0) if m is None else _dev(m, "m", torch.float32, d)
    tail = (_dev(counts, "counts", torch.int32, n), int(d), ctypes.c_float(alpha),
            _dev(x, "x", torch.float32, d), m_ptr, ctypes.c_float(momentum), ctypes.c_float(lr),
            _stream(stream))
    if tiles is not None:
        _check(lib.sparse_aggregate_apply_tiled(n, idx_arr, val_arr, _tile_array(tiles, n, d),
                                                *tail), "sparse_aggregate_apply_tiled")
        return
    _check(lib.sparse_aggregate_apply(n, idx_arr, val_arr, *tail), "sparse_aggregate_apply")


def ef_scaled_round(g, e, gamma, scale_log2, q_out, unsent_out, stream=None, err_sq_out=None):
    """EF accumulate + scaled integer rounding (``ef_scaled_round_ex``):
    ``q_out`` int32 [d] = RNE(a 2^scale_log2), ``e`` becomes a - q 2^-scale_log2;
    ``unsent_out`` int32 [>= 1] counts the coordinates that did not fit."""
    lib = load_library()
    bf16 = _gradient(g)
    d = e.numel()
    if g.numel() != d:
        raise ValueError("g and e differ in length")
    _check(lib.ef_scaled_round_ex(_dev(g, "g", g.dtype), int(bf16), _dev(e, "e", torch.float32),
                                  ctypes.c_float(gamma), int(scale_log2), d,
                                  _dev(q_out, "q_out", torch.int32, d),
                                  _dev(unsent_out, "unsent_out", torch.int32, 1),
                                  _err(err_sq_out), _stream(stream)), "ef_scaled_round_ex")


def int_aggregate(q_list, d, scale_log2, dense_out, stream=None):
    """Exact integer sum of n dense int32 messages, as RN(S) 2^-scale_log2."""
    lib = load_library()
    n = len(q_list)
    arr = (ctypes.c_void_p * max(n, 1))(*[_dev(t, "q", torch.int32, d) for t in q_list])
    _check(lib.int_aggregate(n, arr, int(d), int(scale_log2),
                             _dev(dense_out, "dense_out", torch.float32, d), _stream(stream)),
           "int_aggregate")


def ef_check_status(stream=None) -> int:
    """Synchronise the stream; return (and clear) the latched device status."""
    return int(load_library().ef_check_status(_stream(stream)))


def ef_workspace_release():
    _check(load_library().ef_workspace_release(), "ef_workspace_release")


def ef_kernel_launches() -> int:
    return int(load_library().ef_kernel_launches())


def ef_test_set_lookback_fault(withheld_tile: int, spin_limit_us: int = 0):
    load_library().ef_test_set_lookback_fault(int(withheld_tile), int(spin_limit_us))


def ef_test_set_stream_kernel(mode: int):
    load_library().ef_test_set_stream_kernel(int(mode))
