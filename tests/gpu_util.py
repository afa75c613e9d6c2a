"""Helpers for the GPU parity tests: move numpy inputs to the device (optionally
at a misaligned base address), call the library through its binding, bring
results back as numpy, compare bit patterns."""
import numpy as np
import torch

import paper_2108_00951_gb300 as efs

DEV = torch.device("cuda:0") if torch.cuda.is_available() else None


def to_dev(x: np.ndarray, offset: int = 0) -> torch.Tensor:
    """Device copy of x whose base address is `offset` elements past an
    allocation boundary (offset 0: 256-byte aligned)."""
    t = torch.from_numpy(np.ascontiguousarray(x))
    buf = torch.empty(t.numel() + offset, dtype=t.dtype, device=DEV)
    view = buf[offset:offset + t.numel()]
    view.copy_(t)
    return view


def bits(x) -> np.ndarray:
    x = np.asarray(x)
    if x.dtype == np.float32:
        return x.view(np.uint32)
    return x


def assert_bits(a, b, what=""):
    """Bit-exact comparison; for float32 a NaN equals any NaN (the oracle's
    reading: a NaN carries no value, so its encoding is not part of the
    result)."""
    a, b = np.asarray(a), np.asarray(b)
    both_nan = (np.isnan(a) & np.isnan(b)) if a.dtype == np.float32 and b.dtype == np.float32 \
        and a.shape == b.shape else None
    a, b = bits(a), bits(b)
    assert a.shape == b.shape, (what, a.shape, b.shape)
    differ = a != b
    if both_nan is not None:
        differ &= ~both_nan
    if differ.any():
        bad = np.nonzero(differ)[0]
        raise AssertionError("%s: %d mismatches, first at %d: %r vs %r"
                             % (what, bad.size, bad[0], a[bad[0]], b[bad[0]]))


def g_device(g: np.ndarray, offset=0) -> torch.Tensor:
    if g.dtype == np.uint16:   # bf16 bit patterns
        t = to_dev(g.view(np.int16), offset)
        return t.view(torch.bfloat16)
    return to_dev(g, offset)


def ht(g, e, gamma, lam, g_off=0, e_off=0, stream=None, out_off=(0, 0)):
    d = e.size
    gd, ed = g_device(g, g_off), to_dev(e, e_off)
    # outputs `out_off` elements past an allocation boundary
    idx = torch.full((max(d, 1) + out_off[0],), -1, dtype=torch.int32, device=DEV)[out_off[0]:]
    val = torch.empty(max(d, 1) + out_off[1], dtype=torch.float32, device=DEV)[out_off[1]:]
    cnt = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    efs.ef_hard_threshold(gd, ed, gamma, lam, idx, val, cnt, stream=stream)
    torch.cuda.synchronize()
    c = int(cnt.item())
    return idx[:c].cpu().numpy().view(np.uint32), val[:c].cpu().numpy(), ed.cpu().numpy()


def topk(g, e, gamma, k, g_off=0, e_off=0):
    d = e.size
    gd, ed = g_device(g, g_off), to_dev(e, e_off)
    idx = torch.full((max(k, 1),), -1, dtype=torch.int32, device=DEV)
    val = torch.empty(max(k, 1), dtype=torch.float32, device=DEV)
    cnt = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    efs.ef_topk(gd, ed, gamma, k, idx, val, cnt)
    torch.cuda.synchronize()
    c = int(cnt.item())
    return idx[:c].cpu().numpy().view(np.uint32), val[:c].cpu().numpy(), ed.cpu().numpy()


def topk_layerwise(g, e, gamma, seg_end, seg_k, g_off=0, e_off=0):
    gd, ed = g_device(g, g_off), to_dev(e, e_off)
    total = int(np.sum(np.asarray(seg_k, dtype=np.uint64)))
    idx = torch.full((max(total, 1),), -1, dtype=torch.int32, device=DEV)
    val = torch.empty(max(total, 1), dtype=torch.float32, device=DEV)
    cnt = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    efs.ef_topk_layerwise(gd, ed, gamma, seg_end, seg_k, idx, val, cnt)
    torch.cuda.synchronize()
    c = int(cnt.item())
    return idx[:c].cpu().numpy().view(np.uint32), val[:c].cpu().numpy(), ed.cpu().numpy()


def aggregate(idx_list, val_list, d, dense_off=0):
    idx_t = [to_dev(np.asarray(i, np.uint32).view(np.int32)) if len(i) else
             torch.zeros(1, dtype=torch.int32, device=DEV) for i in idx_list]
    val_t = [to_dev(np.asarray(v, np.float32)) if len(v) else
             torch.zeros(1, dtype=torch.float32, device=DEV) for v in val_list]
    counts = torch.tensor([len(i) for i in idx_list], dtype=torch.int32, device=DEV)
    buf = torch.full((d + dense_off,), float("nan"), dtype=torch.float32, device=DEV)
    dense = buf[dense_off:]
    efs.sparse_aggregate(idx_t, val_t, counts, d, dense)
    torch.cuda.synchronize()
    return dense.cpu().numpy()
