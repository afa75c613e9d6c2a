"""Seeded synthetic workloads shaped like the paper's benchmarks.

The paper's gradients come from training ResNet-18 / LSTM / NCF (Table 1) and
logistic regression on LIBSVM data (Sec. 6, Appendix logistic-regression
experiments); none of those datasets or models is available here, so each
workload is a seeded synthetic stand-in with the model's exact parameter
count and layer (segment) layout and a heavy- or light-tailed per-segment
gradient distribution. This module only draws inputs: it contains none of the
error-feedback arithmetic. Both the CUDA path and the CPU oracle consume the
tensors it returns (generated once, copied to the other side).

Configurations (index = position in the workload list):
  0 "lr"        d = 100,000 (logistic-regression sized), n = 4, T = 10
  1 "resnet18"  d = 11,173,962 in 62 tensors (ResNet-18 / CIFAR-10, Table 1)
  2 "lstm"      d = 28,949,319 in 14 tensors (LSTM / WikiText-2, Table 1)
  3 "resnet50"  d = 25,557,032 in 161 tensors (ResNet-50 / ImageNet)
  4 "vgg16"     d = 138,357,544 in 32 tensors (VGG-16 / ImageNet)
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional

import torch


# ----------------------------------------------------------------- layouts
def resnet18_cifar_segments() -> List[int]:
    """Parameter tensors of ResNet-18 for CIFAR-10 in definition order
    (3x3 stem, four stages of two BasicBlocks, widths 64..512, 10-way FC)."""
    s = [3 * 3 * 3 * 64, 64, 64]
    cin = 64
    for width, stride in ((64, 1), (128, 2), (256, 2), (512, 2)):
        for b in range(2):
            i = cin if b == 0 else width
            s += [i * width * 9, width, width, width * width * 9, width, width]
            if b == 0 and (stride != 1 or i != width):
                s += [i * width, width, width]     # 1x1 projection shortcut + BN
        cin = width
    return s + [512 * 10, 10]


def lstm_wikitext2_segments() -> List[int]:
    """A 3-layer, 650-wide LSTM language model with a tied 28,869-word
    embedding/decoder: 14 tensors summing to the paper's 28,949,319."""
    s = [28869 * 650]
    for _ in range(3):
        s += [2600 * 650, 2600 * 650, 2600, 2600]  # W_ih, W_hh, b_ih, b_hh
    return s + [28869]                            # decoder bias


def resnet50_imagenet_segments() -> List[int]:
    """Parameter tensors of ResNet-50 (bottleneck stages [3, 4, 6, 3],
    expansion 4, 1000-way FC)."""
    s = [7 * 7 * 3 * 64, 64, 64]
    cin = 64
    for width, blocks in ((64, 3), (128, 4), (256, 6), (512, 3)):
        for b in range(blocks):
            i = cin if b == 0 else 4 * width
            s += [i * width, width, width, width * width * 9, width, width,
                  width * 4 * width, 4 * width, 4 * width]
            if b == 0:
                s += [i * 4 * width, 4 * width, 4 * width]
        cin = 4 * width
    return s + [2048 * 1000, 1000]


def vgg16_imagenet_segments() -> List[int]:
    """Parameter tensors of VGG-16 (13 convolutions with biases, 3 FC layers)."""
    s = []
    cin = 3
    for w in (64, 64, 128, 128, 256, 256, 256, 512, 512, 512, 512, 512, 512):
        s += [cin * w * 9, w]
        cin = w
    return s + [25088 * 4096, 4096, 4096 * 4096, 4096, 4096 * 1000, 1000]


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    d: int
    segments: tuple
    n: int              # simulated workers
    T: int              # EF iterations
    gamma: float
    seed: int
    density: Optional[float] = None   # hard-threshold lambda targets this first-iteration density
    lambdas: tuple = ()               # fixed hard-threshold lambdas
    topk_fracs: tuple = ()            # Top-k k = floor(frac * d)
    topk_k: tuple = ()                # fixed Top-k k values

    def topk_values(self) -> List[int]:
        return list(self.topk_k) + [max(1, int(f * self.d)) for f in self.topk_fracs]


WORKLOADS = [
    Workload("lr", 100_000, (100_000,), n=4, T=10, gamma=0.1, seed=2109,
             lambdas=(2e-3,), topk_k=(1000,)),
    Workload("resnet18", 11_173_962, tuple(resnet18_cifar_segments()), n=8, T=50, gamma=0.1,
             seed=2110, density=1e-3, topk_fracs=(1e-3,)),
    Workload("lstm", 28_949_319, tuple(lstm_wikitext2_segments()), n=8, T=50, gamma=0.1,
             seed=2111, density=1e-2, topk_fracs=(1e-2,)),
    Workload("resnet50", 25_557_032, tuple(resnet50_imagenet_segments()), n=16, T=100,
             gamma=0.1, seed=2112, lambdas=(1e-4, 3e-4, 1e-3), topk_fracs=(1e-3, 1e-2)),
    Workload("vgg16", 138_357_544, tuple(vgg16_imagenet_segments()), n=8, T=20, gamma=0.1,
             seed=2113, density=1e-4, topk_fracs=(1e-4,)),
]
BY_NAME = {w.name: w for w in WORKLOADS}

for _w in WORKLOADS:
    assert sum(_w.segments) == _w.d, _w.name


# ------------------------------------------------------------- generation
def _seed(w: Workload, worker: int, iteration: int, stream: int = 0) -> int:
    return ((w.seed * 1_000_003 + worker) * 1_000_003 + iteration) * 7 + stream


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(seed % (2 ** 63))
    return g


def _segment_scales(w: Workload, lo: float, hi: float, log: bool, device) -> torch.Tensor:
    """One scale per segment, drawn once per workload from its seed, expanded
    to a per-coordinate tensor."""
    cg = torch.Generator().manual_seed(w.seed)
    u = torch.rand(len(w.segments), generator=cg, dtype=torch.float64)
    if log:
        s = torch.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))
    else:
        s = lo + u * (hi - lo)
    sizes = torch.tensor(w.segments, dtype=torch.int64)
    return torch.repeat_interleave(s.to(torch.float32), sizes).to(device)


def _laplace(d, gen, device):
    x = torch.empty(d, device=device, dtype=torch.float32).exponential_(generator=gen)
    sign = torch.rand(d, device=device, generator=gen) < 0.5
    return torch.where(sign, -x, x)


def gradient(w: Workload, worker: int, iteration: int, device="cpu",
             dtype=torch.float32) -> torch.Tensor:
    """Seeded synthetic gradient g_{worker, iteration} of workload w.

    dtype=torch.bfloat16 rounds the fp32 draw to bfloat16 (round to nearest
    even), the VGG-16 bf16-gradient variant.
    """
    d = w.d
    gen = _gen(device, _seed(w, worker, iteration))
    if w.name == "lr":
        g = torch.randn(d, device=device, generator=gen) * 0.01
    elif w.name == "resnet18":
        g = _laplace(d, gen, device) * _segment_scales(w, 1e-5, 1e-2, True, device)
    elif w.name == "lstm":
        emb = w.segments[0]
        rows = emb // 650
        z = torch.randn(d, device=device, generator=gen)
        chi = torch.randn(3, d, device=device, generator=gen).square().sum(0) / 3.0
        g = z / torch.sqrt(chi) * 1e-3                       # Student-t(3) * 1e-3
        zero_rows = torch.rand(rows, device=device, generator=gen) < 0.95
        g[:emb].view(rows, 650).masked_fill_(zero_rows[:, None], 0.0)
    elif w.name == "resnet50":
        s = _segment_scales(w, 1e-6, 1e-2, True, device)
        g = torch.randn(d, device=device, generator=gen) * s
        out = torch.rand(d, device=device, generator=gen) < 1e-4
        g = torch.where(out, torch.randn(d, device=device, generator=gen) * s * 100.0, g)
    elif w.name == "vgg16":
        g = _laplace(d, gen, device) * (1e-4 * _segment_scales(w, 0.5, 2.0, False, device))
    else:
        raise KeyError(w.name)
    g = g.to(torch.float32)
    return g.to(dtype) if dtype != torch.float32 else g


def segment_ends(w: Workload) -> List[int]:
    """Exclusive end of each parameter tensor in the flattened vector."""
    out, acc = [], 0
    for n in w.segments:
        acc += n
        out.append(acc)
    return out


def layerwise_k(w: Workload, frac: float) -> List[int]:
    """Per-tensor Top-k budgets k_s = max(1, floor(frac * d_s)) (0 for an
    empty tensor): the layer-wise compression of the paper's experiments
    keeps the same fraction of every layer."""
    return [max(1, int(frac * n)) if n > 0 else 0 for n in w.segments]


def density_lambda(w: Workload, g0: torch.Tensor, density: float) -> float:
    """lambda such that the first EF iteration (e = 0, so a = gamma g) sends
    about `density` of the coordinates: the ceil(density * d)-th largest
    |gamma g_j| of worker 0, in fp32."""
    m = max(1, math.ceil(density * w.d))
    mag = g0.float().abs()
    kth = torch.topk(mag, m).values[-1].to(torch.float32)
    return float(torch.tensor(w.gamma, dtype=torch.float32) * kth)


def threshold_for_k(k: int) -> float:
    """The paper's tuning rule for the hard-threshold that matches Top-k with
    parameter k in data volume: lambda = 1 / (2 sqrt(k)) (Sec. 6, "How to tune
    the hard-threshold?"; the appendix derivation assumes zeta = 0, sigma = 1/4)."""
    return 1.0 / (2.0 * math.sqrt(k))
