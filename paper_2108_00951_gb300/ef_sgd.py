"""Distributed EF-SGD on l2-regularised logistic regression, through the library.

The paper's convex experiments (Appendix, logistic regression) minimise

    f(x) = (1/N) sum_i log(1 + exp(-y_i A[i,:] x)) + (mu/2) ||x||^2        (eq. 7)

with mu = 1e-4 * lambda_max(A^T A) / (4N), smoothness L = mu + lambda_max(A^T A) / (4N),
step size gamma = 1/L, the rows split over n workers, and a local batch of one
row drawn uniformly at every step. Every step of Algorithm 1 after the local
gradient runs in the library's kernels:

    p_i = e_i + gamma g_i, Delta_i = C(p_i), e_i <- p_i - Delta_i    ef_hard_threshold_ex / ef_topk_ex
    x <- x - (1/n) sum_i Delta_i                                    sparse_aggregate_apply

and each step reports the workers' squared error norms sum_i ||e_i||^2 (the
total error is their sum over the steps) and the elements sent.

The paper uses the LIBSVM datasets madelon and gisette, which are not
available here: `make_problem` draws a seeded synthetic classification set of
the same shape instead (madelon: N = 2000, d = 500; gisette: N = 6000,
d = 5000): Gaussian features around a common positive mean, as madelon's raw
features are (its rows are nearly parallel, so one row's smoothness is close
to L and a batch-of-one step of 1/L is stable: here within a factor 1.5),
labels from a random hyperplane through the mean with flipped signs for 10 %
of the rows. The local gradient
(a dot product and an axpy per worker, the input of the compression step) and
the function value used for reporting are computed with torch; the optimum f*
by accelerated full-batch gradient descent in fp64.

Hard-threshold parameter. The paper's tuning sets d gamma^2 lambda^2 = epsilon
for Delta = gamma C(p / gamma); the library thresholds p itself, so its lambda
is gamma times the paper's and the same rule reads d lambda_lib^2 = epsilon.
`match_volume` instead picks lambda so that hard-threshold sends the same
number of elements as Top-k over the run (the paper's matched-data-volume
comparison, e.g. k = 1 against a lambda with the same volume on madelon).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List

import torch

from . import _binding as efs


@dataclasses.dataclass
class Problem:
    A: torch.Tensor        # N x d, float32, on the device
    y: torch.Tensor        # N, float32 in {-1, +1}
    mu: float
    L: float
    gamma: float
    f_star: float
    name: str

    @property
    def N(self) -> int:
        return self.A.shape[0]

    @property
    def d(self) -> int:
        return self.A.shape[1]


def make_problem(name: str = "madelon", seed: int = 2108, device="cuda") -> Problem:
    """Seeded synthetic stand-in for a LIBSVM set of the paper's convex runs."""
    N, d = {"madelon": (2000, 500), "gisette": (6000, 5000), "tiny": (256, 64)}[name]
    gen = torch.Generator(device="cpu").manual_seed(seed)
    A = 1.0 + 0.5 * torch.randn(N, d, generator=gen, dtype=torch.float64)
    w_true = torch.randn(d, generator=gen, dtype=torch.float64)
    y = torch.sign((A - 1.0) @ w_true)
    y[y == 0] = 1.0
    flip = torch.rand(N, generator=gen, dtype=torch.float64) < 0.1
    y[flip] = -y[flip]
    lam_max = float(torch.linalg.eigvalsh(A.T @ A)[-1])
    base = lam_max / (4.0 * N)
    mu = 1e-4 * base
    L = mu + base
    prob = Problem(A=A.to(torch.float32).to(device), y=y.to(torch.float32).to(device), mu=mu, L=L,
                   gamma=1.0 / L, f_star=float("nan"), name=name)
    prob.f_star = _optimum(A.to(device), y.to(device), mu, L)
    return prob


def loss(A: torch.Tensor, y: torch.Tensor, mu: float, x: torch.Tensor) -> float:
    """f(x) of eq. 7 in fp64."""
    A, y, x = A.double(), y.double(), x.double()
    z = -y * (A @ x)
    return float(torch.nn.functional.softplus(z).mean() + 0.5 * mu * (x @ x))


def _optimum(A: torch.Tensor, y: torch.Tensor, mu: float, L: float, iters: int = 20000) -> float:
    # f is mu-strongly convex and L-smooth: gradient descent with step 1/L
    # contracts by (1 - mu/L) per step; Nesterov's accelerated variant
    # reaches machine precision within these iterations
    x = torch.zeros(A.shape[1], dtype=torch.float64, device=A.device)
    v = x.clone()
    q = mu / L
    beta = (1 - math.sqrt(q)) / (1 + math.sqrt(q))
    for _ in range(iters):
        z = -y * (A @ v)
        grad = -(A.T @ (y * torch.sigmoid(z))) / A.shape[0] + mu * v
        x_new = v - grad / L
        v = x_new + beta * (x_new - x)
        x = x_new
    return loss(A, y, mu, x)


def local_gradients(prob: Problem, x: torch.Tensor, rows: torch.Tensor) -> torch.Tensor:
    """Stochastic gradients of eq. 7, one row (batch size 1) per worker: row w
    of the result is -y_r sigmoid(-y_r A[r,:] x) A[r,:] + mu x for r = rows[w],
    fp32."""
    a = prob.A[rows]
    yr = prob.y[rows]
    s = torch.sigmoid(-yr * (a @ x))
    return (-(yr * s))[:, None] * a + prob.mu * x[None, :]


def run(prob: Problem, n: int, T: int, compressor: str, param: float, seed: int = 7,
        record_every: int = 1) -> Dict[str, List[float]]:
    """T steps of distributed EF-SGD with n workers. compressor: "ht" (param =
    the library's lambda) or "topk" (param = k). Records, every record_every
    steps, f(x_t) - f*, the workers' summed squared error norms of that step,
    and the elements sent so far; also the total error sum_t sum_i ||e_i||^2."""
    dev = prob.A.device
    d = prob.d
    gen = torch.Generator(device="cpu").manual_seed(seed)
    lo = torch.tensor([w * prob.N // n for w in range(n)])
    size = torch.tensor([(w + 1) * prob.N // n - w * prob.N // n for w in range(n)])
    x = torch.zeros(d, device=dev)
    e = torch.zeros(n, d, device=dev)
    idx = [torch.empty(d, dtype=torch.int32, device=dev) for _ in range(n)]
    val = [torch.empty(d, dtype=torch.float32, device=dev) for _ in range(n)]
    counts = torch.empty(n, dtype=torch.int32, device=dev)
    err = torch.empty(n, dtype=torch.float64, device=dev)
    sent = torch.zeros((), dtype=torch.float64, device=dev)
    total_error = torch.zeros((), dtype=torch.float64, device=dev)
    k = int(param)
    hist: Dict[str, List[float]] = {"t": [], "subopt": [], "err_sq": [], "sent": []}
    for t in range(T):
        rows = (lo + (torch.rand(n, generator=gen) * size).long().clamp_max(size - 1)).to(dev)
        g = local_gradients(prob, x, rows)
        for w in range(n):
            if compressor == "ht":
                efs.ef_hard_threshold(g[w], e[w], prob.gamma, param, idx[w], val[w],
                                      counts[w:w + 1], err_sq_out=err[w:w + 1])
            else:
                efs.ef_topk(g[w], e[w], prob.gamma, k, idx[w], val[w], counts[w:w + 1],
                            err_sq_out=err[w:w + 1])
        efs.sparse_aggregate_apply(idx, val, counts, d, 1.0 / n, x)
        sent += counts.sum()
        total_error += err.sum()
        if (t + 1) % record_every == 0 or t == T - 1:
            hist["t"].append(t + 1)
            hist["subopt"].append(loss(prob.A, prob.y, prob.mu, x) - prob.f_star)
            hist["err_sq"].append(float(err.sum()))
            hist["sent"].append(float(sent))
    if efs.ef_check_status() != efs.EF_OK:
        raise RuntimeError("device error during EF-SGD")
    hist["total_error"] = [float(total_error)]
    return hist


def match_volume(prob: Problem, n: int, T: int, target_sent: float, seed: int = 7,
                 iters: int = 20) -> float:
    """The library lambda with which hard-threshold sends about target_sent
    elements over T steps (bisection on log lambda; the volume falls as
    lambda grows)."""
    lo, hi = 1e-8, 1e2
    for _ in range(iters):
        mid = math.sqrt(lo * hi)
        sent = run(prob, n, T, "ht", mid, seed, record_every=T)["sent"][-1]
        if sent > target_sent:
            lo = mid
        else:
            hi = mid
    return math.sqrt(lo * hi)


def compare(name: str = "madelon", n: int = 20, T: int = 2000, k: int = 1, seed: int = 7,
            device="cuda") -> Dict[str, object]:
    """Top-k (k per worker) against hard-threshold at the same data volume."""
    prob = make_problem(name, device=device)
    sgd = run(prob, n, T, "topk", prob.d, seed)  # k = d: no compression
    topk = run(prob, n, T, "topk", k, seed)
    lam = match_volume(prob, n, T, topk["sent"][-1], seed)
    ht = run(prob, n, T, "ht", lam, seed)
    return {"problem": {"name": name, "N": prob.N, "d": prob.d, "mu": prob.mu, "L": prob.L,
                        "gamma": prob.gamma, "f_star": prob.f_star},
            "n": n, "T": T, "k": k, "lambda": lam, "sgd": sgd, "topk": topk, "ht": ht}


if __name__ == "__main__":
    import argparse
    import json
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--problem", default="madelon")
    ap.add_argument("--workers", type=int, default=20)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--k", type=int, default=1)
    args = ap.parse_args()
    out = compare(args.problem, args.workers, args.steps, args.k)
    summary = {key: out[key] for key in ("problem", "n", "T", "k", "lambda")}
    for c in ("sgd", "topk", "ht"):
        h = out[c]
        summary[c] = {"final_subopt": h["subopt"][-1], "elements_sent": h["sent"][-1],
                      "total_error": h["total_error"][0],
                      "subopt_at": {str(t): s for t, s in zip(h["t"], h["subopt"])
                                    if t in (1, 10, 100, 1000, h["t"][-1])}}
    print(json.dumps(summary))
