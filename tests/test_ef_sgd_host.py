"""Host-side checks of the logistic-regression EF-SGD driver (no GPU): the
problem constants follow the paper's definitions (eq. 7 and the text after
it), the local gradient is the gradient of one row's loss, and f* is the
minimum."""
import math

import numpy as np
import pytest
import torch

from paper_2108_00951_gb300 import ef_sgd


@pytest.fixture(scope="module")
def tiny():
    return ef_sgd.make_problem("tiny", device="cpu")


def test_constants_follow_the_paper(tiny):
    A = tiny.A.double().numpy()
    lam_max = np.linalg.eigvalsh(A.T @ A)[-1]
    base = lam_max / (4 * tiny.N)
    assert math.isclose(tiny.mu, 1e-4 * base, rel_tol=1e-5)
    assert math.isclose(tiny.L, tiny.mu + base, rel_tol=1e-5)
    assert tiny.gamma == 1.0 / tiny.L
    assert set(np.unique(tiny.y.numpy())) <= {-1.0, 1.0}


def test_local_gradient_is_the_row_loss_gradient(tiny):
    rng = np.random.default_rng(3)
    x = torch.tensor(rng.standard_normal(tiny.d) * 0.1, dtype=torch.float32)
    rows = torch.tensor([0, 17, 255])
    g = ef_sgd.local_gradients(tiny, x, rows)
    for w, r in enumerate(rows.tolist()):
        xr = x.double().clone().requires_grad_(True)
        a, y = tiny.A[r].double(), tiny.y[r].double()
        f = torch.nn.functional.softplus(-y * (a @ xr)) + 0.5 * tiny.mu * (xr @ xr)
        f.backward()
        assert torch.allclose(g[w].double(), xr.grad, rtol=1e-5, atol=1e-7)


def test_f_star_is_the_minimum(tiny):
    # f is convex: no point, including the origin and random points, is
    # below f*, and the optimum's gradient vanishes to fp64 precision
    assert tiny.f_star <= ef_sgd.loss(tiny.A, tiny.y, tiny.mu, torch.zeros(tiny.d))
    rng = np.random.default_rng(4)
    for _ in range(5):
        x = torch.tensor(rng.standard_normal(tiny.d) * 0.05)
        assert tiny.f_star <= ef_sgd.loss(tiny.A, tiny.y, tiny.mu, x) + 1e-12
    assert tiny.f_star < math.log(2.0)
