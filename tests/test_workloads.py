"""Synthetic workloads: layouts match the paper's parameter counts; the
tuning rule reproduces the thresholds the paper prints; draws are seeded."""
import os

import numpy as np
import torch

from paper_2108_00951_gb300 import workloads

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "tuning_lambdas.txt")


def test_parameter_counts_match_table_1():
    # Table 1: ResNet-18 11,173,962; LSTM 28,949,319
    assert sum(workloads.resnet18_cifar_segments()) == 11_173_962
    assert sum(workloads.lstm_wikitext2_segments()) == 28_949_319
    assert len(workloads.resnet18_cifar_segments()) == 62
    assert len(workloads.lstm_wikitext2_segments()) == 14
    assert sum(workloads.resnet50_imagenet_segments()) == 25_557_032
    assert len(workloads.resnet50_imagenet_segments()) == 161
    assert sum(workloads.vgg16_imagenet_segments()) == 138_357_544
    assert len(workloads.vgg16_imagenet_segments()) == 32


def test_tuning_rule_reproduces_printed_thresholds():
    rows = [l.split() for l in open(GOLDEN) if l.strip() and not l.startswith("#")]
    assert rows
    for name, d, printed in rows:
        k_min = int(0.001 * int(d))
        lam = workloads.threshold_for_k(k_min)
        assert round(lam, 5) == float(printed), (name, lam, printed)


def test_gradients_are_seeded_and_distinct():
    w = workloads.BY_NAME["lr"]
    a = workloads.gradient(w, 0, 0)
    b = workloads.gradient(w, 0, 0)
    c = workloads.gradient(w, 1, 0)
    d = workloads.gradient(w, 0, 1)
    assert torch.equal(a, b)
    assert not torch.equal(a, c) and not torch.equal(a, d)
    assert abs(float(a.std()) - 0.01) < 5e-4


def test_density_lambda_hits_target():
    w = workloads.BY_NAME["lr"]
    g = workloads.gradient(w, 0, 0)
    lam = workloads.density_lambda(w, g, 0.01)
    a = (np.float32(w.gamma) * g.numpy()).astype(np.float32)
    assert int(np.sum(np.abs(a) >= lam)) == 1000


def test_bf16_variant_is_rne_rounding():
    w = workloads.BY_NAME["lr"]
    g32 = workloads.gradient(w, 2, 3)
    g16 = workloads.gradient(w, 2, 3, dtype=torch.bfloat16)
    assert torch.equal(g16, g32.to(torch.bfloat16))
