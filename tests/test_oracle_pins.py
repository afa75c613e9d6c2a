"""Pins of the CPU oracle to what the paper and the mathematics fix (no GPU).

Each test checks the oracle against something other than itself: exact
rational arithmetic, brute-force search over supports, closed-form special
cases, bounds stated in the paper, or a library routine. Together they are
chosen so that a dropped term, a wrong sign, a swapped operand, a '>' for
'>=', a wrong tie rule or a wrong summation order each fails at least one.
"""
from fractions import Fraction
import itertools
import math

import numpy as np
import pytest

import oracle
from exact_fp32 import fma_f32, round_f32, to_frac, ulp_f32

RNG = np.random.default_rng(2108)


def _f32(x):
    return np.asarray(x, dtype=np.float32)


def _exact_a(g, e, gamma):
    gamma = np.float32(gamma)           # the library takes gamma as fp32
    return np.array([fma_f32(gamma, gj, ej) for gj, ej in zip(g, e)], dtype=np.float32)


def _same_bits(x, y):
    x = np.asarray(x, np.float32)
    y = np.asarray(y, np.float32)
    return x.shape == y.shape and np.array_equal(x.view(np.uint32), y.view(np.uint32))


# --------------------------------------------------------------------------
# a = e + gamma g (Algorithm 1, first step), one correctly rounded fma
# --------------------------------------------------------------------------

def _fma_sensitive_triples(count):
    """Random (gamma, g, e) with wide exponents, plus cases where the product
    must not be rounded before the addition (fma != mul-then-add)."""
    gam = _f32(RNG.uniform(0.01, 2.0, count) * np.exp2(RNG.integers(-8, 4, count)))
    g = _f32(RNG.standard_normal(count) * np.exp2(RNG.integers(-20, 6, count)))
    e = _f32(RNG.standard_normal(count) * np.exp2(RNG.integers(-20, 6, count)))
    # cancellation cases: e = -round(gamma*g), so a is the product's rounding error
    c = count // 4
    e[:c] = -(gam[:c] * g[:c])
    return gam, g, e


def test_accumulate_is_one_rounded_fma():
    gam, g, e = _fma_sensitive_triples(4000)
    mismatched_two_step = 0
    for gm, gj, ej in zip(gam, g, e):
        a_exact = fma_f32(gm, gj, ej)
        two_step = np.float32(np.float32(gm) * np.float32(gj)) + np.float32(ej)
        if not _same_bits(two_step, a_exact):
            mismatched_two_step += 1
        # lambda = inf sends nothing finite, so e' = a exactly
        idx, val, e_new = oracle.ef_hard_threshold(_f32([gj]), _f32([ej]), float(gm), math.inf)
        assert idx.size == 0
        assert _same_bits(e_new, [a_exact]), (gm, gj, ej)
    # the set really distinguishes a fused from a two-step evaluation
    assert mismatched_two_step > 500


def test_accumulate_operand_roles():
    # a = e + gamma*g; swapping g and e, or the sign, gives a different value
    g, e, gamma = _f32([3.0]), _f32([5.0]), 0.5
    _, _, e_new = oracle.ef_hard_threshold(g, e, gamma, math.inf)
    assert e_new[0] == 5.0 + 0.5 * 3.0


# --------------------------------------------------------------------------
# hard-threshold S_lambda(a) = {j : |a_j| >= lambda} (Sec. 1, Sec. 4.2)
# --------------------------------------------------------------------------

def test_ht_threshold_is_inclusive():
    # |a| == lambda exactly must be sent (">=", Sec. 1); just below must not
    lam = 0.25
    below = np.nextafter(np.float32(lam), np.float32(0))
    e = _f32([lam, -lam, below, -below, 1.0])
    g = np.zeros(5, np.float32)
    idx, val, e_new = oracle.ef_hard_threshold(g, e, 1.0, lam)
    assert idx.tolist() == [0, 1, 4]
    assert val.tolist() == [lam, -lam, 1.0]
    assert _same_bits(e_new, [0.0, 0.0, below, -below, 0.0])


def test_ht_lambda_zero_sends_exactly_the_nonzeros():
    # special case lambda = 0: every non-zero coordinate is sent, e' = 0 there
    tiny = np.float32(np.finfo(np.float32).smallest_subnormal)
    e = _f32([0.0, -0.0, tiny, -tiny, 3.5, 0.0, -2.0])
    g = np.zeros_like(e)
    g[1] = -0.0            # (-0)*0.1 + (-0) = -0: a signed zero stays unsent
    idx, val, e_new = oracle.ef_hard_threshold(g, e, 0.1, 0.0)
    assert idx.tolist() == [2, 3, 4, 6]
    assert _same_bits(val, [tiny, -tiny, 3.5, -2.0])
    assert _same_bits(e_new, [0.0, -0.0, 0.0, 0.0, 0.0, 0.0, 0.0])


def test_ht_lambda_above_max_sends_nothing():
    g = _f32(RNG.standard_normal(1000))
    e = _f32(RNG.standard_normal(1000))
    a = _exact_a(g, e, 0.1)
    lam = float(np.nextafter(np.max(np.abs(a)), np.float32(np.inf)))
    idx, val, e_new = oracle.ef_hard_threshold(g, e, 0.1, lam)
    assert idx.size == 0
    assert _same_bits(e_new, a)


def test_ht_nan_and_inf():
    # NaN never passes |a| >= lambda; +-inf does; 0 * inf is NaN (invalid)
    e = _f32([np.nan, np.inf, -np.inf, 1.0, 5.0])
    g = _f32([0.0, 0.0, 0.0, 0.0, np.inf])
    idx, val, e_new = oracle.ef_hard_threshold(g, e, 1.0, 0.5)
    assert idx.tolist() == [1, 2, 3, 4]
    assert val.tolist() == [np.inf, -np.inf, 1.0, np.inf]
    assert e_new[1:].tolist() == [0.0, 0.0, 0.0, 0.0]
    # a NaN accumulator (a NaN error, or 0 * inf) is never sent and stays in
    # the residual as a NaN, whatever its encoding (reading R6)
    e = _f32([np.nan, 2.0, -1.0])
    e[0] = np.uint32(0xFFC00001).view(np.float32)        # a negative NaN with a payload
    idx, _, e_new = oracle.ef_hard_threshold(_f32([0.0, np.inf, 0.0]), e, 0.0, 0.5)
    assert idx.tolist() == [2]
    assert np.isnan(e_new[0]) and np.isnan(e_new[1]) and e_new[2] == 0.0


@pytest.mark.parametrize("d", [1, 7, 64, 3001])
def test_ht_reconstruction_and_absolute_bound(d):
    # a = C(a) + e' exactly (Algorithm 1 error update) and ||e'||_inf < lambda,
    # hence ||e'||^2 <= d lambda^2 (absolute compressor, kappa^2 = d lambda^2)
    g = _f32(RNG.standard_normal(d) * 0.01)
    e = _f32(RNG.standard_normal(d) * 0.001)
    gamma, lam = 0.1, 1.5e-3
    a = _exact_a(g, e, gamma)
    idx, val, e_new = oracle.ef_hard_threshold(g, e, gamma, lam)
    assert np.all(np.diff(idx.astype(np.int64)) > 0)
    dense = np.zeros(d, np.float32)
    dense[idx] = val
    assert _same_bits(dense + e_new, a)
    assert np.all(np.abs(e_new) < lam)
    assert float(np.sum(e_new.astype(np.float64) ** 2)) <= d * lam * lam
    assert idx.size == int(np.sum((np.abs(a) >= lam) & (a != 0)))


def test_ht_monotone_in_lambda():
    g = _f32(RNG.standard_normal(2000))
    e = np.zeros(2000, np.float32)
    prev = None
    for lam in [0.0, 0.1, 0.5, 1.0, 2.0, 3.0]:
        idx, _, _ = oracle.ef_hard_threshold(g, e, 1.0, lam)
        s = set(idx.tolist())
        if prev is not None:
            assert s <= prev
        prev = s


def test_ht_bf16_widening():
    # a bf16 value denotes exactly the fp32 value with the same high 16 bits
    torch = pytest.importorskip("torch")
    x = torch.randn(5000, generator=torch.Generator().manual_seed(3)) * 0.01
    gb = x.to(torch.bfloat16)
    bits = gb.view(torch.int16).numpy().view(np.uint16)
    widened = gb.to(torch.float32).numpy()
    e = _f32(RNG.standard_normal(5000) * 1e-3)
    r16 = oracle.ef_hard_threshold(bits, e, 0.1, 2e-3)
    r32 = oracle.ef_hard_threshold(widened, e, 0.1, 2e-3)
    for u, v in zip(r16, r32):
        assert _same_bits(u, v) if u.dtype == np.float32 else np.array_equal(u, v)
    t16 = oracle.ef_topk(bits, e, 0.1, 50)
    t32 = oracle.ef_topk(widened, e, 0.1, 50)
    for u, v in zip(t16, t32):
        assert _same_bits(u, v) if u.dtype == np.float32 else np.array_equal(u, v)


# --------------------------------------------------------------------------
# Top-k (Lemma 1 / Lemma 2): the support of size k minimising ||a - C(a)||^2
# --------------------------------------------------------------------------

def _bruteforce_topk(a, k):
    """All size-k supports minimising the exact squared error; the minimiser
    with the lexicographically smallest ascending index tuple (lowest-index
    tie rule)."""
    d = len(a)
    sq = [to_frac(x) ** 2 for x in a]
    total = sum(sq, Fraction(0))
    best, best_err = None, None
    for s in itertools.combinations(range(d), k):
        err = total - sum((sq[j] for j in s), Fraction(0))
        if best_err is None or err < best_err:
            best, best_err = s, err
        # combinations() enumerates in lexicographic order, so the first
        # minimiser found is the lexicographically smallest one
    return list(best), best_err


@pytest.mark.parametrize("seed", range(12))
def test_topk_matches_bruteforce_optimum(seed):
    rng = np.random.default_rng(seed)
    d = int(rng.integers(1, 11))
    if seed % 3 == 0:   # heavy ties, signed zeros
        pool = _f32([0.0, -0.0, 1.0, -1.0, 0.5, -0.5, 2.0])
        e = pool[rng.integers(0, len(pool), d)]
    else:
        e = _f32(rng.standard_normal(d))
    g = np.zeros(d, np.float32)
    a = _exact_a(g, e, 1.0)             # 1*0 + e, with (+0) + (-0) = +0
    for k in range(d + 1):
        idx, val, e_new = oracle.ef_topk(g, e, 1.0, k)
        want, err = _bruteforce_topk(a.tolist(), k)
        assert idx.tolist() == want, (e, k)
        assert _same_bits(val, a[want])
        assert sum((to_frac(x) ** 2 for x in e_new), Fraction(0)) == err
        assert int(np.count_nonzero(np.isin(np.arange(d), idx))) == k


def test_topk_matches_stable_argsort_with_ties():
    # library cross-check: a stable sort by decreasing |a| takes the lowest
    # index first among equal magnitudes
    d, k = 20000, 777
    e = _f32(np.round(RNG.standard_normal(d) * 4) / 4)   # many exact ties
    g = np.zeros(d, np.float32)
    idx, val, e_new = oracle.ef_topk(g, e, 1.0, k)
    want = np.sort(np.argsort(-np.abs(e), kind="stable")[:k])
    assert np.array_equal(idx, want.astype(np.uint32))


def test_topk_special_cases():
    g = _f32(RNG.standard_normal(500))
    e = _f32(RNG.standard_normal(500))
    a = _exact_a(g, e, 0.3)
    idx, val, e_new = oracle.ef_topk(g, e, 0.3, 0)          # k = 0: nothing sent
    assert idx.size == 0 and _same_bits(e_new, a)
    idx, val, e_new = oracle.ef_topk(g, e, 0.3, 500)        # k = d: identity
    assert idx.tolist() == list(range(500)) and _same_bits(val, a)
    assert not np.any(e_new)
    z = np.zeros(10, np.float32)                             # short support filled by zeros
    z[7] = -3.0
    idx, val, _ = oracle.ef_topk(np.zeros(10, np.float32), z, 1.0, 4)
    assert idx.tolist() == [0, 1, 2, 7]


@pytest.mark.parametrize("k", [1, 10, 100, 999])
def test_topk_delta_contraction_bound(k):
    # Top-k is a delta-contraction with delta = k/d (Sec. 4.4):
    # ||a - C(a)||^2 <= (1 - k/d) ||a||^2
    d = 1000
    g = _f32(RNG.standard_normal(d))
    e = _f32(RNG.standard_normal(d))
    a = _exact_a(g, e, 0.2).astype(np.float64)
    _, _, e_new = oracle.ef_topk(g, e, 0.2, k)
    assert np.sum(e_new.astype(np.float64) ** 2) <= (1 - k / d) * np.sum(a ** 2) + 1e-12


def test_topk_nan_inf_order():
    e = _f32([1.0, np.inf, np.nan, -np.inf, 5.0, -0.0])
    g = np.zeros(6, np.float32)
    idx, _, _ = oracle.ef_topk(g, e, 1.0, 1)
    assert idx.tolist() == [2]          # NaN ranks above +inf
    idx, _, _ = oracle.ef_topk(g, e, 1.0, 3)
    assert idx.tolist() == [1, 2, 3]    # +inf and -inf tie: lower index first
    idx, _, _ = oracle.ef_topk(g, e, 1.0, 4)
    assert idx.tolist() == [1, 2, 3, 4]
    # every NaN is one magnitude (a NaN carries no value): NaNs with different
    # payloads and signs tie, so the lowest indices win, never the payloads
    nans = np.array([0x7FC00001, 0x7FFFFFFF, 0xFFC00000, 0x7FC00002], np.uint32).view(np.float32)
    e = _f32([1.0, nans[0], np.inf, nans[1], nans[2], nans[3]])
    idx, val, e_new = oracle.ef_topk(np.zeros(6, np.float32), e, 1.0, 2)
    assert idx.tolist() == [1, 3] and np.all(np.isnan(val))
    assert e_new[1] == 0.0 and e_new[3] == 0.0 and np.isnan(e_new[4]) and np.isnan(e_new[5])
    idx, _, _ = oracle.ef_topk(np.zeros(6, np.float32), e, 1.0, 5)
    assert idx.tolist() == [1, 2, 3, 4, 5]


# --------------------------------------------------------------------------
# Layer-wise Top-k (Appendix: in layer-wise sparsification the sparsifier is
# invoked on each layer's tensor separately; hard-threshold is element-wise,
# so for it layer-wise and entire-model coincide, while Top-k differs)
# --------------------------------------------------------------------------

def test_topk_layerwise_hand_example():
    # tensors [1, -5, 2, 0.5] and [3, -1, 4] with k = (2, 1): the two largest
    # magnitudes of the first are -5 (index 1) and 2 (index 2), the largest of
    # the second is 4 (index 6); entire-model Top-3 takes -5, 3 and 4 instead
    g = _f32([1, -5, 2, 0.5, 3, -1, 4])
    e = np.zeros(7, np.float32)
    idx, val, e_new = oracle.ef_topk_layerwise(g, e, 1.0, [4, 7], [2, 1])
    assert idx.tolist() == [1, 2, 6]
    assert val.tolist() == [-5.0, 2.0, 4.0]
    assert e_new.tolist() == [1.0, 0.0, 0.0, 0.5, 3.0, -1.0, 0.0]
    assert oracle.ef_topk(g, e, 1.0, 3)[0].tolist() == [1, 4, 6]


def _random_table(rng, d):
    """Segment ends (empty segments allowed) and k_s in [0, d_s]."""
    cuts = np.sort(rng.integers(0, d + 1, int(rng.integers(0, 4))))
    ends = [int(c) for c in cuts] + [d]
    lo, ks = 0, []
    for hi in ends:
        ks.append(int(rng.integers(0, hi - lo + 1)))
        lo = hi
    return ends, ks


@pytest.mark.parametrize("seed", range(10))
def test_topk_layerwise_matches_bruteforce_per_segment(seed):
    rng = np.random.default_rng(100 + seed)
    d = int(rng.integers(1, 12))
    pool = _f32([0.0, -0.0, 1.0, -1.0, 0.5, -2.0, 2.0])
    e = pool[rng.integers(0, len(pool), d)] if seed % 2 else _f32(rng.standard_normal(d))
    g = np.zeros(d, np.float32)
    a = _exact_a(g, e, 1.0)
    ends, ks = _random_table(rng, d)
    idx, val, e_new = oracle.ef_topk_layerwise(g, e, 1.0, ends, ks)
    want, err, lo = [], Fraction(0), 0
    for hi, k in zip(ends, ks):   # each tensor's own optimum, at its offset
        sel, seg_err = _bruteforce_topk(a[lo:hi].tolist(), k)
        want += [lo + j for j in sel]
        err += seg_err
        lo = hi
    assert idx.tolist() == want, (e, ends, ks)
    assert _same_bits(val, a[want])
    assert sum((to_frac(x) ** 2 for x in e_new), Fraction(0)) == err
    rest = np.ones(d, bool)
    rest[want] = False
    assert _same_bits(e_new[rest], a[rest]) and not np.any(e_new[~rest])


def test_topk_layerwise_one_segment_is_entire_model():
    g = _f32(RNG.standard_normal(5000))
    e = _f32(RNG.standard_normal(5000))
    for k in (0, 1, 77, 5000):
        got = oracle.ef_topk_layerwise(g, e, 0.4, [5000], [k])
        ref = oracle.ef_topk(g, e, 0.4, k)
        for x, y in zip(got, ref):
            assert _same_bits(x, y) if x.dtype == np.float32 else np.array_equal(x, y)


def test_ht_is_the_same_layerwise_and_entire_model():
    # hard-threshold is element-wise: per-tensor calls, concatenated with
    # their offsets, give the entire-model result
    g = _f32(RNG.standard_normal(3000) * 0.01)
    e = _f32(RNG.standard_normal(3000) * 0.001)
    ref = oracle.ef_hard_threshold(g, e, 0.1, 2e-3)
    parts, lo = [], 0
    for hi in (700, 701, 2500, 3000):
        i, v, en = oracle.ef_hard_threshold(g[lo:hi], e[lo:hi], 0.1, 2e-3)
        parts.append((i + lo, v, en))
        lo = hi
    assert np.array_equal(np.concatenate([p[0] for p in parts]), ref[0])
    assert _same_bits(np.concatenate([p[1] for p in parts]), ref[1])
    assert _same_bits(np.concatenate([p[2] for p in parts]), ref[2])


def test_topk_layerwise_bf16_is_the_widened_fp32():
    g32 = _f32(RNG.standard_normal(4000))
    g16 = (g32.view(np.uint32) >> 16).astype(np.uint16)     # truncation: exact bf16 values
    gw = (g16.astype(np.uint32) << 16).view(np.float32)
    e = _f32(RNG.standard_normal(4000))
    got = oracle.ef_topk_layerwise(g16, e, 0.25, [1000, 1000, 4000], [10, 0, 300])
    ref = oracle.ef_topk_layerwise(gw, e, 0.25, [1000, 1000, 4000], [10, 0, 300])
    for x, y in zip(got, ref):
        assert _same_bits(x, y) if x.dtype == np.float32 else np.array_equal(x, y)


def test_topk_layerwise_rejects_bad_tables():
    g = np.zeros(10, np.float32)
    e = np.zeros(10, np.float32)
    for ends, ks in (([5, 10], [6, 0]),      # k_s above the segment's length
                     ([5, 9], [1, 1]),       # does not end at d
                     ([6, 5, 10], [0, 0, 0])):  # decreasing ends
        with pytest.raises(ValueError):
            oracle.ef_topk_layerwise(g, e, 1.0, ends, ks)


def test_ht_at_kth_magnitude_selects_topk():
    # Sec. 4.3 (Lemma 3 argument): with distinct magnitudes and
    # lambda in (|a|_(k+1), |a|_(k)], C_lambda keeps exactly the Top-k set
    for seed in range(5):
        rng = np.random.default_rng(100 + seed)
        d = 9
        e = _f32(rng.permutation(np.arange(1, d + 1)) * rng.choice([-1, 1], d) / 8)
        g = np.zeros(d, np.float32)
        mags = np.sort(np.abs(e))[::-1]
        for k in range(1, d + 1):
            lam = float(mags[k - 1])
            ht_idx, _, ht_e = oracle.ef_hard_threshold(g, e, 1.0, lam)
            want, _ = _bruteforce_topk(e.tolist(), k)
            assert ht_idx.tolist() == want
            tk_idx, _, tk_e = oracle.ef_topk(g, e, 1.0, k)
            assert tk_idx.tolist() == want and _same_bits(ht_e, tk_e)


# --------------------------------------------------------------------------
# aggregation (Algorithm 1, exchange step): ordered fp32 sum from +0.0
# --------------------------------------------------------------------------

def test_aggregate_single_worker_is_scatter():
    d = 50
    idx = np.array([0, 3, 17, 49], np.uint32)
    val = _f32([1.5, -2.25, -0.0, 7.0])
    dense = oracle.sparse_aggregate([idx], [val], d)
    want = np.zeros(d, np.float32)
    want[[0, 3, 49]] = [1.5, -2.25, 7.0]      # 0 + (-0) = +0
    assert _same_bits(dense, want)


def test_aggregate_disjoint_and_integer_sums_are_exact():
    d = 1000
    perm = RNG.permutation(d)
    idx_list = [np.sort(perm[i::4][:100]).astype(np.uint32) for i in range(4)]
    val_list = [_f32(RNG.integers(-1000, 1000, 100)) for _ in range(4)]
    dense = oracle.sparse_aggregate(idx_list, val_list, d)
    want = np.zeros(d, np.float64)
    for i, v in zip(idx_list, val_list):
        want[i] += v
    assert np.array_equal(dense, want.astype(np.float32))
    # overlapping supports with small integers: every partial sum is exact
    idx_list = [np.arange(0, d, s, dtype=np.uint32) for s in (1, 2, 3)]
    val_list = [_f32(RNG.integers(-50, 50, len(i))) for i in idx_list]
    dense = oracle.sparse_aggregate(idx_list, val_list, d)
    want = np.zeros(d, np.float64)
    for i, v in zip(idx_list, val_list):
        want[i] += v
    assert np.array_equal(dense, want.astype(np.float32))


def test_aggregate_sums_in_worker_order():
    # fp32: (0 + 2^24) + 1 = 2^24 (tie to even), then - 2^24 = 0;
    # any other order gives 1 or -2^24 + ... != 0
    big = np.float32(2.0 ** 24)
    idx = [np.array([5], np.uint32)] * 3
    dense = oracle.sparse_aggregate(idx, [_f32([big]), _f32([1.0]), _f32([-big])], 8)
    assert dense[5] == 0.0
    dense = oracle.sparse_aggregate(idx, [_f32([-big]), _f32([1.0]), _f32([big])], 8)
    assert dense[5] == 1.0


def test_aggregate_nan_propagates():
    nan = np.uint32(0x7FC00001).view(np.float32)
    dense = oracle.sparse_aggregate([np.array([1], np.uint32), np.array([1, 2], np.uint32)],
                                    [_f32([nan]), _f32([1.0, np.inf])], 3)
    assert dense[0] == 0.0 and np.isnan(dense[1]) and dense[2] == np.inf


def test_aggregate_rejects_out_of_range():
    with pytest.raises(RuntimeError):
        oracle.sparse_aggregate([np.array([10], np.uint32)], [_f32([1.0])], 10)


# --------------------------------------------------------------------------
# model update after the exchange step: Algorithm 1 (x <- x - mean of the
# Delta_i) and the Appendix's EF SGD with momentum by gradient compression
# (m <- mu m + Delta', x <- x - lr (Delta' + m))
# --------------------------------------------------------------------------
def test_update_algorithm1_subtracts_the_mean():
    # dyadic values keep every quantity exact, so the mean is a Fraction
    rng = np.random.default_rng(11)
    n, d = 4, 40
    idx_list, val_list = [], []
    for _ in range(n):
        ix = np.sort(rng.choice(d, 12, replace=False)).astype(np.uint32)
        idx_list.append(ix)
        val_list.append(_f32(rng.integers(-64, 65, 12) / 64.0))
    x0 = _f32(rng.integers(-32, 33, d) / 16.0)
    x, m = oracle.sparse_aggregate_apply(idx_list, val_list, d, 1.0 / n, x0)
    assert m is None
    want = [Fraction(float(v)) for v in x0]
    for ix, vv in zip(idx_list, val_list):
        for j, v in zip(ix, vv):
            want[j] -= Fraction(float(v)) / n
    assert [Fraction(float(v)) for v in x] == want


def test_update_momentum_closed_form():
    # a constant aggregate Delta' = c: m_t = c (1 - mu^t) / (1 - mu) and
    # x_t = x_{t-1} - lr (c + m_t); with mu = 1/2, lr = 1/4, c = 3/8 every
    # value is dyadic and exact in fp32 over these iterations
    mu, lr, c = Fraction(1, 2), Fraction(1, 4), Fraction(3, 8)
    d = 6
    idx = [np.array([1, 4], np.uint32), np.array([1, 4], np.uint32)]
    val = [_f32([0.375, 0.375]), _f32([0.375, 0.375])]  # alpha = 1/2: Delta' = 3/8
    x = _f32([0.5] * d)
    m = np.zeros(d, np.float32)
    xf, mf = Fraction(1, 2), Fraction(0)
    for t in range(1, 13):
        x, m = oracle.sparse_aggregate_apply(idx, val, d, 0.5, x, m, float(mu), float(lr))
        mf = mu * mf + c
        xf = xf - lr * (c + mf)
        assert mf == c * (1 - mu ** t) / (1 - mu)
        assert Fraction(float(m[1])) == mf and Fraction(float(m[4])) == mf
        assert Fraction(float(x[1])) == xf and Fraction(float(x[4])) == xf
        assert m[0] == 0.0 and x[0] == 0.5  # nothing sent: Delta' = 0, m stays 0


def test_update_momentum_zero_factor():
    # mu = 0: m = Delta' and x <- x - lr (Delta' + Delta'), as the algorithm is written
    idx = [np.array([0, 2], np.uint32)]
    val = [_f32([1.5, -2.0])]
    x, m = oracle.sparse_aggregate_apply(idx, val, 3, 1.0, _f32([1.0, 1.0, 1.0]),
                                         _f32([9.0, 9.0, 9.0]), 0.0, 0.25)
    assert list(m) == [1.5, 0.0, -2.0]
    assert list(x) == [1.0 - 0.25 * 3.0, 1.0, 1.0 + 0.25 * 4.0]


def test_update_rounding_follows_r12():
    # each step rounded as R12 states, predicted with exact rational arithmetic:
    # Delta' = RN(alpha s), m' = RN(mu m + Delta'), u = RN(Delta' + m'),
    # x' = RN(x - lr u); includes cases where a two-step mu m + Delta' differs
    rng = np.random.default_rng(12)
    d = 2000
    s_vals = _f32(rng.standard_normal(d) * rng.choice([1e-3, 1.0, 1e3], d))
    x0 = _f32(rng.standard_normal(d))
    m0 = _f32(rng.standard_normal(d) * 0.1)
    mu, lr, alpha = np.float32(0.9), np.float32(0.0123), np.float32(0.125)
    idx = [np.arange(d, dtype=np.uint32)]
    x, m = oracle.sparse_aggregate_apply(idx, [s_vals], d, float(alpha), x0, m0, float(mu),
                                         float(lr))
    differs = 0
    for j in range(d):
        delta = round_f32(to_frac(alpha) * to_frac(s_vals[j]))
        mj = fma_f32(mu, m0[j], delta)
        two_step = round_f32(to_frac(round_f32(to_frac(mu) * to_frac(m0[j]))) + to_frac(delta))
        differs += two_step != mj
        u = round_f32(to_frac(delta) + to_frac(mj))
        xj = fma_f32(-lr, u, x0[j])
        assert float(m[j]) == mj, j
        assert float(x[j]) == xj, j
    assert differs > 0


def test_update_sums_workers_in_order():
    # the update sees the worker-ordered sum: (0 + 2^24) + 1 - 2^24 = 0
    big = np.float32(2.0 ** 24)
    idx = [np.array([2], np.uint32)] * 3
    x, _ = oracle.sparse_aggregate_apply(idx, [_f32([big]), _f32([1.0]), _f32([-big])], 4, 1.0,
                                         _f32([5.0, 5.0, 5.0, 5.0]))
    assert x[2] == 5.0


# --------------------------------------------------------------------------
# per-step error norm ||e_{t+1}||^2 (the total error is its sum over t)
# --------------------------------------------------------------------------
def test_error_norm_hand_values_and_exactness():
    assert oracle.error_norm_sq(_f32([3.0, -4.0, 0.0])) == 25.0
    assert oracle.error_norm_sq(_f32([])) == 0.0
    # squares that fp32 cannot hold exactly are exact in fp64: (1 + 2^-23)^2
    x = np.float32(1.0) + np.float32(2.0 ** -23)
    assert oracle.error_norm_sq(_f32([x])) == float(Fraction(float(x)) ** 2)
    # tiny and huge values are neither flushed nor overflowed
    assert oracle.error_norm_sq(_f32([1e-30])) == float(np.float32(1e-30)) ** 2
    assert oracle.error_norm_sq(_f32([1e30])) == float(np.float32(1e30)) ** 2


def test_error_norm_bounds_of_the_sparsifiers():
    # hard-threshold: ||e'||_inf < lambda, so ||e'||^2 <= d lambda^2 (Sec. 5,
    # absolute compressor with kappa^2 = d lambda^2); Top-k: ||e'||^2 <=
    # (1 - k/d) ||a||^2 (the delta-contraction with delta = k/d)
    rng = np.random.default_rng(21)
    d = 5000
    g = _f32(rng.standard_normal(d))
    e = _f32(rng.standard_normal(d) * 0.1)
    for lam in (0.05, 0.2, 1.0):
        _, _, e_new = oracle.ef_hard_threshold(g, e, 0.1, lam)
        assert oracle.error_norm_sq(e_new) <= d * lam * lam
    _, _, a = oracle.ef_hard_threshold(g, e, 0.1, float("inf"))
    for k in (1, 50, 2500, 4999):
        _, _, e_new = oracle.ef_topk(g, e, 0.1, k)
        assert oracle.error_norm_sq(e_new) <= (1.0 - k / d) * oracle.error_norm_sq(a)
    _, _, e_new = oracle.ef_topk(g, e, 0.1, d)
    assert oracle.error_norm_sq(e_new) == 0.0


# --------------------------------------------------------------------------
# scaled integer rounding (Sec. 5: an absolute compressor)
# --------------------------------------------------------------------------
def test_scaled_round_hand_example():
    # grid 2^-2: 0.1 -> 0 (0.4), 0.125 -> 0 (0.5, to even), 0.375 -> 2 (1.5,
    # to even), -0.625 -> -2 (-2.5, to even), 3.0 -> 12, 0.25 + tiny -> 1
    a = _f32([0.1, 0.125, 0.375, -0.625, 3.0, 0.26])
    q, e_new, unsent = oracle.ef_scaled_round(np.zeros(6, np.float32), a, 1.0, 2)
    assert list(q) == [0, 0, 2, -2, 12, 1] and unsent == 0
    assert list(e_new) == [np.float32(0.1), 0.125, -0.125, -0.125, 0.0, np.float32(0.26) - 0.25]


def test_scaled_round_is_an_absolute_compressor():
    # |e'_j| <= 2^(-m-1) for every coordinate, so ||e'||^2 <= d 2^(-2m-2)
    # (kappa^2 = d eps^2, Sec. 5), and a = C(a) + e' exactly
    rng = np.random.default_rng(31)
    d = 4000
    g = _f32(rng.standard_normal(d) * 10.0)
    e = _f32(rng.standard_normal(d))
    for m in (-3, 0, 4, 17):
        q, e_new, unsent = oracle.ef_scaled_round(g, e, 0.1, m)
        assert unsent == 0
        a = [fma_f32(np.float32(0.1), gj, ej) for gj, ej in zip(g, e)]
        eps = Fraction(2) ** (-m - 1)
        for j in range(d):
            c = Fraction(int(q[j])) * Fraction(2) ** (-m)
            assert Fraction(float(a[j])) == c + Fraction(float(e_new[j]))
            assert abs(Fraction(float(e_new[j]))) <= eps
            # q is the nearest integer to a 2^m, ties to even
            t = Fraction(float(a[j])) * Fraction(2) ** m
            fl = t.numerator // t.denominator
            want = fl + 1 if (t - fl > Fraction(1, 2) or (t - fl == Fraction(1, 2) and fl % 2)) else fl
            assert int(q[j]) == want
        assert oracle.error_norm_sq(e_new) <= d * float(eps) ** 2


def test_scaled_round_unsent_coordinates():
    # a 2^m at or beyond 2^31, infinities and NaN are not sent: q = 0, e' = a
    a = _f32([2.0 ** 31, -(2.0 ** 31), 2.0 ** 31 - 128.0, np.inf, np.nan, 1.0])
    q, e_new, unsent = oracle.ef_scaled_round(np.zeros(6, np.float32), a, 1.0, 0)
    assert unsent == 4
    assert list(q[:3]) == [0, 0, 2 ** 31 - 128] and q[3] == 0 and q[4] == 0 and q[5] == 1
    assert e_new[0] == 2.0 ** 31 and e_new[1] == -(2.0 ** 31) and e_new[2] == 0.0
    assert np.isinf(e_new[3]) and np.isnan(e_new[4]) and e_new[5] == 0.0


def test_scaled_round_bf16_hand_example():
    # bf16 bit patterns widened by hand: 0x3F80 = 1.0, 0xBFC0 = -1.5,
    # 0x4049 = 3.140625, 0x0001 = 2^-133 (a subnormal), 0x7F80 = +inf,
    # 0xC780 = -65536; grid 2^-2 (m = 2), gamma = 1, e = 0
    bits = np.array([0x3F80, 0xBFC0, 0x4049, 0x0001, 0x7F80, 0xC780], np.uint16)
    q, e_new, unsent = oracle.ef_scaled_round(bits, np.zeros(6, np.float32), 1.0, 2)
    assert list(q) == [4, -6, 13, 0, 0, -262144] and unsent == 1
    assert e_new[0] == 0.0 and e_new[1] == 0.0 and e_new[2] == 3.140625 - 3.25
    assert e_new[3] == np.float32(2.0 ** -133) and e_new[4] == np.inf and e_new[5] == 0.0


def test_scaled_round_bf16_is_the_widened_fp32():
    # on bf16 bit patterns the step equals the fp32 step on the values they
    # denote, bit for bit: q, e' and the unsent count; the widening here is
    # torch's own bf16 -> fp32 conversion
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(77)
    x = torch.from_numpy(_f32(rng.standard_normal(6000) *
                              np.exp2(rng.integers(-130, 40, 6000))))
    gb = x.to(torch.bfloat16)
    bits = gb.view(torch.int16).numpy().view(np.uint16).copy()
    bits[:4] = [0x7F80, 0xFF80, 0x7FC0, 0x8000]           # +inf, -inf, NaN, -0
    widened = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float32).numpy()
    e = _f32(rng.standard_normal(6000) * 1e-3)
    for m in (0, 7, 20, 40):
        q16, e16, u16 = oracle.ef_scaled_round(bits, e, 0.1, m)
        q32, e32, u32 = oracle.ef_scaled_round(widened, e, 0.1, m)
        assert u16 == u32 and u16 >= 3
        assert np.array_equal(q16, q32)
        assert np.array_equal(np.isnan(e16), np.isnan(e32))
        ok = ~np.isnan(e16)
        assert _same_bits(e16[ok], e32[ok])


def test_int_aggregate_is_exact_and_order_free():
    # the integer sum is exact whatever the order; one rounding at the end
    big = 2 ** 30
    q1 = np.array([big, 1, -7], np.int32)
    q2 = np.array([big, 2, 7], np.int32)
    q3 = np.array([-big, 4, 0], np.int32)
    for order in ([q1, q2, q3], [q3, q2, q1], [q2, q3, q1]):
        dense = oracle.int_aggregate(order, 3, 3)
        assert list(dense) == [float(big) / 8, 7 / 8, 0.0]
    # 2^25 + 1 rounds once to 2^25 (ties to even), then scales
    dense = oracle.int_aggregate([np.array([2 ** 24 + 1], np.int32),
                                  np.array([2 ** 24], np.int32)], 1, 0)
    assert dense[0] == 2.0 ** 25
    # (2^24 + 1) + 1 - 2^24 = 2 exactly; an fp32 running sum would give 0
    dense = oracle.int_aggregate([np.array([2 ** 24 + 1], np.int32), np.array([1], np.int32),
                                  np.array([-(2 ** 24)], np.int32)], 1, 0)
    assert dense[0] == 2.0


# --------------------------------------------------------------------------
# multi-iteration EF: Lemma 9 (virtual iterate) per worker
# --------------------------------------------------------------------------

@pytest.mark.parametrize("method", ["ht", "topk"])
def test_error_feedback_conserves_mass(method):
    # sum_t Delta_t + e_T = sum_t gamma g_t exactly, up to the single rounding
    # of each fma: |gap_j| <= sum_t ulp(a_t[j]) / 2
    d, T, gamma = 300, 12, 0.1
    e = np.zeros(d, np.float32)
    sent = [Fraction(0)] * d
    target = [Fraction(0)] * d
    slack = [Fraction(0)] * d
    for t in range(T):
        g = _f32(RNG.standard_normal(d) * 0.01)
        a = _exact_a(g, e, gamma)
        if method == "ht":
            idx, val, e = oracle.ef_hard_threshold(g, e, gamma, 2e-3)
        else:
            idx, val, e = oracle.ef_topk(g, e, gamma, 15)
        for j, v in zip(idx.tolist(), val.tolist()):
            sent[j] += to_frac(v)
        for j in range(d):
            target[j] += to_frac(np.float32(gamma)) * to_frac(g[j])
            slack[j] += ulp_f32(a[j]) / 2
    for j in range(d):
        gap = abs(sent[j] + to_frac(e[j]) - target[j])
        assert gap <= slack[j], j


def test_round_f32_helper_agrees_with_numpy_on_doubles():
    # the exact helper itself: rounding a double to binary32 matches numpy
    xs = RNG.standard_normal(2000) * np.exp2(RNG.integers(-140, 100, 2000))
    for x in xs:
        assert _same_bits([round_f32(Fraction(float(x)))], [np.float32(x)])
