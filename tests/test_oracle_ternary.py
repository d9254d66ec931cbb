"""Pins of the oracle's ternary bitwise coding (Sec. II-C, Eq. (7)-(8)) and of the
linear on ternary spikes, against values and identities the paper and arithmetic fix
(no GPU)."""
import math

import numpy as np
import pytest

import oracle


def test_hand_worked_example():
    # mean|a| = (1 + 2 + 0.5 + 3) / 4 = 1.625, K = 2 -> V_th = 0.8125 (exact in fp32);
    # a / V_th = 1.23, -2.46, 0.615, 3.69 -> round -> 1, -2, 1, 4; T = 3 planes:
    # 1 = +2^0, -2 = -2^1, 4 = +2^2.
    a = np.array([[1.0, -2.0, 0.5, 3.0]], np.float32)
    s, ah, vth = oracle.ternary_encode(a, 2.0, 3)
    assert vth[0] == np.float32(0.8125)
    assert ah.tolist() == [[1, -2, 1, 4]]
    assert s[0, :, 0].tolist() == [1, 0, 0]
    assert s[0, :, 1].tolist() == [0, -1, 0]
    assert s[0, :, 2].tolist() == [1, 0, 0]
    assert s[0, :, 3].tolist() == [0, 0, 1]


@pytest.mark.parametrize("K,T", [(1.0, 4), (3.0, 6), (8.0, 8)])
def test_bitwise_reconstruction_eq8(K, T):
    g = np.random.default_rng(7)
    a = g.standard_normal((5, 300)).astype(np.float32) * 3
    s, ah, _ = oracle.ternary_encode(a, K, T)
    assert set(np.unique(s)) <= {-1, 0, 1}
    w = (1 << np.arange(T)).astype(np.int64)
    assert np.array_equal((s.astype(np.int64) * w[None, :, None]).sum(1), ah)
    # every nonzero spike carries the sign of its value
    sg = np.sign(ah)[:, None, :]
    assert np.all((s == 0) | (s == sg))


def test_quantiser_closed_forms():
    # a constant vector: mean|a| = c, V_th = c / K, a / V_th = K
    for K in (1.0, 3.0, 5.0):
        s, ah, vth = oracle.ternary_encode(np.full((1, 64), 0.75, np.float32), K, 8)
        assert np.all(ah == round(K))
    # +-x: same magnitude, opposite signs
    s, ah, _ = oracle.ternary_encode(np.array([[2.5, -2.5, 2.5, -2.5]], np.float32), 4.0, 8)
    assert ah.tolist() == [[4, -4, 4, -4]]
    # scaling by a power of two changes V_th by the same factor and nothing else
    g = np.random.default_rng(3)
    a = g.standard_normal((3, 129)).astype(np.float32)
    s1, ah1, v1 = oracle.ternary_encode(a, 2.0, 8)
    s2, ah2, v2 = oracle.ternary_encode(a * np.float32(4.0), 2.0, 8)
    assert np.array_equal(ah1, ah2) and np.array_equal(s1, s2)
    assert np.array_equal(v2, v1 * np.float32(4.0))


def test_mean_magnitude_is_K_within_half():
    # mean_i |a_i / V_th| = K exactly, and rounding moves each |ahat_i| by at most 1/2,
    # so without clamping |mean|ahat| - K| <= 1/2.
    g = np.random.default_rng(11)
    a = g.standard_normal((8, 1000)).astype(np.float32)
    for K in (0.5, 1.0, 2.0, 4.0, 8.0):
        _, ah, _ = oracle.ternary_encode(a, K, 16)
        m = np.abs(ah).mean(axis=1)
        assert np.all(np.abs(m - K) <= 0.5 + 1e-4), (K, m)


def test_more_levels_fewer_zero_spikes():
    # Larger K, finer steps: the share of zero-valued activations falls and the spike
    # count rises (the K-sparsity trade-off of Sec. IV).
    g = np.random.default_rng(5)
    a = g.standard_normal((4, 4096)).astype(np.float32)
    zeros, spikes = [], []
    for K in (0.5, 1.0, 2.0, 4.0, 8.0):
        s, ah, _ = oracle.ternary_encode(a, K, 12)
        zeros.append(float((ah == 0).mean()))
        spikes.append(int(np.count_nonzero(s)))
    assert all(x > y for x, y in zip(zeros, zeros[1:]))
    assert all(x < y for x, y in zip(spikes, spikes[1:]))


def test_degenerate_rows():
    a = np.zeros((2, 33), np.float32)
    a[1, 5] = np.nan
    a[1, 6] = 1.0
    s, ah, vth = oracle.ternary_encode(a, 2.0, 4)
    assert vth[0] == 0 and not ah[0].any() and not s[0].any()
    # a NaN makes the row's mean NaN: V_th is NaN and every value quantises to 0
    assert not ah[1].any() and not s[1].any()


def test_clamp_at_T_planes():
    T = 4
    a = np.zeros((1, 100), np.float32)
    a[0, 0] = 1000.0   # far beyond 2^T - 1 steps
    a[0, 1:] = 0.01
    s, ah, _ = oracle.ternary_encode(a, 1.0, T)
    assert ah[0, 0] == (1 << T) - 1
    assert s[0, :, 0].tolist() == [1] * T


def test_planes_needed_and_the_printed_formula():
    # Eq. (8) with T planes reaches at most 2^T - 1; the bit length of m is the least
    # T that reaches m, one more than floor(log2 m).
    assert oracle.ternary_planes_needed(0) == 0
    for m in range(1, 2049):
        n = oracle.ternary_planes_needed(m)
        assert n == int(math.floor(math.log2(m))) + 1
        assert (1 << n) - 1 >= m > (1 << (n - 1)) - 1


def test_ternary_linear_equals_weights_times_ahat():
    g = np.random.default_rng(21)
    N, D, d_out, T = 3, 97, 40, 6
    a = g.standard_normal((N, D)).astype(np.float32)
    w = g.integers(-127, 128, (D, d_out), dtype=np.int64).astype(np.int8)
    s, ah, _ = oracle.ternary_encode(a, 4.0, T)
    I, y = oracle.ternary_linear(s, w)
    # distributivity: sum_t 2^{t-1} (W^T s_t) = W^T (sum_t 2^{t-1} s_t) = W^T ahat
    assert np.array_equal(y, ah.astype(np.int64) @ w.astype(np.int64))
    for t in range(T):
        assert np.array_equal(I[:, t, :], s[:, t, :].astype(np.int64) @ w.astype(np.int64))


def test_ternary_linear_brute_force_tiny():
    s = np.array([[[1, 0, -1], [0, 1, 1]]], np.int8)          # N 1, T 2, D 3
    w = np.array([[2, -1], [3, 4], [-5, 6]], np.int8)           # D 3, d_out 2
    I, y = oracle.ternary_linear(s, w)
    # t = 1: 2 - (-5) = 7, -1 - 6 = -7;  t = 2: 3 + (-5) = -2, 4 + 6 = 10
    assert I.tolist() == [[[7, -7], [-2, 10]]]
    assert y.tolist() == [[7 - 4, -7 + 20]]


def _exact_abs_sum(row):
    """Python's exact rational sum of |a|, converted with correct rounding."""
    from fractions import Fraction
    return float(sum((Fraction(float(abs(x))) for x in row), Fraction(0)))


@pytest.mark.parametrize("case", ["normal", "wide", "subnormal", "ties", "big"])
def test_abs_sum_exact_is_the_rational_sum(case):
    # Eq. (7)'s sum of |a| is taken exactly and rounded once: it must equal the exact
    # rational sum (Python fractions, an arithmetic independent of the oracle) rounded to
    # the nearest double, for any mix of magnitudes, including exact ties.
    g = np.random.default_rng({"normal": 1, "wide": 2, "subnormal": 3, "ties": 4, "big": 5}[case])
    if case == "normal":
        row = g.standard_normal(4096).astype(np.float32)
    elif case == "wide":  # 60 decades of magnitude: an fp64 running sum loses bits here
        row = (g.standard_normal(999) * 10.0 ** g.integers(-30, 30, 999)).astype(np.float32)
    elif case == "subnormal":
        row = (g.standard_normal(300) * 1e-39).astype(np.float32)
    elif case == "ties":  # 2^53 + 1 and 2^54 + 2: halfway cases, ties to even
        row = np.array([2.0 ** 53, 1.0, 2.0 ** 54, 2.0, 2.0 ** 53, 1.0], np.float32)
    else:
        row = np.full(5000, 3.0e38, np.float32)
    assert oracle.abs_sum_exact(row) == _exact_abs_sum(row)


def test_abs_sum_exact_ignores_order_and_flags_non_finite():
    g = np.random.default_rng(9)
    row = (g.standard_normal(2048) * 10.0 ** g.integers(-20, 20, 2048)).astype(np.float32)
    s = oracle.abs_sum_exact(row)
    for _ in range(3):
        assert oracle.abs_sum_exact(g.permutation(row)) == s
    # an fp64 running sum in two different orders can differ; the exact sum cannot
    assert oracle.abs_sum_exact(np.array([1.0, -np.inf, 2.0], np.float32)) == math.inf
    assert math.isnan(oracle.abs_sum_exact(np.array([1.0, np.nan, -np.inf], np.float32)))
    assert oracle.abs_sum_exact(np.zeros(7, np.float32)) == 0.0


def test_vth_from_the_exact_sum():
    # V_th = fp32((sum / D) / K) with sum the correctly rounded exact sum of |a|
    g = np.random.default_rng(12)
    a = (g.standard_normal((4, 777)) * 10.0 ** g.integers(-8, 8, (4, 777))).astype(np.float32)
    _, _, vth = oracle.ternary_encode(a, 3.0, 8)
    for n in range(4):
        assert vth[n] == np.float32((_exact_abs_sum(a[n]) / 777) / 3.0)


def test_modified_if_hand_worked():
    # Eq. (9)-(10), most significant step first (header reading):
    # y = 5, T = 3, theta = 1: 5 >= 4 -> +1 (V 1); 1 < 2 -> 0; 1 >= 1 -> +1 (V 0)
    # y = -6: -6 <= -4 -> -1 (V -2); -2 <= -2 -> -1 (V 0); 0
    # theta = 2, y = 7: 7 < 8 -> 0; 7 >= 4 -> +1 (V 3); 3 >= 2 -> +1 (V 1)
    s, v = oracle.ternary_if(np.array([[5, -6]]), 3, 1)
    assert s[0, :, 0].tolist() == [1, 0, 1] and s[0, :, 1].tolist() == [0, -1, -1]
    assert v.tolist() == [[0, 0]]
    s, v = oracle.ternary_if(np.array([[7]]), 3, 2)
    assert s[0, :, 0].tolist() == [1, 1, 0] and v.tolist() == [[1]]


def test_modified_if_with_unit_step_is_the_bitwise_coding():
    # theta = 1 re-encodes y exactly as Eq. (8) codes an integer: sign(y) * bits of |y|
    g = np.random.default_rng(21)
    T = 7
    y = g.integers(-(2 ** T) + 1, 2 ** T, (4, 50))
    s, v = oracle.ternary_if(y, T, 1)
    assert not v.any()
    mag = np.abs(y)
    want = np.stack([((mag >> t) & 1) * np.sign(y) for t in range(T)], axis=1)
    assert np.array_equal(s, want)


@pytest.mark.parametrize("theta", [1, 3, 17])
def test_modified_if_reconstruction_eq11(theta):
    # theta * sum_t 2^{t-1} s_t = y - V_T with |V_T| < theta whenever |y| < 2^T theta
    g = np.random.default_rng(theta)
    T = 6
    y = g.integers(-(2 ** T) * theta + 1, (2 ** T) * theta, (3, 200))
    s, v = oracle.ternary_if(y, T, theta)
    w = (1 << np.arange(T)).astype(np.int64)
    rec = theta * (s.astype(np.int64) * w[None, :, None]).sum(1)
    assert np.array_equal(rec, y - v)
    assert np.all(np.abs(v) < theta)
