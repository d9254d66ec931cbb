"""Pins of the oracle's IF neuron (Sec. II-B, Eq. (3)-(4)) to hand-worked values,
invariants and closed forms."""
import numpy as np
import pytest

import oracle
from conftest import golden


def test_if_int_hand_worked():
    g = golden("if_worked.json")
    for case in g["int_cases"]:
        order = (oracle.IF_FIRE_THEN_CHARGE if case["order"] == "fire_then_charge"
                 else oracle.IF_CHARGE_THEN_FIRE)
        cur = np.array(case["current"], np.int64).reshape(1, -1, 1)
        s, v = oracle.if_int(cur, case["theta"], order)
        assert s.reshape(-1).tolist() == case["spikes"], case
        if order == oracle.IF_CHARGE_THEN_FIRE:
            assert int(v[0, 0]) == case["v_final"], case


def test_if_f32_hand_worked():
    g = golden("if_worked.json")
    for case in g["f32_cases"]:
        cur = np.array(case["current"], np.float32).reshape(1, -1, 1)
        s, v, m = oracle.if_f32(cur, case["theta"])
        assert s.reshape(-1).tolist() == case["spikes"]
        assert float(v[0, 0]) == case["v_final"]
        assert float(m[0, 0]) == 0.0  # both cases hit the threshold exactly


def test_if_charge_conservation():
    # Eq. (4) summed over t: sum_t s_t * th = sum_t I_t - V_T (reset by subtraction).
    g = np.random.default_rng(11)
    cur = g.integers(-300, 300, size=(5, 9, 37)).astype(np.int64)
    for theta in (1, 7, 64, 500):
        s, v = oracle.if_int(cur, theta)
        lhs = s.sum(axis=1).astype(np.int64) * theta
        rhs = cur.sum(axis=1) - v
        assert np.array_equal(lhs, rhs)
        # at most one spike per step, and V stays below the threshold after a spike
        assert s.max() <= 1


def test_if_constant_current_closed_form():
    # For constant 0 <= I <= th the count after T steps is floor(T*I/th).
    T, theta = 8, 64
    I = np.arange(0, theta + 1, dtype=np.int64)
    cur = np.repeat(I[None, None, :], T, axis=1)
    s, _ = oracle.if_int(cur, theta)
    assert np.array_equal(s.sum(axis=1)[0], (T * I) // theta)
    # I >= th fires at every step
    s2, _ = oracle.if_int(np.full((1, T, 3), 3 * theta, np.int64), theta)
    assert s2.sum() == 3 * T


def test_if_zero_current_no_spikes():
    s, v = oracle.if_int(np.zeros((3, 4, 10), np.int64), 64)
    assert s.sum() == 0 and np.all(v == 0)
    s, v, _ = oracle.if_f32(np.zeros((3, 4, 10), np.float32), 1.0)
    assert s.sum() == 0


@pytest.mark.parametrize("k", [0, -3, -7])
def test_if_f32_matches_int_on_dyadic_currents(k):
    # Integer currents scaled by 2^k are exact in fp32, so the fp32 neuron with the
    # threshold scaled the same way must reproduce the integer neuron bit for bit.
    g = np.random.default_rng(5)
    cur = g.integers(-200, 200, size=(4, 6, 50)).astype(np.int64)
    theta = 64
    s_i, v_i = oracle.if_int(cur, theta)
    sc = np.float32(2.0 ** k)
    s_f, v_f, _ = oracle.if_f32(cur.astype(np.float32) * sc, float(theta * sc))
    assert np.array_equal(s_i, s_f)
    assert np.array_equal(v_i.astype(np.float32) * sc, v_f)


def test_if_literal_order_loses_first_step():
    # With the literal Eq. (3)-(4) order and V_1 = 0 the first step never fires.
    g = np.random.default_rng(3)
    cur = g.integers(0, 500, size=(2, 4, 40)).astype(np.int64)
    s, _ = oracle.if_int(cur, 64, oracle.IF_FIRE_THEN_CHARGE)
    assert s[:, 0, :].sum() == 0
