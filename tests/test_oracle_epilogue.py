"""Pins of the oracle's spiking-linear IF epilogue (scale, residual, gate)."""
import numpy as np

import oracle


def test_int_epilogue_is_if_on_raw_sums():
    g = np.random.default_rng(1)
    B, T, d = 3, 4, 40
    acc = g.integers(-200, 200, size=(B * T, d)).astype(np.int64)
    sc = np.full(d, 0.5, np.float32)
    cur, s, _ = oracle.if_epilogue(acc, B, T, scale=sc, kind=oracle.EPI_INT, theta_i=64)
    ref, _ = oracle.if_int(acc.reshape(B, T, d), 64)
    assert np.array_equal(s.reshape(B, T, d), ref)
    assert np.array_equal(cur, acc.astype(np.float32) * np.float32(0.5))


def test_f32_epilogue_dyadic_scale_matches_int():
    # scale 2^-6 with threshold 1.0 is the integer threshold 64 on the raw sum.
    g = np.random.default_rng(2)
    B, T, d = 4, 4, 50
    acc = g.integers(-300, 300, size=(B * T, d)).astype(np.int64)
    sc = np.full(d, 2.0 ** -6, np.float32)
    cur, s, m = oracle.if_epilogue(acc, B, T, scale=sc, kind=oracle.EPI_F32, theta_f=1.0)
    ref, _ = oracle.if_int(acc.reshape(B, T, d), 64)
    assert np.array_equal(s.reshape(B, T, d), ref)
    assert np.all(m >= 0)


def test_residual_only_and_gate():
    g = np.random.default_rng(3)
    B, T, d = 2, 4, 30
    res = g.standard_normal((B * T, d)).astype(np.float32)
    zero = np.zeros((B * T, d), np.int64)
    sc = np.ones(d, np.float32)
    cur, s, _ = oracle.if_epilogue(zero, B, T, scale=sc, residual=res, kind=oracle.EPI_F32)
    ref, _, _ = oracle.if_f32(res.reshape(B, T, d), 1.0)
    assert np.array_equal(s.reshape(B, T, d), ref) and np.array_equal(cur, res)
    # a closed gate blocks every current; an open gate changes nothing
    acc = g.integers(0, 300, size=(B * T, d)).astype(np.int64)
    sc2 = np.full(d, 0.01, np.float32)
    _, s0, _ = oracle.if_epilogue(acc, B, T, scale=sc2, gate=np.zeros((B * T, d), np.uint8))
    assert s0.sum() == 0
    _, s1, _ = oracle.if_epilogue(acc, B, T, scale=sc2, gate=np.ones((B * T, d), np.uint8))
    _, sn, _ = oracle.if_epilogue(acc, B, T, scale=sc2)
    assert np.array_equal(s1, sn) and sn.sum() > 0


def test_residual_current_hand_worked():
    # one channel, T=4: acc=[100,0,0,50], scale=0.01 -> I=[1,0,0,0.5]; residual 0.25
    # each step -> currents [1.25, .25, .25, .75] -> H: 1.25 fire V=.25; .5; .75; 1.5 fire
    acc = np.array([[100], [0], [0], [50]], np.int64)
    res = np.full((4, 1), 0.25, np.float32)
    cur, s, _ = oracle.if_epilogue(acc, 1, 4, scale=np.array([0.01], np.float32), residual=res)
    assert s.reshape(-1).tolist() == [1, 0, 0, 1]
    exp = [np.float32(100) * np.float32(0.01) + np.float32(0.25), np.float32(0.25),
           np.float32(0.25), np.float32(50) * np.float32(0.01) + np.float32(0.25)]
    assert cur.reshape(-1).tolist() == [float(x) for x in exp]
