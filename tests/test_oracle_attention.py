"""Pins of the oracle's BBM spike attention to a hand-worked example, closed forms
and library routines (numpy popcount, scipy softmax)."""
import math

import numpy as np
import pytest
from scipy.special import softmax

import oracle
from conftest import golden


def test_attention_hand_worked():
    g = golden("attention_worked.json")
    q = np.array(g["q"], np.uint8).reshape(1, 4)
    k = np.array(g["k"], np.uint8).reshape(1, 3, 4)
    v = np.array(g["v"], np.uint8).reshape(1, 3, 4)
    out = oracle.attention(q, k, v, B=1, T=1, H=1, dh=4)
    assert np.allclose(out[0], g["out"], atol=1e-7)


def _case(seed, B, T, L, H, dh, p):
    g = np.random.default_rng(seed)
    D = H * dh
    q = (g.random((B * T, D)) < p).astype(np.uint8)
    k = (g.random((T, L, D)) < p).astype(np.uint8)
    v = (g.random((T, L, D)) < p).astype(np.uint8)
    return q, k, v


def test_equal_scores_give_column_mean():
    # q = 0 makes every score 0: the softmax is uniform and out = mean_j v_j.
    B, T, L, H, dh = 3, 2, 17, 2, 32
    _, k, v = _case(1, B, T, L, H, dh, 0.3)
    q = np.zeros((B * T, H * dh), np.uint8)
    out = oracle.attention(q, k, v, B, T, H, dh).reshape(B, T, H * dh)
    mean = v.mean(axis=1)  # [T, D]
    for b in range(B):
        assert np.allclose(out[b], mean, rtol=0, atol=1e-6)


def test_single_key_returns_v():
    B, T, H, dh = 4, 3, 2, 32
    q, k, v = _case(2, B, T, 1, H, dh, 0.4)
    out = oracle.attention(q, k, v, B, T, H, dh).reshape(B, T, H * dh)
    for b in range(B):
        assert np.array_equal(out[b], v[:, 0, :].astype(np.float32))


def test_one_hot_values_expose_softmax_of_popcounts():
    # V_j = e_j (one-hot over channels) makes out[c=j] the softmax weight p_j, so the
    # score path (AND + popcount, numpy bitwise_count), alpha scaling and softmax
    # (scipy) are checked together on every query.
    B, T, H, dh = 3, 2, 1, 64
    L = dh
    q, k, _ = _case(3, B, T, L, H, dh, 0.35)
    v = np.zeros((T, L, dh), np.uint8)
    for t in range(T):
        v[t] = np.eye(L, dtype=np.uint8)
    out = oracle.attention(q, k, v, B, T, H, dh).reshape(B, T, dh)
    qb = np.packbits(q.reshape(B, T, dh), axis=-1)
    kb = np.packbits(k, axis=-1)
    alpha = 1.0 / math.sqrt(dh)
    for b in range(B):
        for t in range(T):
            sc = np.bitwise_count(qb[b, t][None, :] & kb[t]).sum(axis=-1)
            p = softmax(alpha * sc.astype(np.float64))
            assert np.allclose(out[b, t], p, rtol=1e-6, atol=1e-7)


def test_heads_and_timesteps_are_independent():
    B, T, L, H, dh = 2, 3, 9, 3, 32
    q, k, v = _case(4, B, T, L, H, dh, 0.3)
    base = oracle.attention(q, k, v, B, T, H, dh).reshape(B, T, H, dh)
    k2 = k.copy()
    k2[1, :, 2 * dh:] ^= 1  # perturb head 2 at timestep 1 only
    pert = oracle.attention(q, k2, v, B, T, H, dh).reshape(B, T, H, dh)
    assert np.array_equal(base[:, :, :2], pert[:, :, :2])
    assert np.array_equal(base[:, [0, 2], 2], pert[:, [0, 2], 2])
    assert not np.array_equal(base[:, 1, 2], pert[:, 1, 2])


def test_output_is_convex_mixture():
    B, T, L, H, dh = 4, 2, 50, 2, 32
    q, k, v = _case(5, B, T, L, H, dh, 0.2)
    out = oracle.attention(q, k, v, B, T, H, dh)
    assert out.min() >= 0.0 and out.max() <= 1.0 + 1e-7
    # channels whose V column is all ones get exactly 1, all zeros get exactly 0
    v2 = v.copy()
    v2[:, :, 0] = 1
    v2[:, :, 1] = 0
    out2 = oracle.attention(q, k, v2, B, T, H, dh).reshape(B, T, H * dh)
    assert np.allclose(out2[:, :, 0], 1.0, atol=1e-6) and np.all(out2[:, :, 1] == 0)
