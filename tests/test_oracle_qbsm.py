"""Pins of the oracle's packing, QBSM product and event counts (Sec. IV-A,
Eq. (12)-(13)) to library routines, hand-worked values, identities and statistics."""
import math

import numpy as np
import pytest

import oracle
from conftest import golden


def _bits_le(a):
    """numpy packbits, little bit order, grouped in uint32 words."""
    a = np.asarray(a, np.uint8)
    n = a.shape[-1]
    pad = (-n) % 32
    a = np.concatenate([a, np.zeros(a.shape[:-1] + (pad,), np.uint8)], axis=-1)
    by = np.packbits(a, axis=-1, bitorder="little")
    return by.view("<u4")


@pytest.mark.parametrize("BT,D,p", [(16, 256, 0.2), (5, 77, 0.1), (33, 40, 0.5), (1, 1, 1.0),
                                    (128, 300, 0.02)])
def test_pack_matches_numpy_bit_routines(BT, D, p):
    g = np.random.default_rng(BT * 1000 + D)
    s = (g.random((BT, D)) < p).astype(np.uint8)
    r = oracle.pack(s)
    assert np.array_equal(r["row_bits"], _bits_le(s))
    assert np.array_equal(r["col_masks"], _bits_le(s.T))
    idx = np.nonzero(s.any(axis=0))[0]
    assert np.array_equal(r["active_idx"], idx)
    assert r["n_active"] == idx.size
    mask = _bits_le(s.any(axis=0).astype(np.uint8)[None, :])[0]
    assert np.array_equal(r["active_mask"], mask)


def test_pack_zero_spikes():
    r = oracle.pack(np.zeros((16, 256), np.uint8))
    assert r["n_active"] == 0 and r["active_idx"].size == 0
    assert r["row_bits"].sum() == 0 and r["col_masks"].sum() == 0


@pytest.mark.parametrize("p,BT,expect", [(0.2, 16, 0.9719), (0.02, 4, 0.0776),
                                         (0.1, 128, 1.0)])
def test_active_fraction_statistics(p, BT, expect):
    # Sec. IV-A: each row of W is loaded with probability 1 - sigma^{BT}, sigma = 1-p.
    D = 4096
    q = 1.0 - (1.0 - p) ** BT
    assert abs(q - expect) < 1e-3
    g = np.random.default_rng(7)
    s = (g.random((BT, D)) < p).astype(np.uint8)
    n = oracle.pack(s)["n_active"]
    sd = math.sqrt(D * q * (1 - q)) + 1e-9
    assert abs(n - D * q) <= 5 * sd + 1


def test_qbsm_hand_worked():
    g = golden("qbsm_worked.json")
    s = np.array(g["spikes"], np.uint8)
    w = np.array(g["wT"], np.int8)
    acc = oracle.qbsm(s, w)
    assert acc.tolist() == g["acc"]
    rows, sops = oracle.qbsm_counts(s, w.shape[1])
    assert rows == g["rows_fetched"] and sops == g["sops"]
    assert oracle.pack(s)["active_idx"].tolist() == g["active_idx"]
    # integer IF on the raw sums, one token over T=3 steps
    _, spk, _ = oracle.if_epilogue(acc, 1, 3, kind=oracle.EPI_INT, theta_i=g["if_theta"])
    assert spk.tolist() == g["if_spikes"]


@pytest.mark.parametrize("BT,d_in,d_out,p", [(3, 5, 7, 0.5), (16, 256, 256, 0.2),
                                             (7, 130, 45, 0.05), (64, 96, 200, 0.5)])
def test_qbsm_matches_numpy_matmul(BT, d_in, d_out, p):
    g = np.random.default_rng(d_in)
    s = (g.random((BT, d_in)) < p).astype(np.uint8)
    w = g.integers(-127, 128, size=(d_in, d_out)).astype(np.int8)
    ref = np.matmul(s.astype(np.int64), w.astype(np.int64))
    assert np.array_equal(oracle.qbsm(s, w), ref)


def test_qbsm_identity_reproduces_rows():
    g = np.random.default_rng(2)
    w = g.integers(-127, 128, size=(9, 13)).astype(np.int8)
    acc = oracle.qbsm(np.eye(9, dtype=np.uint8), w)
    assert np.array_equal(acc, w.astype(np.int64))


def test_qbsm_linear_in_disjoint_spikes():
    g = np.random.default_rng(4)
    s = (g.random((12, 60)) < 0.4).astype(np.uint8)
    split = (g.random(s.shape) < 0.5).astype(np.uint8)
    s1, s2 = s * split, s * (1 - split)
    w = g.integers(-127, 128, size=(60, 33)).astype(np.int8)
    assert np.array_equal(oracle.qbsm(s, w), oracle.qbsm(s1, w) + oracle.qbsm(s2, w))


def test_zero_spikes_zero_work():
    # Sec. II-B: inactive neurons incur neither computation nor memory access.
    s = np.zeros((16, 256), np.uint8)
    w = np.full((256, 256), 127, np.int8)
    assert not oracle.qbsm(s, w).any()
    assert oracle.qbsm_counts(s, 256) == (0, 0)


def test_qbsm_at_matches_full():
    g = np.random.default_rng(9)
    s = (g.random((20, 70)) < 0.3).astype(np.uint8)
    w = g.integers(-127, 128, size=(70, 50)).astype(np.int8)
    full = oracle.qbsm(s, w)
    bi = g.integers(0, 20, size=40)
    oi = g.integers(0, 50, size=40)
    assert np.array_equal(oracle.qbsm_at(s, w, bi, oi), full[bi, oi])


def test_qbsm_extreme_sums_fit_int32():
    # the largest d_in of the workloads with every weight at +-127 and every spike on
    s = np.ones((2, 11008), np.uint8)
    w = np.full((11008, 3), 127, np.int8)
    w[:, 1] = -127
    acc = oracle.qbsm(s, w)
    assert acc[0, 0] == 127 * 11008 and acc[0, 1] == -127 * 11008 and acc[0, 0] < 2 ** 24


@pytest.mark.parametrize("B,T,D,sigma", [(4, 4, 512, 0.8), (1, 8, 512, 0.9), (8, 4, 256, 0.95)])
def test_counts_match_eq12_eq13(B, T, D, sigma):
    # Eq. (12): N_ops = 2 T D^2 (1 - sigma) per token; Eq. (13): rows loaded with
    # probability 1 - sigma^{BT}, so N_data = D^2 (1 - sigma^{BT}) b_W / B per token.
    g = np.random.default_rng(D + B)
    reps, ops, rows = 20, 0.0, 0.0
    for _ in range(reps):
        s = (g.random((B * T, D)) >= sigma).astype(np.uint8)
        r, sops = oracle.qbsm_counts(s, D)
        ops += 2 * sops / B
        rows += r
    ops /= reps
    rows /= reps
    n_ops = 2 * T * D * D * (1 - sigma)
    assert abs(ops - n_ops) / n_ops < 0.03
    q = 1 - sigma ** (B * T)
    sd = math.sqrt(D * q * (1 - q) / reps) + 1e-9
    assert abs(rows - D * q) <= 5 * sd + 0.5
