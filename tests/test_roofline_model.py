"""Pins of the roofline / energy model (Sec. IV, Eq. (12)-(16), Table I) against values
worked from the equations by hand and the regimes the paper states (no GPU)."""
import math

import pytest

from paper_2607_24841_gb300 import roofline as R


def test_eq12_eq13_by_hand():
    # D = 4, T = 2, sigma = 0.5, B = 2, b_W = 16:
    # N_ops = 2 * 2 * 16 * 0.5 = 32; N_data = 16 * (1 - 0.5^4) * 16 / 2 = 16 * 0.9375 * 8 = 120
    l = R.Linear(4, 4, 2, 2, 0.5)
    assert R.n_ops(l) == 32.0
    assert R.n_data(l, 16) == 120.0


def test_ar_and_mdlm_special_cases():
    # Sec. IV-A: the AR model is B = 1, sigma = 0; an MDLM sigma = 0 with B >= 1
    l = R.Linear(512, 512, 8, 8, 0.7)
    ar = R.autoregressive([l])[0]
    assert R.n_ops(ar) == 2 * 8 * 512 * 512 and R.n_data(ar, 16) == 512 * 512 * 16
    md = R.dense([l])[0]
    assert R.n_data(md, 16) == 512 * 512 * 16 / 8  # every row, amortised over B tokens


def test_latency_max_of_the_two_bounds():
    p = R.Platform("toy", 100.0, 1000.0, 0.0, 0.0)
    l = R.Linear(2, 2, 1, 1, 0.0)      # N_ops = 8, N_data = 4 b_W
    assert R.token_latency(l, p, 8) == max(8 / 100.0, 32 / 1000.0)
    assert R.bound(l, p, 8) == "compute"
    assert R.bound(l, p, 1000) == "memory"


def test_regimes_the_paper_states():
    # compute-bound: latency falls linearly with sigma whatever B is
    p = R.Platform("slow compute", 1e9, 1e18, 0.0, 0.0)
    for B in (1, 4, 16):
        t0 = R.token_latency(R.Linear(64, 64, B, 8, 0.0), p, 16)
        t = R.token_latency(R.Linear(64, 64, B, 8, 0.75), p, 16)
        assert t == pytest.approx(0.25 * t0)
    # memory-bound: the effective data sparsity is sigma^{BT}, so a larger block keeps
    # less of the benefit
    p = R.Platform("slow memory", 1e18, 1e6, 0.0, 0.0)
    gain = [R.token_latency(R.Linear(64, 64, B, 2, 0.0), p, 16) /
            R.token_latency(R.Linear(64, 64, B, 2, 0.9), p, 16) for B in (1, 2, 4)]
    assert gain[0] == pytest.approx(1 / (1 - 0.9 ** 2))
    assert gain[0] > gain[1] > gain[2] > 1.0


def test_eq15_eq16_encoder_once_decoder_per_step():
    p = R.Platform("toy", 1e3, 1e3, 2.0, 3.0)
    enc = R.Linear(1, 1, 1, 1, 0.0, "enc")   # N_ops = 2, N_data = b_W = 1
    dec = R.Linear(1, 1, 1, 1, 0.0, "dec")
    # TL = max(2/1e3, 1/1e3) = 2e-3 each; S = 3: 2e-3 + 3 * 2e-3 = 8e-3 s/token
    assert R.e2e_throughput([enc, dec], p, 1, 3) == pytest.approx(125.0)
    # energy: (2*2 + 1*3) * (1 + 3) = 28 J/token
    assert R.energy_per_token([enc, dec], p, 1, 3) == pytest.approx(28.0)


def test_measured_rows_replace_the_iid_fraction():
    l = R.Linear(100, 10, 4, 4, 0.9, rows_frac=0.5)
    assert R.n_data(l, 8) == pytest.approx(100 * 10 * (1 - 0.9 ** 16) * 8 / 4)
    assert R.n_data(l, 8, measured_rows=True) == pytest.approx(100 * 10 * 0.5 * 8 / 4)


def test_table_one_parameters():
    assert R.OCMS.l_ops == 300e12 and R.OCMS.l_data == 8e12
    assert R.ICMS.l_ops == 20e12 and R.ICMS.l_data == 30e12
    assert R.OCMS.e_data == 10e-12 and R.ICMS.e_data == 0.5e-12
    g = R.gb300(1919.5, 6798.9)
    assert g.l_data == pytest.approx(6798.9e9 * 8) and math.isclose(g.l_ops, 1.9195e15)
