"""Parity of the bitwise ternary coding path (Sec. II-C, Eq. (7)-(8)) through the C ABI
with the CPU oracle.

Bars: V_th bit-exact (both sides take the sum of |a| exactly and round it once, so no
order of summation can move it), quantised values, spike planes and the combined
integer outputs bit-exact.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_24841_gb300 import _lib as L
from paper_2607_24841_gb300 import api, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = api.Context(0)
    yield c
    c.close()


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    return t.cpu().numpy()


def _planes(s):
    """Oracle ternary spikes [N, T, D] -> the +1 and -1 planes as rows n*T + t-1."""
    N, T, D = s.shape
    return ((s > 0).astype(np.uint8).reshape(N * T, D),
            (s < 0).astype(np.uint8).reshape(N * T, D))


@pytest.mark.parametrize("N,D,K,T", [(1, 7, 1.0, 1), (4, 300, 2.0, 6), (8, 1000, 4.0, 8),
                                     (32, 4096, 4.0, 8), (3, 33, 0.5, 24)])
def test_encode_parity(ctx, N, D, K, T):
    a = synth.activation_rows(synth.rng(N * 131 + D), N, D)
    s, ah, vth = oracle.ternary_encode(a, K, T)
    plus, minus, gah, gvth = api.ternary_encode(ctx, dev(a), K, T)
    assert np.array_equal(host(gvth), vth)
    assert np.array_equal(host(gah), ah)
    p, m = _planes(s)
    assert np.array_equal(host(plus), p)
    assert np.array_equal(host(minus), m)


def test_encode_wide_magnitudes(ctx):
    # Rows spanning 60 decades plus subnormals and exact ties: an fp64 running sum gives
    # different V_th in different orders here; the exact sum gives one.
    g = synth.rng(77)
    a = (g.standard_normal((6, 2048)) * 10.0 ** g.integers(-30, 30, (6, 2048))).astype(np.float32)
    a[4] = (g.standard_normal(2048) * 1e-39).astype(np.float32)
    a[5, :6] = [2.0 ** 53, 1.0, 2.0 ** 54, 2.0, 2.0 ** 53, 1.0]
    s, ah, vth = oracle.ternary_encode(a, 3.0, 8)
    plus, minus, gah, gvth = api.ternary_encode(ctx, dev(a), 3.0, 8)
    assert np.array_equal(host(gvth), vth)
    assert np.array_equal(host(gah), ah)
    p, m = _planes(s)
    assert np.array_equal(host(plus), p) and np.array_equal(host(minus), m)


def test_encode_degenerate_rows(ctx):
    a = synth.activation_rows(synth.rng(5), 4, 96)
    a[0] = 0.0                     # V_th = 0: nothing spikes
    a[1, 3] = np.nan               # NaN row: V_th is NaN, every value quantises to 0
    a[2, 7] = 1e30                 # far beyond 2^T - 1 steps: clamped
    a[3, 5] = np.inf               # an infinite value: V_th = +Inf, every value to 0
    s, ah, vth = oracle.ternary_encode(a, 3.0, 5)
    plus, minus, gah, gvth = api.ternary_encode(ctx, dev(a), 3.0, 5)
    assert np.array_equal(host(gvth), vth, equal_nan=True)
    assert np.array_equal(host(gah), ah)
    p, m = _planes(s)
    assert np.array_equal(host(plus), p) and np.array_equal(host(minus), m)
    assert not ah[0].any() and not ah[1].any() and ah[2, 7] == 31 and not ah[3].any()


@pytest.mark.parametrize("N,D,d_out,K,T,mode", [
    (4, 257, 96, 2.0, 6, L.MODE_AUTO),         # both planes as one 48-row block
    (8, 1024, 384, 4.0, 8, L.MODE_AUTO),       # one 128-row block of both planes
    (8, 1024, 384, 4.0, 8, L.MODE_SPARSE),
    (16, 1024, 384, 4.0, 8, L.MODE_AUTO),      # 128 rows per plane: two launches
    (16, 1024, 384, 4.0, 8, L.MODE_SPARSE),
    (32, 4096, 512, 4.0, 8, L.MODE_AUTO),      # 256 spike rows
    (2, 300, 48, 0.5, 3, L.MODE_DENSE),
])
def test_ternary_linear_parity(ctx, N, D, d_out, K, T, mode):
    a, w = synth.ternary_case(N * 17 + D + d_out, N, D, d_out)
    s, ah, vth = oracle.ternary_encode(a, K, T)
    _, y = oracle.ternary_linear(s, w)
    out = api.ternary_linear(ctx, dev(a), dev(w), K, T, mode=mode, want_ahat=True)
    assert np.array_equal(host(out["vth"]), vth)
    assert np.array_equal(host(out["ahat"]), ah)
    assert np.array_equal(host(out["y"]).astype(np.int64), y)


def test_combine_parity(ctx):
    g = synth.rng(9)
    N, T, d_out = 5, 7, 130
    accp = g.integers(-50000, 50000, (N * T, d_out)).astype(np.int32)
    accm = g.integers(-50000, 50000, (N * T, d_out)).astype(np.int32)
    want = ((accp.astype(np.int64) - accm).reshape(N, T, d_out) *
            (1 << np.arange(T))[None, :, None]).sum(1)
    y = api.ternary_combine(ctx, dev(accp), dev(accm), N, T)
    assert np.array_equal(host(y).astype(np.int64), want)


def test_ternary_argument_errors(ctx):
    a = torch.zeros(64, 8, dtype=torch.float32, device="cuda")
    w = torch.zeros(8, 16, dtype=torch.int8, device="cuda")
    with pytest.raises(L.NmdlmError) as e:
        api.ternary_linear(ctx, a, w, 2.0, 8)          # 64 * 8 spike rows > 256
    assert e.value.status == L.ERR_UNSUPPORTED
    huge = torch.zeros(100000, 8, dtype=torch.float32, device="cuda")
    with pytest.raises(L.NmdlmError) as e:
        api.ternary_linear(ctx, huge, w, 2.0, 8)       # N * T would overflow without the check
    assert e.value.status == L.ERR_UNSUPPORTED
    with pytest.raises(L.NmdlmError) as e:
        api.ternary_linear(ctx, a[:2], w, 0.0, 4)      # K must be > 0
    assert e.value.status == L.ERR_INVALID_ARG
    big = torch.zeros(1, 70000, dtype=torch.float32, device="cuda")
    wb = torch.zeros(70000, 16, dtype=torch.int8, device="cuda")
    with pytest.raises(L.NmdlmError) as e:
        api.ternary_linear(ctx, big, wb, 2.0, 8)       # 127 * 255 * 70000 >= 2^31
    assert e.value.status == L.ERR_UNSUPPORTED
    ctx.sync()


@pytest.mark.parametrize("N,d_out,T,theta", [(3, 70, 1, 1), (5, 130, 6, 1), (4, 257, 10, 3),
                                             (2, 33, 24, 1), (6, 64, 8, 1000)])
def test_ternary_if_parity(ctx, N, d_out, T, theta):
    # The modified IF (Sec. II-C, Eq. (9)-(10) as read) against the oracle: random inputs
    # over the full range the T steps can emit and beyond it (saturation), plus the
    # exact thresholds +-2^{t-1} theta, their neighbours and zero.
    g = synth.rng(N * 31 + T + theta)
    span = min(2 ** 31 - 1, 2 * theta * (2 ** T - 1) + 7)
    y = g.integers(-span, span + 1, (N, d_out)).astype(np.int64)
    edge = []
    for t in range(1, T + 1):
        thr = theta << (t - 1)
        edge += [thr, -thr, thr - 1, -(thr - 1), thr + 1, -(thr + 1)]
    edge += [0, theta * (2 ** T - 1), -theta * (2 ** T - 1)]
    edge = np.array([e for e in edge if abs(e) < 2 ** 31], np.int64)
    flat = y.reshape(-1)
    flat[:min(len(edge), flat.size)] = edge[:flat.size]
    s_want, v_want = oracle.ternary_if(y, T, theta)
    s, v = api.ternary_if(ctx, dev(y.astype(np.int32)), T, theta)
    assert np.array_equal(host(s), s_want)
    assert np.array_equal(host(v).astype(np.int64), v_want)


def test_ternary_if_reencodes_the_linear_output(ctx):
    # With theta 1 the modified IF re-encodes any |y| <= 2^T - 1 in Eq. (8)'s bit planes
    # exactly (sum_t 2^{t-1} s_t = y, residual 0): run it on the ternary linear's own
    # output, with T planes wide enough for the outputs that occur.
    a, w = synth.ternary_case(11, 4, 96, 40)
    out = api.ternary_linear(ctx, dev(a), dev(w), 2.0, 4)
    y = host(out["y"]).astype(np.int64)
    T = int(np.abs(y).max()).bit_length() + 1
    s, v = api.ternary_if(ctx, out["y"], T, 1)
    s = host(s).astype(np.int64)
    assert np.array_equal((s * (1 << np.arange(T))[None, :, None]).sum(1), y)
    assert not host(v).any()
