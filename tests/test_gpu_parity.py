"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Bars: integer sums, packed spikes, active sets and indices bit-exact; fp32 currents and
attention outputs within rtol 1e-3 (abs 1e-6 near zero); spikes decided on currents
that went through exp/softmax may differ only where the oracle's membrane came within
MARGIN of the threshold (both sides decide in fp32, the exp implementations differ).
"""
import numpy as np
import pytest
import torch

import oracle
from bits import pack_rows, unpack_rows
from paper_2607_24841_gb300 import _lib as L
from paper_2607_24841_gb300 import api, synth
from parity_helpers import check_block

pytestmark = pytest.mark.gpu

RTOL, ATOL = 1e-3, 1e-6
MARGIN = 1e-5


@pytest.fixture(scope="module")
def ctx():
    c = api.Context(0)
    yield c
    c.close()


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    return t.cpu().numpy()


def _block_check(blk, spikes_u8, check_idx=False):
    r = oracle.pack(spikes_u8)
    BT, D = spikes_u8.shape
    assert np.array_equal(unpack_rows(host(blk.row_bits), D), spikes_u8)
    assert np.array_equal(host(blk.row_bits).view(np.uint32), r["row_bits"])
    if blk.col_masks is not None:
        assert np.array_equal(host(blk.col_masks).view(np.uint32), r["col_masks"])
    if blk.active_mask is not None:
        assert np.array_equal(host(blk.active_mask).view(np.uint32), r["active_mask"])
    if check_idx:
        n = int(host(blk.n_active)[0])
        assert n == r["n_active"]
        assert np.array_equal(host(blk.active_idx)[:n], r["active_idx"])


# ------------------------------------------------------------------ packing
@pytest.mark.parametrize("BT,D,p", [(16, 256, 0.2), (5, 77, 0.1), (128, 300, 0.02),
                                    (256, 4096, 0.05), (1, 1, 1.0), (33, 100, 0.0),
                                    (64, 11008, 0.01)])
def test_pack_parity(ctx, BT, D, p):
    s = synth.bernoulli_spikes(synth.rng(BT + D), (BT, D), p)
    blk = api.pack_spikes(ctx, dev(s), T=1)
    ctx.sync()
    _block_check(blk, s, check_idx=True)


def test_pack_rejects_non_binary(ctx):
    s = np.zeros((4, 64), np.uint8)
    s[2, 5] = 2
    api.pack_spikes(ctx, dev(s), T=1)
    assert ctx.sync_status() == L.ERR_INVALID_ARG
    ctx.sync()  # cleared


# ------------------------------------------------------------------------ IF
@pytest.mark.parametrize("B,T,N", [(4, 4, 256), (3, 1, 77), (32, 4, 4096), (2, 32, 40)])
def test_if_neuron_int_parity(ctx, B, T, N):
    g = synth.rng(B * 100 + T)
    cur = g.integers(-150, 200, size=(B, T, N)).astype(np.int32)
    blk = api.if_neuron(ctx, dev(cur), 64)
    ctx.sync()
    s, _ = oracle.if_int(cur.astype(np.int64), 64)
    _block_check(blk, s.reshape(B * T, N))


@pytest.mark.parametrize("B,T,N", [(16, 4, 768), (1, 8, 33), (32, 4, 4096)])
def test_if_neuron_f32_parity(ctx, B, T, N):
    g = synth.rng(B + T + N)
    cur = synth.normal_currents(g, (B, T, N))
    blk = api.if_neuron(ctx, dev(cur), 1.0)
    ctx.sync()
    s, _, _ = oracle.if_f32(cur, 1.0)
    _block_check(blk, s.reshape(B * T, N))


def test_if_neuron_state_carries_over(ctx):
    # Running T1 steps and then T2 steps with the carried membrane equals T1+T2 steps.
    g = synth.rng(5)
    B, N = 3, 96
    cur = synth.normal_currents(g, (B, 6, N))
    v = torch.zeros(B, N, dtype=torch.float32, device="cuda")
    b1 = api.if_neuron(ctx, dev(cur[:, :2]), 1.0, v_state=v)
    b2 = api.if_neuron(ctx, dev(cur[:, 2:]), 1.0, v_state=v)
    ctx.sync()
    s, vfin, _ = oracle.if_f32(cur, 1.0)
    got = np.concatenate([unpack_rows(host(b1.row_bits), N).reshape(B, 2, N),
                          unpack_rows(host(b2.row_bits), N).reshape(B, 4, N)], axis=1)
    assert np.array_equal(got, s)
    assert np.array_equal(host(v), vfin)


# -------------------------------------------------------------------- linear
def _linear_case(BT, T, d_in, d_out, p, seed, weights="uniform"):
    s, w, sc = synth.linear_case(seed, BT, d_in, d_out, p, weights)
    return s, w, sc


def _run_linear(ctx, s, w, sc, T, impl, mode, kind=L.IF_INT, thr=64, residual=None,
                gate_bits=None):
    ctx.set_impl(impl)
    blk = api.pack_spikes(ctx, dev(s), T)
    stats = torch.zeros(2, dtype=torch.int64, device="cuda")
    out = api.spike_linear(ctx, blk, dev(w), dev(sc), mode=mode, want_acc=True, kind=kind,
                           threshold=thr, residual=None if residual is None else dev(residual),
                           gate_bits=gate_bits, want_current=True, stats=stats)
    ctx.sync()
    ctx.set_impl(L.IMPL_AUTO)
    return out, host(stats)


IMPLS = [L.IMPL_SIMT, L.IMPL_TC]
MODES = [L.MODE_SPARSE, L.MODE_DENSE]


@pytest.mark.parametrize("impl", IMPLS)
@pytest.mark.parametrize("mode", MODES)
def test_linear_config0(ctx, impl, mode):
    # d_in = d_out = 256, 4 tokens x T=4, Bernoulli(0.2), uniform int8, U(0.001, 0.01)
    # scales, integer IF threshold 64, seed 0.
    B, T = 4, 4
    s, w, sc = _linear_case(B * T, T, 256, 256, 0.2, 0)
    out, stats = _run_linear(ctx, s, w, sc, T, impl, mode)
    acc = oracle.qbsm(s, w)
    assert np.array_equal(host(out["acc"]), acc)
    cur, spk, _ = oracle.if_epilogue(acc, B, T, scale=sc, kind=oracle.EPI_INT, theta_i=64)
    _block_check(out["block"], spk)
    assert np.array_equal(host(out["current"]), cur)
    rows, sops = oracle.qbsm_counts(s, 256)
    assert stats[1] == sops
    assert stats[0] == (256 if mode == L.MODE_DENSE else rows)


LIN_SHAPES = [
    # BT, T, d_in, d_out, p
    (1, 1, 64, 64, 0.5),
    (4, 4, 77, 48, 0.3),
    (16, 4, 300, 128, 0.1),
    (16, 1, 130, 256, 0.0),
    (32, 4, 256, 384, 1.0),
    (64, 4, 1000, 256, 0.05),
    (128, 4, 700, 128, 0.1),
    (128, 32, 96, 144, 0.2),
    (200, 8, 256, 128, 0.1),
    (256, 4, 512, 256, 0.02),
]


@pytest.mark.parametrize("impl", IMPLS)
@pytest.mark.parametrize("BT,T,d_in,d_out,p", LIN_SHAPES)
def test_linear_shapes(ctx, impl, BT, T, d_in, d_out, p):
    s, w, sc = _linear_case(BT, T, d_in, d_out, p, BT * 7 + d_in)
    out, stats = _run_linear(ctx, s, w, sc, T, impl, L.MODE_AUTO)
    acc = oracle.qbsm(s, w)
    assert np.array_equal(host(out["acc"]), acc)
    _, spk, _ = oracle.if_epilogue(acc, BT // T, T, scale=sc, kind=oracle.EPI_INT, theta_i=64)
    _block_check(out["block"], spk)


def test_linear_ragged_d_out_uses_cuda_cores(ctx):
    s, w, sc = _linear_case(16, 4, 100, 45, 0.3, 3)
    out, _ = _run_linear(ctx, s, w, sc, 4, L.IMPL_AUTO, L.MODE_AUTO)
    assert np.array_equal(host(out["acc"]), oracle.qbsm(s, w))
    with pytest.raises(L.NmdlmError):
        _run_linear(ctx, s, w, sc, 4, L.IMPL_TC, L.MODE_AUTO)


@pytest.mark.parametrize("impl", IMPLS)
def test_linear_fp32_residual_and_gate(ctx, impl):
    B, T, d_in, d_out = 8, 4, 384, 256
    s, w, sc = _linear_case(B * T, T, d_in, d_out, 0.15, 11, weights="gaussian")
    g = synth.rng(12)
    res = synth.normal_currents(g, (B * T, d_out))
    gate = synth.bernoulli_spikes(g, (B * T, d_out), 0.5)
    acc = oracle.qbsm(s, w)
    out, _ = _run_linear(ctx, s, w, sc, T, impl, L.MODE_AUTO, kind=L.IF_FP32, thr=1.0,
                         residual=res)
    cur, spk, _ = oracle.if_epilogue(acc, B, T, scale=sc, residual=res, theta_f=1.0)
    assert np.array_equal(host(out["current"]), cur)
    _block_check(out["block"], spk)
    out, _ = _run_linear(ctx, s, w, sc, T, impl, L.MODE_AUTO, kind=L.IF_FP32, thr=1.0,
                         gate_bits=dev(pack_rows(gate)))
    cur, spk, _ = oracle.if_epilogue(acc, B, T, scale=sc, gate=gate, theta_f=1.0)
    assert np.array_equal(host(out["current"]), cur)
    _block_check(out["block"], spk)


# ----------------------------------------------------------------- attention
def _attn_case(seed, B, T, L_ctx, H, dh, p_q, p_kv):
    g = synth.rng(seed)
    D = H * dh
    Lk = L_ctx + B
    q = synth.bernoulli_spikes(g, (B * T, D), p_q)
    k = synth.bernoulli_spikes(g, (T, Lk, D), p_kv)
    v = synth.bernoulli_spikes(g, (T, Lk, D), p_kv)
    return q, k, v


def _spikes_with_margin(got, want, margin, B, T, D, theta):
    """Spikes equal except at (token, channel) neurons whose oracle membrane came
    within MARGIN*max(1, theta) of the threshold; returns the number exempted."""
    bad = (got.reshape(B, T, D) != want.reshape(B, T, D)).any(axis=1)
    near = margin < MARGIN * max(1.0, theta)
    assert not np.any(bad & ~near), "spike mismatch away from the threshold"
    return int(bad.sum())


@pytest.mark.parametrize("B,T,L_ctx,H,dh,p", [(16, 4, 1024, 12, 64, 0.1),
                                              (8, 4, 100, 2, 32, 0.3),
                                              (32, 4, 2048, 4, 128, 0.1),
                                              (1, 1, 0, 1, 32, 0.5),
                                              (5, 2, 37, 3, 96, 0.2),
                                              (4, 2, 50, 1, 192, 0.2),
                                              (1, 4, 0, 2, 32, 0.5),
                                              (1, 4, 2, 2, 32, 0.5),
                                              (2, 4, 5, 2, 32, 0.5),
                                              (64, 4, 300, 2, 64, 0.15),
                                              (65, 2, 40, 2, 64, 0.15),
                                              # d_head 128, short contexts: three stages
                                              (3, 1, 0, 1, 128, 0.5),
                                              (33, 2, 200, 2, 128, 0.3),
                                              (8, 2, 120, 1, 128, 0.9),
                                              (40, 3, 600, 2, 128, 0.05),
                                              # long contexts
                                              (4, 1, 2996, 1, 128, 0.1),
                                              (4, 1, 4496, 1, 128, 0.1),
                                              # T 4 and 8 with partial and full token
                                              # tiles (column masks across words)
                                              (20, 4, 300, 2, 128, 0.2),
                                              (8, 8, 100, 2, 128, 0.3),
                                              (32, 8, 500, 1, 128, 0.1)])
def test_attention_parity(ctx, B, T, L_ctx, H, dh, p):
    q, k, v = _attn_case(B * 31 + L_ctx, B, T, L_ctx, H, dh, p, p)
    D = H * dh
    cur, blk = api.spike_attention(ctx, dev(pack_rows(q)), dev(pack_rows(k)), dev(pack_rows(v)),
                                   T, B, L_ctx + B, H, dh, theta=0.05)
    ctx.sync()
    want = oracle.attention(q, k, v, B, T, H, dh)
    np.testing.assert_allclose(host(cur), want, rtol=RTOL, atol=ATOL)
    s, _, m = oracle.if_f32(want.reshape(B, T, D), 0.05)
    got = unpack_rows(host(blk.row_bits), D)
    _spikes_with_margin(got, s.reshape(B * T, D), m, B, T, D, 0.05)
    # the column masks and active mask written with the row bits agree with them
    check_block(blk, got)


def test_attention_rejects_bad_head_width(ctx):
    q = torch.zeros(4, 1, dtype=torch.int32, device="cuda")
    with pytest.raises(L.NmdlmError) as e:
        api.spike_attention(ctx, q, torch.zeros(1, 4, 1, dtype=torch.int32, device="cuda"),
                            torch.zeros(1, 4, 1, dtype=torch.int32, device="cuda"), 1, 4, 4, 1,
                            16)
    assert e.value.status == L.ERR_UNSUPPORTED


# ----------------------------------------------------------- failure paths
def test_bounded_wait_times_out_and_context_survives(ctx):
    ctx.debug_wait_test(2_000_000)  # 2 ms
    assert ctx.sync_status() == L.ERR_TIMEOUT
    ctx.sync()
    test_linear_config0(ctx, L.IMPL_TC, L.MODE_SPARSE)


# Split-K of the spiking linear, three ways: through distributed shared memory inside a
# thread-block cluster (IF epilogue in the kernel); through per-split L2 slots summed by
# the separate IF-epilogue kernel; and through L2 slots that the tile's splits sum in the
# kernel, each its own slice, after meeting at a counter.  Debug key 3 forces one mode
# (1, 2, 3) and prefers splitting.
SPLIT_SHAPES = [
    # BT, T, d_in, d_out, p
    (128, 4, 1000, 384, 0.1),
    (64, 8, 2048, 256, 0.05),
    (32, 4, 777, 528, 0.2),
    (16, 4, 4096, 512, 0.005),   # sparse: only the active rows are gathered
]


@pytest.mark.parametrize("force", [1, 2, 3])
@pytest.mark.parametrize("BT,T,d_in,d_out,p", SPLIT_SHAPES)
def test_linear_split_modes(ctx, force, BT, T, d_in, d_out, p):
    s, w, sc = _linear_case(BT, T, d_in, d_out, p, BT * 5 + d_in + force)
    acc = oracle.qbsm(s, w)
    ctx.debug_set(3, force)
    try:
        out, _ = _run_linear(ctx, s, w, sc, T, L.IMPL_AUTO, L.MODE_AUTO)
        assert np.array_equal(host(out["acc"]), acc)
        _, spk, _ = oracle.if_epilogue(acc, BT // T, T, scale=sc, kind=oracle.EPI_INT, theta_i=64)
        _block_check(out["block"], spk)
        g = synth.rng(BT + d_out)
        res = synth.normal_currents(g, (BT, d_out))
        gate = synth.bernoulli_spikes(g, (BT, d_out), 0.5)
        out, _ = _run_linear(ctx, s, w, sc, T, L.IMPL_AUTO, L.MODE_AUTO, kind=L.IF_FP32,
                             thr=1.0, residual=res)
        cur, spk, _ = oracle.if_epilogue(acc, BT // T, T, scale=sc, residual=res, theta_f=1.0)
        assert np.array_equal(host(out["current"]), cur)
        _block_check(out["block"], spk)
        out, _ = _run_linear(ctx, s, w, sc, T, L.IMPL_AUTO, L.MODE_AUTO, kind=L.IF_FP32,
                             thr=1.0, gate_bits=dev(pack_rows(gate)))
        cur, spk, _ = oracle.if_epilogue(acc, BT // T, T, scale=sc, gate=gate, theta_f=1.0)
        assert np.array_equal(host(out["current"]), cur)
        _block_check(out["block"], spk)
    finally:
        ctx.debug_set(3, 0)
