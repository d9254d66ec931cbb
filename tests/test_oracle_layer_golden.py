"""Pin of the oracle's layer and step composition against a layer worked by hand
(tests/golden/layer_worked.json; no GPU).

Each building block of the layer has its own pins; this one checks how they are put
together (Fig. 1, Sec. III-A): which projection feeds which IF, where the block's K/V
land, that the block attends to the context and to itself, where the residual current
enters, and how the gate acts.  The expected spikes and currents are the file's, worked
out by hand; only the attention currents at t = 1 involve an exponential, written as
the closed form the file states.
"""
import math

import numpy as np
import pytest

import oracle
from conftest import golden

G = golden("layer_worked.json")
SH = G["shape"]
D, F, T, B, V, CTX, LMAX = SH["D"], SH["F"], SH["T"], SH["B"], SH["V"], SH["ctx"], SH["Lmax"]


def _w(entries, d_in=32, d_out=32):
    w = np.zeros((d_in, d_out), np.int8)
    for d, o, v in entries:
        w[d, o] = v
    return w


def _layer_weights():
    half = np.full(32, 0.5, np.float32)
    ident = _w([(d, d, 2) for d in range(32)])
    shift1 = _w([(d, (d + 1) % 32, 2) for d in range(32)])
    shift2 = _w([(d, (d + 2) % 32, 2) for d in range(32)])
    up = _w([(d, d, 2) for d in range(32)] + [(d, d + 1, 2) for d in range(31)])
    return {"q": (ident, half), "k": (shift1, half), "v": (shift2, half), "o": (ident, half),
            "gate": (ident, half), "up": (up, half), "down": (ident, half)}


def _rows(chan_lists, n=32):
    """[[channels at t1], [channels at t2]] -> uint8 [T, n]."""
    a = np.zeros((len(chan_lists), n), np.uint8)
    for t, chans in enumerate(chan_lists):
        a[t, chans] = 1
    return a


def _cur(dicts, n=32):
    a = np.zeros((len(dicts), n), np.float32)
    for t, d in enumerate(dicts):
        for c, v in d.items():
            a[t, int(c)] = v
    return a


def _desc(gated):
    return dict(n_layers=1, D=D, H=SH["H"], dh=SH["dh"], F=F, gated=int(gated), V=V, T=T, B=B,
                S=SH["S"], Lmax=LMAX, theta=SH["theta"])


def _context_caches():
    k = np.zeros((T, LMAX, D), np.uint8)
    v = np.zeros((T, LMAX, D), np.uint8)
    for t in range(T):
        for j in range(CTX):
            k[t, j, G["context"]["k"][t][j]] = 1
            v[t, j, G["context"]["v"][t][j]] = 1
    return k, v


def _u0():
    u = np.zeros(32, np.float32)
    for c, val in G["expected"]["u0"].items():
        u[int(c)] = val
    return np.stack([u, u])  # constant over T


def test_golden_inputs_are_consistent():
    # u0 = tok_emb[mask] + pos_emb[ctx], and x = IF(u0)
    e = G["embedding"]
    u = np.zeros(32, np.float32)
    for c, val in e["tok_emb_mask"].items():
        u[int(c)] += val
    for c, val in e["pos_emb_3"].items():
        u[int(c)] += val
    assert np.array_equal(np.stack([u, u]), _u0())
    x, _, _ = oracle.if_f32(_u0().reshape(1, T, D), SH["theta"])
    assert np.array_equal(x.reshape(T, D), _rows(G["expected"]["x"]))


@pytest.mark.parametrize("gated", [True, False])
def test_layer_composition_worked_by_hand(gated):
    ex = G["expected"]
    x = _rows(ex["x"])
    k, v = _context_caches()
    x_out, u_out, tr = oracle.layer(_desc(gated), _layer_weights(), x, _u0(), k, v, CTX)
    # Q from its own projection and IF
    assert np.array_equal(tr["q"], _rows(ex["q"]))
    # the block's K and V at cache position ctx, every earlier position untouched
    assert np.array_equal(k[:, CTX, :], _rows(ex["k_block"]))
    assert np.array_equal(v[:, CTX, :], _rows(ex["v_block"]))
    k0, v0 = _context_caches()
    assert np.array_equal(k[:, :CTX], k0[:, :CTX]) and np.array_equal(v[:, :CTX], v0[:, :CTX])
    # attention over the three context keys and the block's own key
    a = 1.0 / math.sqrt(SH["dh"])
    z = math.exp(a) + 3.0
    p0, p1 = math.exp(a) / z, 1.0 / z
    want = np.zeros((T, D), np.float64)
    want[0, 7], want[0, 8], want[0, 30], want[0, 2] = p0 + p1, p1, p1, p1
    for c, val in ex["attn_current"]["t2"].items():
        want[1, int(c)] = float(val)
    np.testing.assert_allclose(tr["attn_cur"], want, rtol=1e-6, atol=1e-7)
    assert np.array_equal(tr["attn"], _rows(ex["attn"]))
    # output projection: residual added before the IF
    assert np.array_equal(tr["u1"], _cur(ex["u1"]))
    assert np.array_equal(tr["x1"], _rows(ex["x1"]))
    part = ex["gated"] if gated else ex["plain"]
    if gated:
        assert np.array_equal(tr["g"], _rows(part["g"]))
    assert np.array_equal(tr["h"], _rows(part["h"]))
    assert np.array_equal(u_out, _cur(part["u_out"]))
    assert np.array_equal(x_out, _rows(part["x_out"]))


def test_denoising_step_worked_by_hand():
    ex = G["expected"]
    e = G["embedding"]
    tok_emb = np.zeros((V + 1, D), np.float32)
    for c, val in e["tok_emb_mask"].items():
        tok_emb[V, int(c)] = val
    pos_emb = np.zeros((LMAX, D), np.float32)
    for c, val in e["pos_emb_3"].items():
        pos_emb[CTX, int(c)] = val
    head = (_w(G["weights"]["head"], 32, V), np.full(V, 0.5, np.float32))
    k, v = _context_caches()
    k, v = k[None].copy(), v[None].copy()  # one layer
    tokens = np.full(B, V, np.int32)  # the mask id
    mask = np.ones(B, np.uint8)
    tk, mk, logits, chosen = oracle.block_step(_desc(True), [_layer_weights()], tok_emb,
                                               pos_emb, head, tokens, mask, k, v, CTX)
    assert np.array_equal(logits, np.array([ex["step_gated"]["logits"]], np.float32))
    assert tk.tolist() == [ex["step_gated"]["token"]] and mk.tolist() == [0]
    assert chosen.tolist() == ex["step_gated"]["chosen"]
    # the step wrote the block's K/V (the same as in the layer worked above)
    assert np.array_equal(k[0, :, CTX, :], _rows(ex["k_block"]))
    assert np.array_equal(v[0, :, CTX, :], _rows(ex["v_block"]))


def test_encoder_decoder_context_pass_worked_by_hand():
    # Eq. (5)-(6): one encoder layer (the layer above, gated) and one decoder layer whose K
    # and V weights shift by one and by two channels.  The context pass over the block
    # writes the encoder's own block K/V into the encoder cache, and the decoder's K/V
    # projections of h, the encoder's output (x_out above: t1 {0}, t2 {0, 1, 2, 7}), into
    # the decoder cache: K = h shifted by one, V = h shifted by two.  A denoising step then
    # leaves the encoder cache alone.
    ex = G["expected"]
    desc = dict(_desc(True), n_enc=1)
    e = G["embedding"]
    tok_emb = np.zeros((V + 1, D), np.float32)
    for c, val in e["tok_emb_mask"].items():
        tok_emb[V, int(c)] = val
    pos_emb = np.zeros((LMAX, D), np.float32)
    for c, val in e["pos_emb_3"].items():
        pos_emb[CTX, int(c)] = val
    head = (_w(G["weights"]["head"], 32, V), np.full(V, 0.5, np.float32))
    k1, v1 = _context_caches()
    k = np.stack([k1, np.zeros_like(k1)])
    v = np.stack([v1, np.zeros_like(v1)])
    tokens = np.full(B, V, np.int32)  # the block re-embedded like the step above
    oracle.block_step(desc, [_layer_weights(), _layer_weights()], tok_emb, pos_emb, head,
                      tokens, np.zeros(B, np.uint8), k, v, CTX, commit=True)
    assert np.array_equal(k[0, :, CTX, :], _rows(ex["k_block"]))   # encoder: its own K
    assert np.array_equal(v[0, :, CTX, :], _rows(ex["v_block"]))
    h = ex["gated"]["x_out"]
    assert np.array_equal(k[1, :, CTX, :], _rows([[(c + 1) % 32 for c in row] for row in h]))
    assert np.array_equal(v[1, :, CTX, :], _rows([[(c + 2) % 32 for c in row] for row in h]))
    assert not k[1, :, :CTX].any() and not v[1, :, :CTX].any()
    k_enc = k[0].copy()
    oracle.block_step(desc, [_layer_weights(), _layer_weights()], tok_emb, pos_emb, head,
                      np.full(B, V, np.int32), np.ones(B, np.uint8), k, v, CTX)
    assert np.array_equal(k[0], k_enc)
