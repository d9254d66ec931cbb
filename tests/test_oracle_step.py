"""Pins of the oracle's head, unmasking, embedding and block-denoise step
(Sec. III-A, Eq. (2) and (6)); the layer composition itself is parity-unpinned and
checked here only for the invariants it must keep."""
import numpy as np
import pytest

import oracle
from conftest import golden
from paper_2607_24841_gb300 import synth


def test_head_hand_worked():
    g = golden("head_unmask_worked.json")["head"]
    x = np.array(g["x"], np.uint8)
    lg = oracle.head(x, np.array(g["wT"], np.int8), np.array(g["scale"], np.float32), 1, 2)
    assert lg.tolist() == g["logits"]


def test_unmask_hand_worked():
    g = golden("head_unmask_worked.json")["unmask"]
    lg = np.array(g["logits"], np.float32)
    tk = np.array(g["initial_tokens"], np.int32)
    mk = np.ones(4, np.uint8)
    tk, mk, conf, tok, chosen = oracle.unmask(lg, 2, tk, mk)
    assert np.allclose(conf, g["conf"], rtol=1e-8)
    assert tok.tolist() == g["tok"]
    assert chosen.tolist() == g["step1_chosen"]
    assert tk.tolist() == g["step1_tokens"] and mk.tolist() == g["step1_mask"]
    tk, mk, _, _, chosen = oracle.unmask(lg, 2, tk, mk)
    assert chosen.tolist() == g["step2_chosen"]
    assert tk.tolist() == g["step2_tokens"] and mk.tolist() == g["step2_mask"]


def test_unmask_softmax_confidence_matches_scipy():
    from scipy.special import softmax
    g = np.random.default_rng(0)
    lg = g.standard_normal((6, 50)).astype(np.float32) * 3
    _, _, conf, tok, _ = oracle.unmask(lg, 1, np.zeros(6, np.int32), np.ones(6, np.uint8))
    p = softmax(lg.astype(np.float64), axis=1)
    assert np.allclose(conf, p.max(axis=1), rtol=1e-12)
    assert np.array_equal(tok, p.argmax(axis=1))


def test_embedding_current_is_constant_over_t_and_rate_coded():
    D, T, V = 16, 4, 10
    tok_emb = np.zeros((V + 1, D), np.float32)
    pos_emb = np.zeros((8, D), np.float32)
    tok_emb[3, :] = np.linspace(0, 1, D, dtype=np.float32)
    u0 = oracle.embed(tok_emb, pos_emb, np.array([3], np.int32), T, 0)
    assert np.array_equal(u0, np.repeat(tok_emb[3][None, :], T, axis=0))
    # constant current c in [0, 1] with threshold 1 fires floor(T*c) times
    cur = np.array([0.0, 0.25, 0.5, 0.75, 1.0], np.float32)
    s, _, _ = oracle.if_f32(np.repeat(cur[None, None, :], T, axis=1), 1.0)
    assert s.sum(axis=1)[0].tolist() == [0, 1, 2, 3, 4]


def _tiny(B=4, S=2, gated=False, n_layers=2, ctx=6):
    desc = synth.model_desc(n_layers=n_layers, D=64, H=2, F=96, V=50, T=4, B=B, S=S,
                            Lmax=ctx + B + 3, gated=gated)
    m = synth.host_model(21, desc)
    k, v = synth.context_spikes(22, n_layers, 4, desc["Lmax"], 64, ctx, 0.2)
    return desc, m, k, v


@pytest.mark.parametrize("gated", [False, True])
def test_step_unmasks_b_over_s_and_keeps_tokens(gated):
    B, S, ctx = 4, 2, 6
    desc, m, k, v = _tiny(B, S, gated, ctx=ctx)
    V = desc["V"]
    tokens = np.full(B, V, np.int32)
    mask = np.ones(B, np.uint8)
    seen = {}
    for s in range(1, S + 1):
        tokens, mask, logits, chosen = oracle.block_step(desc, m["layers"], m["tok_emb"],
                                                         m["pos_emb"], m["head"], tokens, mask,
                                                         k, v, ctx)
        assert logits.shape == (B, V)
        assert int((mask == 0).sum()) == s * B // S
        assert chosen.size == B // S
        for b, t in seen.items():
            assert tokens[b] == t  # unmasked tokens never change
        for b in chosen:
            seen[int(b)] = int(tokens[b])
            assert 0 <= tokens[b] < V  # the mask id is never chosen
    assert mask.sum() == 0


def test_commit_writes_only_block_positions():
    B, S, ctx = 4, 2, 6
    desc, m, k, v = _tiny(B, S, ctx=ctx)
    k0, v0 = k.copy(), v.copy()
    tokens = np.arange(B, dtype=np.int32)
    oracle.block_step(desc, m["layers"], m["tok_emb"], m["pos_emb"], m["head"], tokens,
                      np.zeros(B, np.uint8), k, v, ctx, commit=True)
    assert np.array_equal(k[:, :, :ctx], k0[:, :, :ctx])
    assert np.array_equal(v[:, :, :ctx], v0[:, :, :ctx])
    # the block's K spikes equal those of the first layer computed piecewise
    x_in = None
    u0 = oracle.embed(m["tok_emb"], m["pos_emb"], tokens, 4, ctx)
    x_in, _, _ = oracle.if_f32(u0.reshape(B, 4, -1), 1.0)
    x_in = x_in.reshape(B * 4, -1)
    acc = oracle.qbsm(x_in, m["layers"][0]["k"][0])
    _, kb, _ = oracle.if_epilogue(acc, B, 4, scale=m["layers"][0]["k"][1])
    got = k[0][:, ctx:ctx + B].transpose(1, 0, 2).reshape(B * 4, -1)
    assert np.array_equal(got, kb)


def test_ar_special_case_b1_s1():
    # B = 1, S = 1 is greedy autoregressive decoding (the N-AR-LLM point of Sec. V-C):
    # the single position takes the argmax of its logits.
    desc, m, k, v = _tiny(B=1, S=1, ctx=6)
    tokens = np.full(1, desc["V"], np.int32)
    tokens2, mask, logits, chosen = oracle.block_step(desc, m["layers"], m["tok_emb"],
                                                      m["pos_emb"], m["head"], tokens,
                                                      np.ones(1, np.uint8), k, v, 6)
    assert chosen.tolist() == [0] and mask.tolist() == [0]
    assert tokens2[0] == int(np.argmax(logits[0]))


def test_layer_residual_stream_and_kv_positions():
    desc, m, k, v = _tiny(B=4, S=2, ctx=6)
    g = np.random.default_rng(8)
    B, T, D = 4, 4, 64
    u = g.standard_normal((B * T, D)).astype(np.float32)
    x, _, _ = oracle.if_f32(u.reshape(B, T, D), 1.0)
    x = x.reshape(B * T, D)
    kc, vc = k[0].copy(), v[0].copy()
    x2, u2, tr = oracle.layer(desc, m["layers"][0], x, u, kc, vc, 6)
    lw = m["layers"][0]
    # the residual stream after the output projection is u + scale_o * (A W_o^T)
    acc_o = oracle.qbsm(tr["attn"], lw["o"][0])
    u1, x1, _ = oracle.if_epilogue(acc_o, B, T, scale=lw["o"][1], residual=u)
    assert np.array_equal(u1, tr["u1"]) and np.array_equal(x1, tr["x1"])
    acc_d = oracle.qbsm(tr["h"], lw["down"][0])
    u2r, x2r, _ = oracle.if_epilogue(acc_d, B, T, scale=lw["down"][1], residual=u1)
    assert np.array_equal(u2r, u2) and np.array_equal(x2r, x2)
    # keys beyond the block stay untouched
    assert np.array_equal(kc[:, 10:], k[0][:, 10:])


def test_step_margin_is_min_attention_margin_of_the_pass():
    # A one-layer step recomputed piecewise: embedding -> IF -> layer; the margin the
    # step reports is the smallest attention membrane distance of that layer.
    B, S, ctx = 4, 2, 6
    desc, m, k, v = _tiny(B, S, n_layers=1, ctx=ctx)
    tokens = np.full(B, desc["V"], np.int32)
    kc, vc = k.copy(), v.copy()
    *_, margin = oracle.block_step(desc, m["layers"], m["tok_emb"], m["pos_emb"], m["head"],
                                   tokens, np.ones(B, np.uint8), kc, vc, ctx,
                                   return_margin=True)
    u0 = oracle.embed(m["tok_emb"], m["pos_emb"], tokens, 4, ctx)
    x, _, _ = oracle.if_f32(u0.reshape(B, 4, -1), 1.0)
    k1, v1 = k[0].copy(), v[0].copy()
    _, _, tr = oracle.layer(desc, m["layers"][0], x.reshape(B * 4, -1), u0, k1, v1, ctx)
    assert margin == tr["attn_margin"].min()
    assert 0.0 <= margin < np.inf
