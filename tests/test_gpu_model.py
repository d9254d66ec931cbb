"""Parity of one spiking transformer layer and of the block-denoise generation loop
(CUDA path through the C ABI vs the CPU oracle)."""
import numpy as np
import pytest
import torch

import oracle
from bits import pack_rows, unpack_rows
from paper_2607_24841_gb300 import _lib as L
from paper_2607_24841_gb300 import api, synth
from parity_helpers import compare_layer, trace_pass
from test_gpu_parity import _block_check, dev, host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = api.Context(0)
    yield c
    c.close()


def device_weights(m):
    def lin(p):
        return (dev(p[0]), dev(p[1]))
    layers = [{n: lin(p) for n, p in lw.items()} for lw in m["layers"]]
    return dict(layers=layers, tok_emb=dev(m["tok_emb"]), pos_emb=dev(m["pos_emb"]),
                head=lin(m["head"]))


def _layer_case(ctx, desc, seed, ctx_len, p_ctx, impl=L.IMPL_AUTO):
    """One layer from IF-encoded N(0,1) currents over a Bernoulli context, compared
    per neuron (parity_helpers.compare_layer)."""
    m = synth.host_model(seed, desc)
    B, T, D = desc["B"], desc["T"], desc["D"]
    g = synth.rng(seed + 1)
    u = synth.normal_currents(g, (B, T, D))
    k, v = synth.context_spikes(seed + 2, 1, T, desc["Lmax"], D, ctx_len, p_ctx)
    model = api.Model(ctx, desc, device_weights(m))
    ctx.set_impl(impl)
    try:
        x_blk = api.if_neuron(ctx, dev(u), desc["theta"])
        ctx.sync()
        x, _, _ = oracle.if_f32(u, desc["theta"])
        x = x.reshape(B * T, D)
        _block_check(x_blk, x)
        flipped, _ = compare_layer(ctx, model, desc, 0, m["layers"][0], x,
                                   u.reshape(B * T, D), k[0], v[0], ctx_len)
    finally:
        ctx.set_impl(L.IMPL_AUTO)
    return flipped


@pytest.mark.parametrize("impl,gated", [(L.IMPL_AUTO, False), (L.IMPL_SIMT, False),
                                        (L.IMPL_AUTO, True)])
def test_layer_config1(ctx, impl, gated):
    # One layer: d_model 768, 12 heads x 64, MLP 3072, 16 masked tokens over a
    # 1024-token context, T = 4, IF threshold 1.0, N(0,1) input currents, seed 1.  The
    # gated variant runs gate and up as one paired tensor-core launch.
    desc = synth.model_desc(n_layers=1, D=768, H=12, F=3072, V=64, T=4, B=16, S=4, Lmax=1040,
                            gated=gated)
    _layer_case(ctx, desc, 1, 1024, 0.1, impl)


@pytest.mark.parametrize("gated", [False, True])
def test_layer_small(ctx, gated):
    desc = synth.model_desc(n_layers=1, D=256, H=4, F=384, V=64, T=4, B=8, S=2, Lmax=80,
                            gated=gated)
    _layer_case(ctx, desc, 7, 64, 0.2)


def _caches_equal(blk, ko, vo, D):
    return (np.array_equal(unpack_rows(host(blk.k_cache), D), ko)
            and np.array_equal(unpack_rows(host(blk.v_cache), D), vo))


def _explain(ctx, model, desc, m, tokens, ko_before, vo_before, ctx_len, commit, what):
    """A pass differed: it must trace to attention neurons that sat within the threshold
    band (checked per neuron, layer by layer, teacher-forced from the oracle)."""
    flipped = trace_pass(ctx, model, desc, m, tokens, ko_before.copy(), vo_before.copy(),
                         ctx_len, commit)
    assert flipped > 0, f"{what} differs from the oracle but no attention neuron flipped"
    return flipped


def _generate_both(ctx, desc, seed, prompt_blocks, gen_blocks, m=None):
    """Prompt commits, then gen_blocks blocks of S denoising steps and a commit, on the
    GPU (public API) and in the oracle; every pass compared exactly, a differing pass
    traced per neuron and the device state set to the oracle's to go on."""
    m = m if m is not None else synth.host_model(seed, desc)
    model = api.Model(ctx, desc, device_weights(m))
    n = synth.n_all_layers(desc)
    T, Lmax, D, B, V = desc["T"], desc["Lmax"], desc["D"], desc["B"], desc["V"]
    g = synth.rng(seed + 5)
    prompt = g.integers(0, V, size=prompt_blocks * B).astype(np.int32)
    ko = np.zeros((n, T, Lmax, D), np.uint8)
    vo = np.zeros((n, T, Lmax, D), np.uint8)
    blk = api.Block(model)
    ctx_len = 0
    traced = 0
    # prompt: commit passes over clean blocks (Eq. (2): they become x^{<b})
    for i in range(prompt_blocks):
        toks = prompt[i * B:(i + 1) * B]
        blk.tokens.copy_(dev(toks))
        blk.commit()
        kb, vb = ko.copy(), vo.copy()
        oracle.block_step(desc, m["layers"], m["tok_emb"], m["pos_emb"], m["head"], toks,
                          np.zeros(B, np.uint8), ko, vo, ctx_len, commit=True)
        ctx.sync()
        if not _caches_equal(blk, ko, vo, D):
            traced += _explain(ctx, model, desc, m, toks, kb, vb, ctx_len, True, "prompt commit")
            blk.k_cache.copy_(dev(pack_rows(ko)))
            blk.v_cache.copy_(dev(pack_rows(vo)))
        ctx_len += B
    out_tokens = []
    for _ in range(gen_blocks):
        tk = np.full(B, V, np.int32)
        mk = np.ones(B, np.uint8)
        for s in range(desc["S"]):
            logits = torch.empty(B, V, dtype=torch.float32, device="cuda")
            unm = torch.empty(B // desc["S"], dtype=torch.int32, device="cuda")
            blk.denoise_step(unmasked_out=unm, logits_out=logits)
            kb, vb, tk_in = ko.copy(), vo.copy(), tk.copy()
            tk, mk, lo, chosen = oracle.block_step(desc, m["layers"], m["tok_emb"],
                                                   m["pos_emb"], m["head"], tk, mk, ko, vo,
                                                   ctx_len)
            ctx.sync()
            same = (np.array_equal(host(logits), lo) and np.array_equal(host(unm), chosen)
                    and np.array_equal(host(blk.tokens), tk)
                    and np.array_equal(host(blk.mask), mk.astype(np.int32)))
            if not same:
                traced += _explain(ctx, model, desc, m, tk_in, kb, vb, ctx_len, False,
                                   f"denoising step {s}")
                blk.tokens.copy_(dev(tk))
                blk.mask.copy_(dev(mk.astype(np.int32)))
        assert mk.sum() == 0
        blk.commit()
        kb, vb = ko.copy(), vo.copy()
        oracle.block_step(desc, m["layers"], m["tok_emb"], m["pos_emb"], m["head"], tk, mk, ko,
                          vo, ctx_len, commit=True)
        ctx.sync()
        if not _caches_equal(blk, ko, vo, D):
            traced += _explain(ctx, model, desc, m, tk, kb, vb, ctx_len, True, "block commit")
            blk.k_cache.copy_(dev(pack_rows(ko)))
            blk.v_cache.copy_(dev(pack_rows(vo)))
        ctx_len += B
        assert blk.ctx_len == ctx_len
        out_tokens.append(tk)
    return out_tokens, traced


@pytest.mark.parametrize("gated", [False, True])
def test_generation_small_model(ctx, gated):
    # 2 layers, d_model 128, B = 8 tokens per block, S = 4 steps, T = 4.
    desc = synth.model_desc(n_layers=2, D=128, H=2, F=256, V=97, T=4, B=8, S=4, Lmax=48,
                            gated=gated)
    _generate_both(ctx, desc, 30 + gated, prompt_blocks=2, gen_blocks=2)


@pytest.mark.parametrize("gated", [False, True])
def test_generation_encoder_decoder(ctx, gated):
    # The encoder-decoder split (Sec. III-A, Eq. (5)-(6)): 3 encoder layers run on the
    # context passes, 2 decoder layers on the denoising steps, attending to their own K/V
    # projections of the encoder's output.  T = 8 (the paper's bitwise steps), B = 4, S = B.
    desc = synth.model_desc(n_layers=2, D=128, H=2, F=384, V=97, T=8, B=4, S=4, Lmax=24,
                            gated=gated, n_enc=3)
    _generate_both(ctx, desc, 50 + gated, prompt_blocks=3, gen_blocks=3)


def test_generation_ar_special_case(ctx):
    # B = 1, S = 1: one token per block, greedy autoregressive decoding (N-AR-LLM).
    desc = synth.model_desc(n_layers=2, D=64, H=2, F=96, V=50, T=4, B=1, S=1, Lmax=8)
    _generate_both(ctx, desc, 40, prompt_blocks=3, gen_blocks=3)


def test_step_argument_errors(ctx):
    desc = synth.model_desc(n_layers=1, D=64, H=2, F=96, V=50, T=4, B=4, S=2, Lmax=8)
    m = synth.host_model(3, desc)
    model = api.Model(ctx, desc, device_weights(m))
    blk = api.Block(model, ctx_len=6)  # 6 + 4 > Lmax
    with pytest.raises(L.NmdlmError) as e:
        blk.denoise_step()
    assert e.value.status == L.ERR_INVALID_ARG
    blk = api.Block(model)
    blk.denoise_step()
    blk.denoise_step()
    with pytest.raises(L.NmdlmError):  # the block has had its S steps
        blk.denoise_step()
    ctx.sync()


@pytest.mark.parametrize("force", [1, 2, 3])
@pytest.mark.parametrize("gated", [False, True])
def test_layer_split_modes(ctx, force, gated):
    # The 768-wide layer with the spiking linear's split-K forced through a cluster
    # (force 1), through L2 slots summed by the separate epilogue kernel (force 2) or in
    # the kernel (force 3); the gated variant covers the paired gate/up epilogue.
    desc = synth.model_desc(n_layers=1, D=768, H=12, F=3072, V=64, T=4, B=16, S=4, Lmax=1040,
                            gated=gated)
    ctx.debug_set(3, force)
    try:
        _layer_case(ctx, desc, 1, 1024, 0.1)
    finally:
        ctx.debug_set(3, 0)


@pytest.mark.parametrize("tile", [192, 256])
@pytest.mark.parametrize("B,gather", [(16, False), (16, True), (4, True)])
def test_layer_gate_up_tiles(ctx, tile, B, gather):
    # The paired gate/up launch at both tile widths: 96 + 96 channels (unswizzled
    # 96-channel boxes) and 128 + 128 (128-byte swizzled boxes), streaming every row or
    # gathering the active ones (debug key 8 forces the gather for every linear).
    desc = synth.model_desc(n_layers=1, D=768, H=12, F=3072, V=64, T=4, B=B, S=4, Lmax=1040,
                            gated=True)
    ctx.debug_set(6, tile)
    ctx.debug_set(8, 1 if gather else 0)
    try:
        _layer_case(ctx, desc, 3, 1024, 0.1, impl=L.IMPL_TC)
    finally:
        ctx.debug_set(6, 0)
        ctx.debug_set(8, 0)


@pytest.mark.parametrize("B", [2, 4, 8])
def test_e2d2_paper_shape_layers(ctx, B):
    # The paper's model shape (Sec. V-A): D_emb 512 (8 heads of 64), plain MLP D_hid 1536,
    # T = 8, blocks of B in {2, 4, 8} over a 256-token context; one encoder layer and one
    # decoder layer (distinct weights) compared per neuron with the oracle.
    desc = synth.model_desc(n_layers=1, D=512, H=8, F=1536, V=64, T=8, B=B, S=B, Lmax=256 + B,
                            gated=False, n_enc=1)
    m = synth.host_model(5, desc)
    model = api.Model(ctx, desc, device_weights(m))
    g = synth.rng(6)
    u = synth.normal_currents(g, (B, 8, 512))
    x, _, _ = oracle.if_f32(u, desc["theta"])
    x = x.reshape(B * 8, 512)
    k, v = synth.context_spikes(7, 2, 8, desc["Lmax"], 512, 256, 0.1)
    for layer in (0, 1):  # encoder layer, decoder layer
        compare_layer(ctx, model, desc, layer, m["layers"][layer], x, u.reshape(B * 8, 512),
                      k[layer], v[layer], 256)
