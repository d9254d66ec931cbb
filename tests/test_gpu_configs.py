"""Every configuration of the workload set at its real sizes, on the GPU through the C ABI,
against the oracle.

- the spiking linear sweep (4096 -> 4096 and 4096 -> 11008 over spike densities and
  block sizes): integer sums, output spikes and the row / synaptic-operation counts
  bit-exact;
- the large decode shape (32 layers, d_model 4096, 32 x 128 heads, gated MLP 11008, vocab
  32000, block 32, T 4, 2048-token context): two sampled layers (the first and the last)
  compared per neuron in the launch configuration the benchmark times, and the
  32000-way head with the unmasking of one denoising step;
- the small model end to end (12 layers, d_model 768, vocab 32000, block 8, 8 steps, a
  128-token prompt): a stated short generation compared pass by pass.
"""
import numpy as np
import pytest
import torch

import oracle
from bits import pack_rows, unpack_rows
from paper_2607_24841_gb300 import _lib as L
from paper_2607_24841_gb300 import api, synth
from parity_helpers import check_block, compare_layer, dev, host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = api.Context(0, workspace_bytes=1 << 30)
    yield c
    c.close()


# ------------------------------------------------------------- linear sweep
SWEEP = [(4096, 4096, B, p) for B in (1, 8, 32) for p in (0.02, 0.1, 0.5)] + \
        [(4096, 11008, B, p) for B in (4, 32) for p in (0.05, 0.5)]


@pytest.mark.parametrize("d_in,d_out,B,p", SWEEP)
def test_config2_linear_sweep_point(ctx, d_in, d_out, B, p):
    # Bernoulli(p) spikes over B tokens x T = 4, uniform int8 weights, U(0.001, 0.01)
    # scales (the sweep's recipe); integer IF (threshold 64) on the raw sums.
    T = 4
    s, w, sc = synth.linear_case(int(1000 * p) + B + d_out, B * T, d_in, d_out, p)
    blk = api.pack_spikes(ctx, dev(s), T)
    stats = torch.zeros(2, dtype=torch.int64, device="cuda")
    out = api.spike_linear(ctx, blk, dev(w), dev(sc), want_acc=True, kind=L.IF_INT,
                           threshold=64, stats=stats)
    ctx.sync()
    acc = oracle.qbsm(s, w)
    assert np.array_equal(host(out["acc"]).astype(np.int64), acc)
    spikes, _ = oracle.if_int(acc.reshape(B, T, d_out), 64)
    check_block(out["block"], spikes.reshape(B * T, d_out))
    rows, sops = oracle.qbsm_counts(s, d_out)
    assert host(stats).tolist() == [rows, sops]


@pytest.mark.parametrize("mode", [L.MODE_SPARSE, L.MODE_DENSE])
def test_config2_forced_modes_at_size(ctx, mode):
    # the same sums whichever rows are streamed (row skipping or all rows)
    T, B, p = 4, 8, 0.05
    s, w, sc = synth.linear_case(77, B * T, 4096, 11008, p)
    blk = api.pack_spikes(ctx, dev(s), T)
    out = api.spike_linear(ctx, blk, dev(w), dev(sc), mode=mode, want_acc=True,
                           kind=L.IF_INT, threshold=64)
    ctx.sync()
    assert np.array_equal(host(out["acc"]).astype(np.int64), oracle.qbsm(s, w))


# ------------------------------------------------------- large decode shape
def _large_desc():
    return synth.model_desc(n_layers=32, D=4096, H=32, F=11008, V=32000, T=4, B=32, S=4,
                            Lmax=2080, gated=True)


def _host_lw(lw):
    return {n: (w.cpu().numpy(), s.cpu().numpy()) for n, (w, s) in lw.items()}


def test_config4_sampled_layers_and_head(ctx):
    """The benchmark's model (seed 3, drawn on the device), its context K/V (density
    0.1), a fully masked block at position 2048.  Layers 0 and 31 are compared per neuron
    from the GPU's own inputs to them; the head and unmasking of the step are compared
    from the GPU's last-layer output."""
    d = _large_desc()
    device = torch.device("cuda", 0)
    B, T, D, V, ctx_len = d["B"], d["T"], d["D"], d["V"], 2048
    weights = synth.device_model(3, d, device)
    k_u8, v_u8 = synth.device_context_spikes(4, d["n_layers"], T, d["Lmax"], D, ctx_len, 0.1,
                                             device)
    model = api.Model(ctx, d, weights)
    words = api.words(D)
    kc = torch.zeros((d["n_layers"], T, d["Lmax"], words), dtype=torch.int32, device=device)
    vc = torch.zeros_like(kc)
    for l in range(d["n_layers"]):
        for t in range(T):
            for j0 in range(0, d["Lmax"], 256):  # the packer takes at most 256 rows
                j1 = min(d["Lmax"], j0 + 256)
                kc[l, t, j0:j1] = api.pack_spikes(ctx, k_u8[l, t, j0:j1].contiguous(), 1).row_bits
                vc[l, t, j0:j1] = api.pack_spikes(ctx, v_u8[l, t, j0:j1].contiguous(), 1).row_bits
    ctx.sync()
    # the block's embedding currents and spikes (mask token at positions 2048..2079)
    tok_row = weights["tok_emb"][V:V + 1].cpu().numpy()
    pos_rows = weights["pos_emb"][ctx_len:ctx_len + B].cpu().numpy()
    tokens = np.full(B, V, np.int32)
    tok_tab = np.zeros((V + 1, D), np.float32)
    tok_tab[V] = tok_row[0]
    pos_tab = np.zeros((d["Lmax"], D), np.float32)
    pos_tab[ctx_len:ctx_len + B] = pos_rows
    u = oracle.embed(tok_tab, pos_tab, tokens, T, ctx_len)
    x, _, _ = oracle.if_f32(u.reshape(B, T, D), d["theta"])
    x = x.reshape(B * T, D)
    # the GPU runs the layers in order; layers 0 and 31 are checked from the GPU's inputs
    x_blk = api.pack_spikes(ctx, dev(x), T)
    u_dev = dev(u)
    flipped = {}
    for l in range(d["n_layers"]):
        if l in (0, d["n_layers"] - 1):
            xin = unpack_rows(host(x_blk.row_bits), D)
            uin = host(u_dev)
            k_h = unpack_rows(host(kc[l]), D)
            v_h = unpack_rows(host(vc[l]), D)
            flipped[l], _ = compare_layer(ctx, model, d, l, _host_lw(weights["layers"][l]), xin,
                                          uin, k_h, v_h, ctx_len)
        kl, vl = kc[l].clone(), vc[l].clone()
        x_blk, u_dev, _ = model.layer_forward(l, x_blk, u_dev, kl, vl, ctx_len)
    ctx.sync()
    x_last = unpack_rows(host(x_blk.row_bits), D)
    # head (4096 -> 32000) and unmasking through the public step on the same state
    blk = api.Block(model, kc, vc, ctx_len=ctx_len)
    logits = torch.empty(B, V, dtype=torch.float32, device=device)
    unm = torch.empty(B // d["S"], dtype=torch.int32, device=device)
    blk.denoise_step(unmasked_out=unm, logits_out=logits)
    ctx.sync()
    hw, hs = (t.cpu().numpy() for t in weights["head"])
    lo = oracle.head(x_last, hw, hs, B, T)
    assert np.array_equal(host(logits), lo)
    tk, mk, conf, _, chosen = oracle.unmask(lo, B // d["S"], tokens, np.ones(B, np.uint8))
    got = host(unm)
    if not np.array_equal(got, chosen):
        # only a near tie of the confidences (both sides in fp64, different exp) may reorder
        c = np.sort(conf)[::-1]
        k = B // d["S"]
        assert abs(c[k - 1] - c[k]) <= 1e-12 * c[k - 1], (got, chosen)
    else:
        assert np.array_equal(host(blk.tokens), tk)


# ------------------------------------------------------- small model end to end
def test_config3_short_generation(ctx):
    """12 layers, d_model 768, 12 x 64 heads, MLP 3072, vocab 32000, block 8, 8 steps,
    T 4, a 128-token prompt (16 commit passes) and 2 generated blocks (16 tokens, 18 more
    passes): every pass compared exactly, a differing pass traced per neuron."""
    from test_gpu_model import _generate_both
    desc = synth.model_desc(n_layers=12, D=768, H=12, F=3072, V=32000, T=4, B=8, S=8,
                            Lmax=144, gated=False)
    toks, traced = _generate_both(ctx, desc, 2, prompt_blocks=16, gen_blocks=2)
    assert len(toks) == 2 and all(((t >= 0) & (t < 32000)).all() for t in toks)
