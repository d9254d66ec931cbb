"""Layer- and pass-level parity checks shared by the model tests (not a test module).

Policy (the readings' parity rule): integer sums and every spike decided on exact or
deterministic fp32 arithmetic are compared bit-exactly.  Attention spikes are decided on
currents that went through exp/softmax, whose last bits differ between the CUDA path
and the oracle; such a spike may differ only where the oracle's attention membrane came
within MARGIN * max(1, theta) of the threshold.  A layer with such a flip is compared
further teacher-forced: the GPU layer is run again with the oracle's attention spikes fed
to its output projection (nmdlm_layer_io.attn_bits_in), and everything after attention
must then match exactly.  A generation pass that differs from the oracle must be traced,
layer by layer, to such near-threshold attention neurons, or the test fails.
"""
import numpy as np
import torch

import oracle
from bits import pack_rows, unpack_rows
from paper_2607_24841_gb300 import api

RTOL, ATOL = 1e-3, 1e-6
MARGIN = 1e-5


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    return t.cpu().numpy()


def near(desc, margin):
    return margin < MARGIN * max(1.0, desc["theta"])


def check_block(blk, spikes_u8):
    """A device SpikeBlock against uint8 spikes [BT, D]: row bits, column masks, mask."""
    r = oracle.pack(spikes_u8)
    BT, D = spikes_u8.shape
    assert np.array_equal(unpack_rows(host(blk.row_bits), D), spikes_u8)
    if blk.col_masks is not None:
        assert np.array_equal(host(blk.col_masks).view(np.uint32), r["col_masks"])
    if blk.active_mask is not None:
        assert np.array_equal(host(blk.active_mask).view(np.uint32), r["active_mask"])


def compare_layer(ctx, model, desc, layer, lw_host, x_u8, u, k_host, v_host, ctx_len):
    """Run layer `layer` on the GPU and in the oracle from the same input spikes x_u8
    [BT, D], residual currents u [BT, D] and K/V caches (host uint8 [T, Lmax, D], not
    modified); compare per the policy above.  Returns (flipped attention neurons, oracle
    outputs (x_out, u_out, k_after, v_after))."""
    B, T, D, F = desc["B"], desc["T"], desc["D"], desc["F"]
    BT = B * T
    ko, vo = k_host.copy(), v_host.copy()
    x2, u2, otr = oracle.layer(desc, lw_host, x_u8, u, ko, vo, ctx_len)

    x_blk = api.pack_spikes(ctx, dev(x_u8), T)
    u_dev = dev(u.reshape(BT, D))

    def run(attn_in=None):
        kc, vc = dev(pack_rows(k_host)), dev(pack_rows(v_host))
        ob, u_out, tr = model.layer_forward(layer, x_blk, u_dev, kc, vc, ctx_len, trace=True,
                                            attn_in=attn_in)
        ctx.sync()
        return ob, u_out, tr, kc, vc

    ob, u_out, tr, kc, vc = run()
    assert np.array_equal(unpack_rows(host(tr["q_bits"]), D), otr["q"])
    assert np.array_equal(unpack_rows(host(kc), D), ko)
    assert np.array_equal(unpack_rows(host(vc), D), vo)
    np.testing.assert_allclose(host(tr["attn_current"]), otr["attn_cur"], rtol=RTOL, atol=ATOL)
    a_gpu = unpack_rows(host(tr["attn_bits"]), D)
    bad = (a_gpu.reshape(B, T, D) != otr["attn"].reshape(B, T, D)).any(axis=1)  # [B, D]
    flipped = int(bad.sum())
    assert not np.any(bad & ~near(desc, otr["attn_margin"])), \
        "attention spikes differ away from the threshold"
    if flipped:
        # continue teacher-forced from the oracle's attention spikes
        ab = api.pack_spikes(ctx, dev(otr["attn"]), T)
        ob, u_out, tr, _, _ = run(attn_in=ab)
    assert np.array_equal(host(tr["u1"]), otr["u1"])
    assert np.array_equal(unpack_rows(host(tr["x1_bits"]), D), otr["x1"])
    if desc["gated"]:
        assert np.array_equal(unpack_rows(host(tr["g_bits"]), F), otr["g"])
    assert np.array_equal(unpack_rows(host(tr["h_bits"]), F), otr["h"])
    assert np.array_equal(host(u_out), u2)
    check_block(ob, x2)
    return flipped, (x2, u2, ko, vo)


def trace_pass(ctx, model, desc, host_model, tokens, ko, vo, ctx_len, commit):
    """A pass that differed: run it layer by layer from the oracle's own layer inputs,
    checking each GPU layer per neuron.  Returns the number of attention neurons that
    flipped within the threshold band (the only accepted cause of a difference) and, for
    a denoising step, whether the oracle's selection had a near tie of confidence."""
    B, T, D = desc["B"], desc["T"], desc["D"]
    u = oracle.embed(host_model["tok_emb"], host_model["pos_emb"], tokens, T, ctx_len)
    x, _, _ = oracle.if_f32(u.reshape(B, T, D), desc["theta"])
    x = x.reshape(B * T, D)
    flipped = 0
    n_enc = desc.get("n_enc", 0)
    # the layers the pass runs: every layer, or the encoders (context pass) / decoders
    first, count = 0, desc["n_layers"]
    if n_enc and commit:
        count = n_enc
    elif n_enc:
        first = n_enc
    for l in range(first, first + count):
        f, (x, u, _, _) = compare_layer(ctx, model, desc, l, host_model["layers"][l], x, u,
                                        ko[l], vo[l], ctx_len)
        flipped += f
    return flipped
