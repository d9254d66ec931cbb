"""Seeded synthetic inputs shared by the CUDA path and the CPU oracle.

This module draws random numbers and formats them; it holds none of the method's
arithmetic (no IF neuron, no synaptic sum, no attention).  Every array it returns is
an *input* to both sides.  Recipes (the paper's WMT14 E2D2 data and trained weights
are not available, so these stand in for them):

* spike blocks: i.i.d. Bernoulli(p) in {0,1}, the i.i.d. model of Sec. IV-A;
* uniform int8 weights in [-127, 127] with fp32 per-output-channel scales ~U(0.001, 0.01);
* Gaussian-quantized int8 weights: W ~ N(0, 1/d_in), per-output-channel scale
  max_d |W[d, o]| / 127, W_q = clamp(round-half-away(W / scale), -127, 127);
* input currents i.i.d. N(0, 1) per (token, timestep, channel);
* token and position embeddings N(0, 1/2) each, so an embedded token's current is N(0, 1);
* context K/V spikes i.i.d. Bernoulli(p_ctx).

Host generation uses numpy's PCG64 (``np.random.default_rng(seed)``).  Models too large
to draw on the host in seconds (several GB of weights) are drawn on the device with
torch's seeded generator by ``device_model``; the oracle then receives host copies of
the sampled layers.
"""
import math

import numpy as np

# ----------------------------------------------------------------- primitives


def rng(seed):
    return np.random.default_rng(seed)


def bernoulli_spikes(g, shape, p):
    return (g.random(shape) < p).astype(np.uint8)


def uniform_int8(g, shape):
    return g.integers(-127, 128, size=shape, dtype=np.int16).astype(np.int8)


def uniform_scales(g, n, lo=0.001, hi=0.01):
    return g.uniform(lo, hi, size=n).astype(np.float32)


def normal_currents(g, shape):
    return g.standard_normal(shape, dtype=np.float32)


def _round_half_away(x):
    return np.sign(x) * np.floor(np.abs(x) + 0.5)


def gaussian_quantized(g, d_in, d_out):
    """(W^T int8 [d_in, d_out], scale float32 [d_out]) from W ~ N(0, 1/d_in)."""
    w = g.standard_normal((d_in, d_out), dtype=np.float32) / np.float32(math.sqrt(d_in))
    scale = (np.abs(w).max(axis=0) / np.float32(127.0)).astype(np.float32)
    scale = np.maximum(scale, np.float32(1e-12))
    q = np.clip(_round_half_away(w / scale[None, :]), -127, 127).astype(np.int8)
    return q, scale


def activation_rows(g, N, D, outlier_frac=0.002, outlier_gain=20.0):
    """Activation vectors [N, D] fp32 for the ternary coding: N(0, 1) values, a
    log-uniform scale per row in [0.1, 10], and a small share of outlier channels
    (gain 20) shared by every row, the heavy tail large-model activations show."""
    a = g.standard_normal((N, D), dtype=np.float32)
    a *= np.exp(g.uniform(math.log(0.1), math.log(10.0), (N, 1))).astype(np.float32)
    n_out = int(round(outlier_frac * D))
    if n_out:
        cols = g.choice(D, n_out, replace=False)
        a[:, cols] *= np.float32(outlier_gain)
    return a


# --------------------------------------------------------------- workloads
def ternary_case(seed, N, D, d_out):
    """Ternary-coded linear: activations [N, D] fp32 and Gaussian-quantised W^T."""
    g = rng(seed)
    a = activation_rows(g, N, D)
    w, _ = gaussian_quantized(g, D, d_out)
    return a, w


def linear_case(seed, BT, d_in, d_out, p, weights="uniform"):
    """One spiking linear layer: spikes [BT, d_in], W^T, scale."""
    g = rng(seed)
    s = bernoulli_spikes(g, (BT, d_in), p)
    if weights == "uniform":
        w = uniform_int8(g, (d_in, d_out))
        sc = uniform_scales(g, d_out)
    else:
        w, sc = gaussian_quantized(g, d_in, d_out)
    return s, w, sc


def model_desc(n_layers, D, H, F, V, T, B, S, Lmax, gated=False, theta=1.0, n_enc=0):
    """n_layers: the layers of a denoising step (the decoder when n_enc > 0); n_enc: the
    encoder layers of the encoder-decoder split (0: one set of layers serves both)."""
    return dict(n_layers=n_layers, D=D, H=H, dh=D // H, F=F, gated=int(bool(gated)), V=V,
                T=T, B=B, S=S, Lmax=Lmax, theta=float(theta), n_enc=int(n_enc))


def n_all_layers(desc):
    """Layers the model holds (encoder layers first), and caches it needs."""
    return desc["n_layers"] + desc.get("n_enc", 0)


def host_layer(g, desc):
    D, F = desc["D"], desc["F"]
    lw = dict(q=gaussian_quantized(g, D, D), k=gaussian_quantized(g, D, D),
              v=gaussian_quantized(g, D, D), o=gaussian_quantized(g, D, D))
    if desc["gated"]:
        lw["gate"] = gaussian_quantized(g, D, F)
    lw["up"] = gaussian_quantized(g, D, F)
    lw["down"] = gaussian_quantized(g, F, D)
    return lw


def host_model(seed, desc, with_head=True):
    """Every weight of a small model on the host (numpy)."""
    g = rng(seed)
    layers = [host_layer(g, desc) for _ in range(n_all_layers(desc))]
    D, V = desc["D"], desc["V"]
    s = np.float32(math.sqrt(0.5))
    tok_emb = g.standard_normal((V + 1, D), dtype=np.float32) * s
    pos_emb = g.standard_normal((desc["Lmax"], D), dtype=np.float32) * s
    head = gaussian_quantized(g, D, V) if with_head else None
    return dict(layers=layers, tok_emb=tok_emb, pos_emb=pos_emb, head=head)


def context_spikes(seed, n_layers, T, Lmax, D, ctx, p_ctx):
    """Context K and V spikes uint8 [n_layers, T, Lmax, D]; positions >= ctx are zero."""
    g = rng(seed)
    k = np.zeros((n_layers, T, Lmax, D), np.uint8)
    v = np.zeros((n_layers, T, Lmax, D), np.uint8)
    k[:, :, :ctx, :] = bernoulli_spikes(g, (n_layers, T, ctx, D), p_ctx)
    v[:, :, :ctx, :] = bernoulli_spikes(g, (n_layers, T, ctx, D), p_ctx)
    return k, v


# ------------------------------------------------------- device-side models
def device_gaussian_quantized(gen, d_in, d_out, device):
    import torch
    w = torch.randn((d_in, d_out), generator=gen, device=device, dtype=torch.float32)
    w = w / math.sqrt(d_in)
    scale = (w.abs().amax(dim=0) / 127.0).clamp_min(1e-12)
    x = w / scale[None, :]
    q = (torch.sign(x) * torch.floor(x.abs() + 0.5)).clamp_(-127, 127).to(torch.int8)
    return q, scale.to(torch.float32)


def device_model(seed, desc, device, with_head=True):
    """The same recipe as ``host_model`` drawn on the device with torch's seeded
    generator, for models of several GB.  Returns torch tensors."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    D, F, V = desc["D"], desc["F"], desc["V"]
    layers = []
    for _ in range(n_all_layers(desc)):
        lw = dict(q=device_gaussian_quantized(gen, D, D, device),
                  k=device_gaussian_quantized(gen, D, D, device),
                  v=device_gaussian_quantized(gen, D, D, device),
                  o=device_gaussian_quantized(gen, D, D, device))
        if desc["gated"]:
            lw["gate"] = device_gaussian_quantized(gen, D, F, device)
        lw["up"] = device_gaussian_quantized(gen, D, F, device)
        lw["down"] = device_gaussian_quantized(gen, F, D, device)
        layers.append(lw)
    s = math.sqrt(0.5)
    tok_emb = torch.randn((V + 1, D), generator=gen, device=device) * s
    pos_emb = torch.randn((desc["Lmax"], D), generator=gen, device=device) * s
    head = device_gaussian_quantized(gen, D, V, device) if with_head else None
    return dict(layers=layers, tok_emb=tok_emb, pos_emb=pos_emb, head=head)


def device_context_spikes(seed, n_layers, T, Lmax, D, ctx, p_ctx, device):
    """Context K/V spikes as uint8 [n_layers, T, Lmax, D] on the device."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    out = []
    for _ in range(2):
        x = torch.zeros((n_layers, T, Lmax, D), dtype=torch.uint8, device=device)
        x[:, :, :ctx, :] = (torch.rand((n_layers, T, ctx, D), generator=gen, device=device)
                            < p_ctx).to(torch.uint8)
        out.append(x)
    return out[0], out[1]
