"""PyTorch-facing wrappers of the C ABI (device memory and streams only).

Every function here allocates its output tensors with torch, passes raw device
pointers and the current CUDA stream to libnmdlm.so, and returns the tensors.  All
arithmetic of the spiking path runs in the library's CUDA kernels.
"""
import ctypes as C
import math
from dataclasses import dataclass
from typing import Optional

import torch

from . import _lib as L


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def words(n):
    return (n + 31) // 32


def _u32(*shape, device):
    # torch has no uint32 arithmetic on every version; int32 storage is bit-identical.
    return torch.empty(*shape, dtype=torch.int32, device=device)


# ----------------------------------------------------------------- context
class Context:
    """Owns an nmdlm_ctx (workspace + device error word) on one device."""

    def __init__(self, device=0, workspace_bytes=0):
        self.lib = L.load()
        self.device = torch.device("cuda", device) if isinstance(device, int) else device
        h = C.c_void_p()
        L.check(self.lib.nmdlm_ctx_create(C.byref(h), self.device.index or 0,
                                          int(workspace_bytes)), "nmdlm_ctx_create")
        self.h = h

    def close(self):
        if getattr(self, "h", None):
            self.lib.nmdlm_ctx_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def sync(self, stream=None):
        """Synchronize and raise NmdlmError on a recorded device-side error."""
        L.check(self.lib.nmdlm_ctx_sync_status(self.h, _stream(stream)), "device status")

    def sync_status(self, stream=None):
        return self.lib.nmdlm_ctx_sync_status(self.h, _stream(stream))

    def set_impl(self, impl):
        L.check(self.lib.nmdlm_ctx_set_impl(self.h, int(impl)), "set_impl")

    def set_wait_limit(self, ns):
        L.check(self.lib.nmdlm_ctx_set_wait_limit(self.h, int(ns)), "set_wait_limit")

    def debug_set(self, key, value):
        L.check(self.lib.nmdlm_debug_set(self.h, int(key), int(value)), "debug_set")

    def probe_rate(self, op, M, N, count, n_acc=1, per_commit=0):
        """Cycles per operation of one CTA (measurement): op 0 tcgen05.mma kind::f16 with
        A in shared memory, 1 with A in tensor memory, 2 kind::f8f6f4 (e4m3), 3
        tcgen05.st of 32 lanes x 16 columns per warp, 4 e4m3 with A and B MN-major, 5
        e4m3 with B MN-major."""
        out = C.c_double(0.0)
        L.check(self.lib.nmdlm_debug_probe_rate(self.h, op, M, N, n_acc, per_commit, count,
                                                C.byref(out)),
                "probe_rate")
        return out.value

    def debug_wait_test(self, ns, stream=None):
        L.check(self.lib.nmdlm_debug_wait_test(self.h, int(ns), _stream(stream)), "wait_test")

    def set_profiling(self, on):
        L.check(self.lib.nmdlm_ctx_set_profiling(self.h, int(bool(on))), "set_profiling")

    def profile_launches(self, max_launches=1 << 14):
        """Per spiking-linear launch since profiling was enabled: a list of dicts
        {ms, rows, sops, d_in, d_out, BT} (call before profile_read)."""
        buf = (C.c_double * (6 * max_launches))()
        n = C.c_int(0)
        L.check(self.lib.nmdlm_ctx_profile_launches(self.h, max_launches, buf, C.byref(n)),
                "profile_launches")
        keys = ("ms", "rows", "sops", "d_in", "d_out", "BT")
        return [{k: buf[6 * i + j] for j, k in enumerate(keys)} for i in range(n.value)]

    def profile_read(self):
        n = C.c_uint64()
        ms = C.c_double()
        by = C.c_double()
        rows = C.c_double()
        L.check(self.lib.nmdlm_ctx_profile_read(self.h, C.byref(n), C.byref(ms), C.byref(by),
                                                C.byref(rows)), "profile_read")
        return dict(launches=n.value, total_ms=ms.value, total_bytes=by.value,
                    rows_fetched=rows.value)


# ------------------------------------------------------------------ spikes
@dataclass
class SpikeBlock:
    """Packed spike block of BT = B*T rows and D channels (see include/nmdlm.h)."""
    row_bits: torch.Tensor      # [BT, words(D)] int32 storage of uint32 words
    col_masks: torch.Tensor     # [D, words(BT)]
    active_mask: torch.Tensor   # [words(D)]
    BT: int
    T: int
    D: int
    active_idx: Optional[torch.Tensor] = None
    n_active: Optional[torch.Tensor] = None

    def struct(self):
        return L.Spikes(_ptr(self.row_bits), _ptr(self.col_masks), _ptr(self.active_mask),
                        _ptr(self.active_idx), _ptr(self.n_active), self.BT, self.T, self.D)


def empty_block(BT, T, D, device):
    return SpikeBlock(_u32(BT, words(D), device=device), _u32(D, words(BT), device=device),
                      _u32(words(D), device=device), BT, T, D)


def pack_spikes(ctx, spikes, T, stream=None):
    """nmdlm_pack_spikes: uint8 0/1 spikes [BT, D] -> SpikeBlock with active list."""
    assert spikes.dtype == torch.uint8 and spikes.is_cuda and spikes.is_contiguous()
    BT, D = spikes.shape
    dev = spikes.device
    blk = empty_block(BT, T, D, dev)
    blk.active_idx = torch.empty(max(D, 1), dtype=torch.int32, device=dev)
    blk.n_active = torch.empty(1, dtype=torch.int32, device=dev)
    L.check(ctx.lib.nmdlm_pack_spikes(ctx.h, _ptr(spikes), BT, D, _ptr(blk.row_bits),
                                      _ptr(blk.col_masks), _ptr(blk.active_mask),
                                      _ptr(blk.active_idx), _ptr(blk.n_active), _stream(stream)),
            "nmdlm_pack_spikes")
    return blk


def if_neuron(ctx, current, threshold, v_state=None, stream=None):
    """nmdlm_if_neuron: current [B, T, N] int32 or float32 -> SpikeBlock of B*T rows."""
    assert current.is_cuda and current.is_contiguous() and current.dim() == 3
    B, T, N = current.shape
    if current.dtype == torch.int32:
        dt, ti, tf = L.I32, int(threshold), 0.0
    else:
        assert current.dtype == torch.float32
        dt, ti, tf = L.F32, 0, float(threshold)
    blk = empty_block(B * T, T, N, current.device)
    L.check(ctx.lib.nmdlm_if_neuron(ctx.h, _ptr(current), dt, B, T, N, ti, tf, _ptr(v_state),
                                    _ptr(blk.row_bits), _ptr(blk.col_masks),
                                    _ptr(blk.active_mask), _stream(stream)), "nmdlm_if_neuron")
    return blk


def spike_linear(ctx, blk, wT, scale, mode=L.MODE_AUTO, want_acc=False, kind=L.IF_FP32,
                 threshold=1.0, residual=None, gate_bits=None, want_current=False,
                 want_block=True, stats=None, stream=None):
    """nmdlm_spike_linear.  Returns dict with acc [BT, d_out] int32 (if want_acc), the
    output SpikeBlock (row bits always; col masks/mask if want_block) and current."""
    d_in, d_out = wT.shape
    assert wT.dtype == torch.int8 and wT.is_contiguous() and blk.D == d_in
    dev = wT.device
    out = {}
    acc = torch.empty(blk.BT, d_out, dtype=torch.int32, device=dev) if want_acc else None
    ob = empty_block(blk.BT, blk.T, d_out, dev)
    if not want_block:
        ob.col_masks = None
        ob.active_mask = None
    cur = torch.empty(blk.BT, d_out, dtype=torch.float32, device=dev) if want_current else None
    epi = L.IfEpilogue(L.IF_INT if kind == L.IF_INT else L.IF_FP32,
                       int(threshold) if kind == L.IF_INT else 0,
                       float(threshold) if kind != L.IF_INT else 0.0,
                       _ptr(residual), _ptr(gate_bits), _ptr(cur), _ptr(ob.row_bits),
                       _ptr(ob.col_masks), _ptr(ob.active_mask))
    s = blk.struct()
    L.check(ctx.lib.nmdlm_spike_linear(ctx.h, C.byref(s), _ptr(wT), _ptr(scale), d_in, d_out,
                                       int(mode), _ptr(acc), C.byref(epi), _ptr(stats),
                                       _stream(stream)), "nmdlm_spike_linear")
    out["acc"] = acc
    out["block"] = ob
    out["current"] = cur
    return out


def spike_linear_acc(ctx, blk, wT, mode=L.MODE_AUTO, stats=None, stream=None):
    """Integer sums only (no epilogue)."""
    d_in, d_out = wT.shape
    acc = torch.empty(blk.BT, d_out, dtype=torch.int32, device=wT.device)
    s = blk.struct()
    L.check(ctx.lib.nmdlm_spike_linear(ctx.h, C.byref(s), _ptr(wT), None, d_in, d_out, int(mode),
                                       _ptr(acc), None, _ptr(stats), _stream(stream)),
            "nmdlm_spike_linear")
    return acc


def ternary_encode(ctx, a, K, T, stream=None):
    """nmdlm_ternary_encode: activations fp32 [N, D] -> (plus, minus) uint8 [N*T, D]
    spike planes (row n*T + t-1), ahat int32 [N, D], V_th fp32 [N] (Sec. II-C)."""
    assert a.dtype == torch.float32 and a.is_cuda and a.is_contiguous() and a.dim() == 2
    N, D = a.shape
    dev = a.device
    plus = torch.empty(N * T, D, dtype=torch.uint8, device=dev)
    minus = torch.empty(N * T, D, dtype=torch.uint8, device=dev)
    ahat = torch.empty(N, D, dtype=torch.int32, device=dev)
    vth = torch.empty(N, dtype=torch.float32, device=dev)
    L.check(ctx.lib.nmdlm_ternary_encode(ctx.h, _ptr(a), N, D, float(K), int(T), _ptr(plus),
                                         _ptr(minus), _ptr(ahat), _ptr(vth), _stream(stream)),
            "nmdlm_ternary_encode")
    return plus, minus, ahat, vth


def ternary_combine(ctx, acc_plus, acc_minus, N, T, stream=None):
    """nmdlm_ternary_combine: y [N, d_out] = sum_t 2^{t-1} (acc+ - acc-) of the planes."""
    assert acc_plus.dtype == torch.int32 and acc_minus.dtype == torch.int32
    assert acc_plus.shape == acc_minus.shape and acc_plus.shape[0] == N * T
    d_out = acc_plus.shape[1]
    y = torch.empty(N, d_out, dtype=torch.int32, device=acc_plus.device)
    L.check(ctx.lib.nmdlm_ternary_combine(ctx.h, _ptr(acc_plus), _ptr(acc_minus), N, int(T),
                                          d_out, _ptr(y), _stream(stream)),
            "nmdlm_ternary_combine")
    return y


def ternary_if(ctx, y, T, theta=1, want_v=True, stream=None):
    """nmdlm_ternary_if: the modified IF on y [N, d_out] int32; returns (spikes int8
    [N, T, d_out] in {-1, 0, 1}, residual V int32 [N, d_out] or None)."""
    assert y.dtype == torch.int32 and y.is_cuda and y.is_contiguous() and y.dim() == 2
    N, d_out = y.shape
    s = torch.empty(N, T, d_out, dtype=torch.int8, device=y.device)
    v = torch.empty(N, d_out, dtype=torch.int32, device=y.device) if want_v else None
    L.check(ctx.lib.nmdlm_ternary_if(ctx.h, _ptr(y), N, d_out, int(T), int(theta), _ptr(s),
                                     _ptr(v), _stream(stream)), "nmdlm_ternary_if")
    return s, v


def ternary_linear(ctx, a, wT, K, T, mode=L.MODE_AUTO, want_ahat=False, y=None, stream=None):
    """nmdlm_ternary_linear: y [N, d_out] int32 = W^T ahat of the bitwise ternary coding of
    a (fp32 [N, D]) with V_th = mean|a| / K over T planes; returns dict(y, ahat, vth)."""
    assert a.dtype == torch.float32 and a.is_cuda and a.is_contiguous() and a.dim() == 2
    assert wT.dtype == torch.int8 and wT.is_contiguous() and wT.shape[0] == a.shape[1]
    N, D = a.shape
    d_out = wT.shape[1]
    dev = a.device
    if y is None:
        y = torch.empty(N, d_out, dtype=torch.int32, device=dev)
    ahat = torch.empty(N, D, dtype=torch.int32, device=dev) if want_ahat else None
    vth = torch.empty(N, dtype=torch.float32, device=dev) if want_ahat else None
    L.check(ctx.lib.nmdlm_ternary_linear(ctx.h, _ptr(a), N, D, float(K), int(T), _ptr(wT), d_out,
                                         int(mode), _ptr(y), _ptr(ahat), _ptr(vth),
                                         _stream(stream)), "nmdlm_ternary_linear")
    return dict(y=y, ahat=ahat, vth=vth)


def spike_attention(ctx, q_bits, k_bits, v_bits, T, B, L_keys, H, d_head, theta=1.0,
                    alpha=None, want_current=True, stream=None):
    """nmdlm_spike_attention.  k_bits/v_bits [T, L_stride, words(H*d_head)]."""
    dev = q_bits.device
    D = H * d_head
    L_stride = k_bits.shape[1]
    if alpha is None:
        alpha = 1.0 / math.sqrt(d_head)
    cur = torch.empty(B * T, D, dtype=torch.float32, device=dev) if want_current else None
    ob = empty_block(B * T, T, D, dev)
    L.check(ctx.lib.nmdlm_spike_attention(ctx.h, _ptr(q_bits), _ptr(k_bits), _ptr(v_bits), T, B,
                                          L_keys, L_stride, H, d_head, float(alpha),
                                          float(theta), _ptr(cur), _ptr(ob.row_bits),
                                          _ptr(ob.col_masks), _ptr(ob.active_mask),
                                          _stream(stream)), "nmdlm_spike_attention")
    return cur, ob


# ------------------------------------------------------------------- model
class Model:
    """nmdlm_model over caller-owned device weights.

    weights: dict(layers=[dict(q=(wT, scale), k=..., v=..., o=..., up=..., down=...,
    [gate=...])], tok_emb, pos_emb, head=(wT, scale)) of CUDA tensors."""

    def __init__(self, ctx, desc, weights):
        self.ctx = ctx
        self.desc = dict(desc)
        self.w = weights
        d = L.ModelDesc(desc["n_layers"], desc["D"], desc["H"], desc["dh"], desc["F"],
                        int(desc["gated"]), desc["V"], desc["T"], float(desc["theta"]),
                        desc["B"], desc["S"], desc["Lmax"], int(desc.get("n_enc", 0)))
        self.cdesc = d
        n_all = desc["n_layers"] + int(desc.get("n_enc", 0))
        assert len(weights["layers"]) == n_all
        arr = (L.LayerW * n_all)()
        for i, lw in enumerate(weights["layers"]):
            for n in ("q", "k", "v", "o", "gate", "up", "down"):
                if n in lw and lw[n] is not None:
                    w, s = lw[n]
                    assert w.dtype == torch.int8 and w.is_contiguous() and w.is_cuda
                    setattr(arr[i], n, L.LinearW(_ptr(w), _ptr(s)))
        self._arr = arr
        hw, hs = weights["head"]
        h = C.c_void_p()
        L.check(ctx.lib.nmdlm_model_create(ctx.h, C.byref(d), arr, _ptr(weights["tok_emb"]),
                                           _ptr(weights["pos_emb"]),
                                           L.LinearW(_ptr(hw), _ptr(hs)), C.byref(h)),
                "nmdlm_model_create")
        self.h = h

    def close(self):
        if getattr(self, "h", None):
            self.ctx.lib.nmdlm_model_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @staticmethod
    def workspace_bytes(desc):
        lib = L.load()
        d = L.ModelDesc(desc["n_layers"], desc["D"], desc["H"], desc["dh"], desc["F"],
                        int(desc["gated"]), desc["V"], desc["T"], float(desc["theta"]),
                        desc["B"], desc["S"], desc["Lmax"], int(desc.get("n_enc", 0)))
        return int(lib.nmdlm_model_workspace_bytes(C.byref(d)))

    def new_caches(self):
        d = self.desc
        shape = (d["n_layers"] + int(d.get("n_enc", 0)), d["T"], d["Lmax"], words(d["D"]))
        dev = self.w["tok_emb"].device
        return (torch.zeros(shape, dtype=torch.int32, device=dev),
                torch.zeros(shape, dtype=torch.int32, device=dev))

    def layer_forward(self, layer, x_blk, u_in, k_cache, v_cache, ctx_len, trace=False,
                      attn_in=None, stream=None):
        """nmdlm_layer_forward.  k_cache/v_cache: this layer's [T, Lmax, words(D)].
        attn_in: a SpikeBlock of attention spikes fed to the output projection in place of
        the layer's own attention (teacher forcing, for parity checks)."""
        d = self.desc
        dev = u_in.device
        BT, D, F = d["B"] * d["T"], d["D"], d["F"]
        ob = empty_block(BT, d["T"], D, dev)
        u_out = torch.empty(BT, D, dtype=torch.float32, device=dev)
        tr = {}
        if trace:
            tr = dict(q_bits=_u32(BT, words(D), device=dev),
                      attn_current=torch.empty(BT, D, dtype=torch.float32, device=dev),
                      attn_bits=_u32(BT, words(D), device=dev),
                      u1=torch.empty(BT, D, dtype=torch.float32, device=dev),
                      x1_bits=_u32(BT, words(D), device=dev),
                      g_bits=_u32(BT, words(F), device=dev) if d["gated"] else None,
                      h_bits=_u32(BT, words(F), device=dev))
        io = L.LayerIO(_ptr(x_blk.row_bits), _ptr(x_blk.col_masks), _ptr(x_blk.active_mask),
                       _ptr(u_in), _ptr(k_cache), _ptr(v_cache), int(ctx_len),
                       _ptr(ob.row_bits), _ptr(ob.col_masks), _ptr(ob.active_mask), _ptr(u_out),
                       *[_ptr(tr.get(n)) for n in ("q_bits", "attn_current", "attn_bits", "u1",
                                                   "x1_bits", "g_bits", "h_bits")],
                       *((_ptr(attn_in.row_bits), _ptr(attn_in.col_masks),
                          _ptr(attn_in.active_mask)) if attn_in is not None
                         else (None, None, None)))
        L.check(self.ctx.lib.nmdlm_layer_forward(self.ctx.h, self.h, int(layer), C.byref(io),
                                                 _stream(stream)), "nmdlm_layer_forward")
        return ob, u_out, tr


class Block:
    """nmdlm_block_state: the block's tokens/mask and the K/V caches."""

    def __init__(self, model, k_cache=None, v_cache=None, ctx_len=0):
        d = model.desc
        dev = model.w["tok_emb"].device
        self.model = model
        self.tokens = torch.full((d["B"],), d["V"], dtype=torch.int32, device=dev)
        self.mask = torch.ones(d["B"], dtype=torch.int32, device=dev)
        if k_cache is None:
            k_cache, v_cache = model.new_caches()
        self.k_cache, self.v_cache = k_cache, v_cache
        self.st = L.BlockState(_ptr(self.tokens), _ptr(self.mask), _ptr(k_cache), _ptr(v_cache),
                               int(ctx_len), 0)

    @property
    def ctx_len(self):
        return self.st.ctx_len

    @property
    def step(self):
        return self.st.step

    def denoise_step(self, unmasked_out=None, logits_out=None, stream=None):
        m = self.model
        L.check(m.ctx.lib.nmdlm_block_denoise_step(m.ctx.h, m.h, C.byref(self.st),
                                                   _ptr(unmasked_out), _ptr(logits_out),
                                                   _stream(stream)), "nmdlm_block_denoise_step")

    def commit(self, stream=None):
        m = self.model
        L.check(m.ctx.lib.nmdlm_block_commit(m.ctx.h, m.h, C.byref(self.st), _stream(stream)),
                "nmdlm_block_commit")
