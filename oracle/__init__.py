"""Python face of the N-MDLM CPU oracle (TEST INFRASTRUCTURE ONLY).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It marshals numpy arrays into the plain C
oracle (``nmdlm_oracle.c``), which restates the definitions of Wu et al.,
"Neuromorphic Diffusion Language Models" (arXiv 2607.24841).  Nothing here shares
code with the CUDA library.

Array conventions: spikes uint8 0/1 ``[B*T, N]`` (row ``b*T + t``), weights int8
``W^T [d_in, d_out]``, scales float32 ``[d_out]``, K/V caches uint8 ``[T, L, D]``.
"""
import ctypes as C
import math

import numpy as np

from . import build as _build

IF_CHARGE_THEN_FIRE = 0
IF_FIRE_THEN_CHARGE = 1
EPI_INT = 0
EPI_F32 = 1

_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(_build.build())
        _declare(_lib)
    return _lib


_p = C.c_void_p
_i = C.c_int


def _declare(L):
    L.orc_version.restype = _i
    L.orc_set_threads.argtypes = [_i]
    L.orc_get_threads.restype = _i
    L.orc_abs_sum_exact.argtypes = [_p, _i]
    L.orc_abs_sum_exact.restype = C.c_double
    L.orc_if_int.argtypes = [_p, _i, _i, _i, C.c_int64, _i, _p, _p]
    L.orc_if_f32.argtypes = [_p, _i, _i, _i, C.c_float, _p, _p, _p]
    L.orc_pack.argtypes = [_p, _i, _i, _p, _p, _p, _p, _p]
    L.orc_qbsm.argtypes = [_p, _p, _i, _i, _i, _p]
    L.orc_qbsm_at.argtypes = [_p, _p, _i, _i, _i, _i, _p, _p, _p]
    L.orc_qbsm_counts.argtypes = [_p, _i, _i, _i, _p, _p]
    L.orc_if_epilogue.argtypes = [_p, _i, _i, _i, _p, _p, _p, _i, C.c_int64, C.c_float,
                                  _p, _p, _p]
    L.orc_attention.argtypes = [_p, _p, _p, _i, _i, _i, _i, _i, C.c_double, _p]
    L.orc_layer.argtypes = [C.POINTER(OrcModel), C.POINTER(OrcLayerW), _p, _p, _p, _p, _i,
                            _p, _p, C.POINTER(OrcLayerTrace)]
    L.orc_embed.argtypes = [_p, _p, _p, _i, _i, _i, _i, _p]
    L.orc_head.argtypes = [_p, _p, _p, _i, _i, _i, _i, _p]
    L.orc_unmask.argtypes = [_p, _i, _i, _i, _p, _p, _p, _p, _p]
    L.orc_unmask.restype = _i
    L.orc_block_step.argtypes = [C.POINTER(OrcModel), C.POINTER(OrcLayerW), _p, _p, OrcLin,
                                 _p, _p, _p, _p, _i, _i, _p, _p]
    L.orc_block_step.restype = _i
    L.orc_block_step_margin.argtypes = [C.POINTER(OrcModel), C.POINTER(OrcLayerW), _p, _p,
                                        OrcLin, _p, _p, _p, _p, _i, _i, _p, _p, _p]
    L.orc_block_step_margin.restype = _i
    L.orc_ternary_encode.argtypes = [_p, _i, _i, C.c_float, _i, _p, _p, _p]
    L.orc_ternary_planes_needed.argtypes = [C.c_int64]
    L.orc_ternary_planes_needed.restype = _i
    L.orc_ternary_linear.argtypes = [_p, _p, _i, _i, _i, _i, _p, _p]
    L.orc_ternary_if.argtypes = [_p, _i, _i, _i, C.c_int64, _p, _p]


class OrcModel(C.Structure):
    _fields_ = [(n, C.c_int) for n in
                ("n_layers", "D", "H", "dh", "F", "gated", "V", "T", "B", "S", "Lmax")] + \
               [("theta", C.c_float), ("n_enc", C.c_int)]


class OrcLin(C.Structure):
    _fields_ = [("w", C.c_void_p), ("scale", C.c_void_p)]


class OrcLayerW(C.Structure):
    _fields_ = [(n, OrcLin) for n in ("q", "k", "v", "o", "gate", "up", "down")]


class OrcLayerTrace(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("q", "attn_cur", "attn", "attn_margin", "u1",
                                            "x1", "g", "h")]


def set_threads(n):
    """Host threads of the oracle's large loops (results do not depend on it)."""
    lib().orc_set_threads(int(n))


def get_threads():
    return lib().orc_get_threads()


def abs_sum_exact(row):
    """Eq. (7)'s sum of |a| over one fp32 row, exact, rounded once to fp64."""
    r = np.ascontiguousarray(row, np.float32)
    return lib().orc_abs_sum_exact(r.ctypes.data_as(C.c_void_p), r.size)


def _c(a, dtype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


# ------------------------------------------------------------------ neurons
def if_int(current, theta, order=IF_CHARGE_THEN_FIRE):
    """IF neuron, Sec. II-B Eq. (3)-(4), integer currents ``[B, T, N]``."""
    cur = _c(current, np.int64)
    B, T, N = cur.shape
    s = np.zeros((B, T, N), np.uint8)
    v = np.zeros((B, N), np.int64)
    lib().orc_if_int(_ptr(cur), B, T, N, int(theta), order, _ptr(s), _ptr(v))
    return s, v


def if_f32(current, theta):
    """IF neuron with fp32 currents ``[B, T, N]``; returns spikes, V_T, margin."""
    cur = _c(current, np.float32)
    B, T, N = cur.shape
    s = np.zeros((B, T, N), np.uint8)
    v = np.zeros((B, N), np.float32)
    m = np.zeros((B, N), np.float64)
    lib().orc_if_f32(_ptr(cur), B, T, N, float(theta), _ptr(s), _ptr(v), _ptr(m))
    return s, v, m


# ---------------------------------------------------------------- packing
def pack(spikes):
    """Packed forms and active set of a ``[BT, D]`` spike block (Sec. IV-A (ii))."""
    s = _c(spikes, np.uint8)
    BT, D = s.shape
    dw, bw = (D + 31) // 32, (BT + 31) // 32
    rb = np.zeros((BT, dw), np.uint32)
    cm = np.zeros((D, bw), np.uint32)
    am = np.zeros((dw,), np.uint32)
    ai = np.zeros((max(D, 1),), np.int32)
    na = np.zeros((1,), np.int32)
    lib().orc_pack(_ptr(s), BT, D, _ptr(rb), _ptr(cm), _ptr(am), _ptr(ai), _ptr(na))
    n = int(na[0])
    return dict(row_bits=rb, col_masks=cm, active_mask=am, active_idx=ai[:n].copy(),
                n_active=n)


# ------------------------------------------------------------------ QBSM
def qbsm(spikes, wT):
    """Y = X W^T over binary spikes (Sec. IV-A), int64 ``[BT, d_out]``."""
    s = _c(spikes, np.uint8)
    w = _c(wT, np.int8)
    BT, d_in = s.shape
    assert w.shape[0] == d_in
    d_out = w.shape[1]
    acc = np.zeros((BT, d_out), np.int64)
    lib().orc_qbsm(_ptr(s), _ptr(w), BT, d_in, d_out, _ptr(acc))
    return acc


# ------------------------------------------------ ternary bitwise coding
def ternary_encode(a, K, T):
    """Adaptive quantiser and bitwise ternary spikes, Sec. II-C Eq. (7)-(8).

    ``a`` fp32 ``[N, D]`` (one activation vector per row).  Returns spikes int8
    ``[N, T, D]`` in {-1, 0, 1} (plane t-1 carries weight 2^{t-1}), ahat int32
    ``[N, D]`` and V_th fp32 ``[N]``."""
    x = _c(a, np.float32)
    N, D = x.shape
    s = np.zeros((N, T, D), np.int8)
    ah = np.zeros((N, D), np.int32)
    vth = np.zeros((N,), np.float32)
    lib().orc_ternary_encode(_ptr(x), N, D, float(K), int(T), _ptr(s), _ptr(ah), _ptr(vth))
    return s, ah, vth


def ternary_planes_needed(m):
    """Bit length of m = max|ahat|: the planes Eq. (8) needs to reach m."""
    return int(lib().orc_ternary_planes_needed(int(m)))


def ternary_linear(s, wT):
    """Currents I_t = W^T s_t of ternary spikes ``[N, T, D]`` and y = sum_t 2^{t-1} I_t
    (Sec. II-C); returns (I int64 ``[N, T, d_out]``, y int64 ``[N, d_out]``)."""
    sp = _c(s, np.int8)
    w = _c(wT, np.int8)
    N, T, D = sp.shape
    assert w.shape[0] == D
    d_out = w.shape[1]
    I = np.zeros((N, T, d_out), np.int64)
    y = np.zeros((N, d_out), np.int64)
    lib().orc_ternary_linear(_ptr(sp), _ptr(w), N, T, D, d_out, _ptr(I), _ptr(y))
    return I, y


def ternary_if(y, T, theta=1):
    """Modified IF of Sec. II-C (Eq. (9)-(10), as read in the header) on y [N, d_out]:
    returns (spikes int8 [N, T, d_out] in {-1, 0, 1}, residual int64 [N, d_out])."""
    yy = _c(y, np.int64)
    N, d_out = yy.shape
    s = np.zeros((N, T, d_out), np.int8)
    v = np.zeros((N, d_out), np.int64)
    lib().orc_ternary_if(_ptr(yy), N, d_out, int(T), int(theta), _ptr(s), _ptr(v))
    return s, v


def qbsm_at(spikes, wT, bt_idx, o_idx):
    s = _c(spikes, np.uint8)
    w = _c(wT, np.int8)
    bi = _c(bt_idx, np.int32)
    oi = _c(o_idx, np.int32)
    acc = np.zeros((bi.size,), np.int64)
    lib().orc_qbsm_at(_ptr(s), _ptr(w), s.shape[0], s.shape[1], w.shape[1], bi.size,
                      _ptr(bi), _ptr(oi), _ptr(acc))
    return acc


def qbsm_counts(spikes, d_out):
    s = _c(spikes, np.uint8)
    rows = np.zeros(1, np.int64)
    sops = np.zeros(1, np.int64)
    lib().orc_qbsm_counts(_ptr(s), s.shape[0], s.shape[1], d_out, _ptr(rows), _ptr(sops))
    return int(rows[0]), int(sops[0])


def if_epilogue(acc, B, T, scale=None, residual=None, gate=None, kind=EPI_F32,
                theta_i=0, theta_f=1.0):
    """IF epilogue of a spiking linear layer; returns (current, spikes, margin)."""
    a = _c(acc, np.int64)
    d_out = a.shape[-1]
    a = a.reshape(B * T, d_out)
    sc = None if scale is None else _c(scale, np.float32)
    res = None if residual is None else _c(residual, np.float32).reshape(B * T, d_out)
    g = None if gate is None else _c(gate, np.uint8).reshape(B * T, d_out)
    cur = np.zeros((B * T, d_out), np.float32)
    s = np.zeros((B * T, d_out), np.uint8)
    m = np.full((B, d_out), np.inf, np.float64)
    lib().orc_if_epilogue(_ptr(a), B, T, d_out, _ptr(sc), _ptr(res), _ptr(g), kind,
                          int(theta_i), float(theta_f), _ptr(cur) if sc is not None else None,
                          _ptr(s), _ptr(m) if kind == EPI_F32 else None)
    return cur, s, m


# -------------------------------------------------------------- attention
def attention(q, k, v, B, T, H, dh, alpha=None):
    """BBM spike attention; q ``[B*T, D]``, k/v ``[T, L, D]`` -> fp32 ``[B*T, D]``."""
    qq = _c(q, np.uint8)
    kk = _c(k, np.uint8)
    vv = _c(v, np.uint8)
    L = kk.shape[1]
    if alpha is None:
        alpha = 1.0 / math.sqrt(dh)
    out = np.zeros((B * T, H * dh), np.float32)
    lib().orc_attention(_ptr(qq), _ptr(kk), _ptr(vv), B, T, L, H, dh, float(alpha), _ptr(out))
    return out


# ------------------------------------------------------------------ model
def model_struct(desc):
    """desc: dict with n_layers, D, H, dh, F, gated, V, T, B, S, Lmax, theta[, n_enc]."""
    return OrcModel(*(int(desc[n]) for n in ("n_layers", "D", "H", "dh", "F", "gated", "V",
                                             "T", "B", "S", "Lmax")), float(desc["theta"]),
                    int(desc.get("n_enc", 0)))


def _lin(keep, w, scale):
    w = _c(w, np.int8)
    s = _c(scale, np.float32)
    keep += [w, s]
    return OrcLin(_ptr(w), _ptr(s))


def layer_struct(keep, lw):
    """lw: dict with q,k,v,o,up,down[,gate] each a (wT, scale) pair."""
    names = ("q", "k", "v", "o", "gate", "up", "down")
    lins = []
    for n in names:
        if n in lw and lw[n] is not None:
            lins.append(_lin(keep, *lw[n]))
        else:
            lins.append(OrcLin(None, None))
    return OrcLayerW(*lins)


def layer(desc, lw, x_in, u_in, k_cache, v_cache, ctx):
    """One spiking transformer layer; caches ``[T, Lmax, D]`` are updated in place at
    positions ctx..ctx+B-1.  Returns (x_out, u_out, trace dict)."""
    m = model_struct(desc)
    keep = []
    w = layer_struct(keep, lw)
    B, T, D, F = m.B, m.T, m.D, m.F
    BT = B * T
    x = _c(x_in, np.uint8).reshape(BT, D)
    u = _c(u_in, np.float32).reshape(BT, D)
    assert k_cache.dtype == np.uint8 and k_cache.flags.c_contiguous
    assert v_cache.dtype == np.uint8 and v_cache.flags.c_contiguous
    assert k_cache.shape == v_cache.shape == (T, m.Lmax, D)
    assert 0 <= ctx and ctx + B <= m.Lmax, "the block must fit in the caches"
    x_out = np.zeros((BT, D), np.uint8)
    u_out = np.zeros((BT, D), np.float32)
    tr = dict(q=np.zeros((BT, D), np.uint8), attn_cur=np.zeros((BT, D), np.float32),
              attn=np.zeros((BT, D), np.uint8), attn_margin=np.zeros((B, D), np.float64),
              u1=np.zeros((BT, D), np.float32), x1=np.zeros((BT, D), np.uint8),
              g=np.zeros((BT, F), np.uint8), h=np.zeros((BT, F), np.uint8))
    t = OrcLayerTrace(*(_ptr(tr[n]) for n in ("q", "attn_cur", "attn", "attn_margin", "u1",
                                               "x1", "g", "h")))
    lib().orc_layer(C.byref(m), C.byref(w), _ptr(x), _ptr(u), _ptr(k_cache), _ptr(v_cache),
                    int(ctx), _ptr(x_out), _ptr(u_out), C.byref(t))
    if not desc["gated"]:
        tr.pop("g")
    return x_out, u_out, tr


def embed(tok_emb, pos_emb, tokens, T, pos0):
    te = _c(tok_emb, np.float32)
    pe = _c(pos_emb, np.float32)
    tk = _c(tokens, np.int32)
    B, D = tk.size, te.shape[1]
    u0 = np.zeros((B * T, D), np.float32)
    lib().orc_embed(_ptr(te), _ptr(pe), _ptr(tk), B, T, D, int(pos0), _ptr(u0))
    return u0


def head(x, wT, scale, B, T):
    xx = _c(x, np.uint8)
    w = _c(wT, np.int8)
    s = _c(scale, np.float32)
    D, V = w.shape
    logits = np.zeros((B, V), np.float32)
    lib().orc_head(_ptr(xx), _ptr(w), _ptr(s), B, T, D, V, _ptr(logits))
    return logits


def unmask(logits, k, tokens, mask):
    """Greedy unmasking; returns (tokens, mask, conf, tok, chosen) as new arrays."""
    lg = _c(logits, np.float32)
    B, V = lg.shape
    tk = _c(tokens, np.int32).copy()
    mk = _c(mask, np.uint8).copy()
    conf = np.zeros(B, np.float64)
    tok = np.zeros(B, np.int32)
    chosen = np.full(max(k, 1), -1, np.int32)
    n = lib().orc_unmask(_ptr(lg), B, V, int(k), _ptr(tk), _ptr(mk), _ptr(conf), _ptr(tok),
                         _ptr(chosen))
    return tk, mk, conf, tok, chosen[:n].copy()


def block_step(desc, layers, tok_emb, pos_emb, head_w, tokens, mask, k_cache, v_cache, ctx,
               commit=False, return_margin=False):
    """One denoising step (or a commit pass).  Caches ``[n_layers, T, Lmax, D]`` are
    updated in place; returns (tokens, mask, logits or None, chosen[, min attention
    membrane margin])."""
    m = model_struct(desc)
    keep = []
    assert len(layers) == m.n_enc + m.n_layers
    arr = (OrcLayerW * len(layers))(*[layer_struct(keep, lw) for lw in layers])
    hw = _lin(keep, *head_w)
    te = _c(tok_emb, np.float32)
    pe = _c(pos_emb, np.float32)
    tk = _c(tokens, np.int32).copy()
    mk = _c(mask, np.uint8).copy()
    assert k_cache.dtype == np.uint8 and k_cache.flags.c_contiguous
    assert v_cache.dtype == np.uint8 and v_cache.flags.c_contiguous
    assert k_cache.shape == v_cache.shape == (len(layers), m.T, m.Lmax, m.D)
    assert 0 <= ctx and ctx + m.B <= m.Lmax, "the block must fit in the caches"
    logits = None if commit else np.zeros((m.B, m.V), np.float32)
    chosen = np.full(max(m.B // m.S, 1), -1, np.int32)
    margin = np.zeros(1, np.float64)
    n = lib().orc_block_step_margin(C.byref(m), arr, _ptr(te), _ptr(pe), hw, _ptr(tk),
                                    _ptr(mk), _ptr(k_cache), _ptr(v_cache), int(ctx),
                                    int(bool(commit)), _ptr(logits), _ptr(chosen),
                                    _ptr(margin))
    if return_margin:
        return tk, mk, logits, chosen[:n].copy(), float(margin[0])
    return tk, mk, logits, chosen[:n].copy()
