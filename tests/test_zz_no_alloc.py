"""The allocation-free spike attention entry point (nmdlm_spike_attention_noalloc).

Some callers cannot call cudaMalloc (a host framework whose allocator owns all device
memory, an embedded runtime with a fixed budget), so they cannot create a context.
This entry point stages its currents in a library-owned static device array instead.
It must give exactly what nmdlm_spike_attention gives, also on back-to-back calls
that share the array.  This file is collected last on purpose.
"""
import ctypes as C
import math

import numpy as np
import pytest
import torch

from bits import pack_rows
from paper_2607_24841_gb300 import _lib as L
from paper_2607_24841_gb300 import api, synth

pytestmark = pytest.mark.gpu


def _case(seed, B, T, L_ctx, H, dh, p):
    g = synth.rng(seed)
    D = H * dh
    Lk = L_ctx + B
    q = synth.bernoulli_spikes(g, (B * T, D), p)
    k = synth.bernoulli_spikes(g, (T, Lk, D), p)
    v = synth.bernoulli_spikes(g, (T, Lk, D), p)
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(pack_rows(a))).cuda()
    return dev(q), dev(k), dev(v), Lk


def _noalloc(lib, q, k, v, T, B, Lk, H, dh, theta):
    D = H * dh
    words = (D + 31) // 32
    bits = torch.empty(B * T, words, dtype=torch.int32, device="cuda")
    cm = torch.empty(D, (B * T + 31) // 32, dtype=torch.int32, device="cuda")
    mask = torch.empty(words, dtype=torch.int32, device="cuda")
    st = lib.nmdlm_spike_attention_noalloc(
        C.c_void_p(q.data_ptr()), C.c_void_p(k.data_ptr()), C.c_void_p(v.data_ptr()), T, B, Lk,
        k.shape[1], H, dh, 1.0 / math.sqrt(dh), theta, C.c_void_p(bits.data_ptr()),
        C.c_void_p(cm.data_ptr()), C.c_void_p(mask.data_ptr()),
        C.c_void_p(torch.cuda.current_stream().cuda_stream))
    return st, bits, cm, mask


@pytest.mark.parametrize("B,T,L_ctx,H,dh,p,theta", [
    (16, 4, 1024, 12, 64, 0.15, 0.05),   # tensor-core kernel, d_head 64
    (32, 4, 2048, 32, 128, 0.1, 0.08),   # tensor-core kernel, d_head 128, 32 queries
    (4, 4, 36, 2, 256, 0.15, 0.05),      # d_head 256: the CUDA-core kernel
    (32, 4, 32, 64, 128, 0.1, 0.08),     # B*T*H*d_head exactly the array's capacity
])
def test_noalloc_attention_matches_context_attention_twice(B, T, L_ctx, H, dh, p, theta):
    lib = L.load()
    ctx = api.Context(0)
    for seed in (1, 2):  # two calls in a row share the static array
        q, k, v, Lk = _case(seed * 100 + B, B, T, L_ctx, H, dh, p)
        st, bits, cm, mask = _noalloc(lib, q, k, v, T, B, Lk, H, dh, theta)
        assert st == L.OK
        _, ref = api.spike_attention(ctx, q, k, v, T, B, Lk, H, dh, theta=theta)
        ctx.sync()
        torch.cuda.synchronize()
        assert torch.equal(bits, ref.row_bits)
        assert torch.equal(cm, ref.col_masks)
        assert torch.equal(mask, ref.active_mask)
    ctx.close()


def test_noalloc_rejects_sizes_beyond_the_array():
    lib = L.load()
    cap = lib.nmdlm_spike_attention_noalloc_max()
    assert cap == 1 << 20
    # B*T*H*d_head = 64 * 4 * 64 * 128 > cap: rejected before any launch
    B, T, H, dh = 64, 4, 64, 128
    q = torch.zeros(B * T, H * dh // 32, dtype=torch.int32, device="cuda")
    kv = torch.zeros(T, B, H * dh // 32, dtype=torch.int32, device="cuda")
    st, *_ = _noalloc(lib, q, kv, kv, T, B, B, H, dh, 1.0)
    assert st == L.ERR_UNSUPPORTED
