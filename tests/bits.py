"""Bit-layout helpers for tests: convert the library's packed words to 0/1 arrays.

Packed layout (include/nmdlm.h): channel c of a row sits at bit c % 32 of word c // 32.
"""
import numpy as np


def unpack_rows(words_i32, n):
    """[..., words(n)] int32/uint32 -> [..., n] uint8."""
    w = np.ascontiguousarray(np.asarray(words_i32).astype(np.int64) & 0xFFFFFFFF, dtype="<u4")
    by = w.view(np.uint8)
    bits = np.unpackbits(by, axis=-1, bitorder="little")
    return bits[..., :n]


def pack_rows(bits_u8):
    """[..., n] 0/1 -> [..., words(n)] int32 (bit c%32 of word c//32)."""
    a = np.asarray(bits_u8, np.uint8)
    n = a.shape[-1]
    pad = (-n) % 32
    a = np.concatenate([a, np.zeros(a.shape[:-1] + (pad,), np.uint8)], axis=-1)
    return np.packbits(a, axis=-1, bitorder="little").view("<u4").astype(np.uint32).view(np.int32)
