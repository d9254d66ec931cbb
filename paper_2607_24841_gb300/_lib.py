"""ctypes view of libnmdlm.so (include/nmdlm.h).  Argument marshalling only.

The library is built in-tree by ``build.py``.  Loading fails loudly when it is
missing or cannot be loaded: there is no CPU fallback for any entry point.
"""
import ctypes as C
import os

from . import build as _build

_p = C.c_void_p
_i = C.c_int
_u64 = C.c_uint64

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_TIMEOUT, ERR_WORKSPACE = range(6)
MODE_AUTO, MODE_SPARSE, MODE_DENSE = range(3)
IMPL_AUTO, IMPL_SIMT, IMPL_TC = range(3)
IF_INT, IF_FP32 = range(2)
I32, F32 = range(2)

# Every symbol include/nmdlm.h declares.
EXPORTS = [
    "nmdlm_status_string", "nmdlm_abi_version", "nmdlm_launch_count", "nmdlm_last_cuda_error",
    "nmdlm_ctx_create", "nmdlm_ctx_destroy",
    "nmdlm_ctx_sync_status", "nmdlm_ctx_set_impl", "nmdlm_ctx_set_wait_limit",
    "nmdlm_debug_wait_test", "nmdlm_ctx_set_profiling", "nmdlm_ctx_profile_read",
    "nmdlm_ctx_profile_launches",
    "nmdlm_pack_spikes", "nmdlm_if_neuron", "nmdlm_spike_linear", "nmdlm_spike_attention",
    "nmdlm_ternary_encode", "nmdlm_ternary_combine", "nmdlm_ternary_linear", "nmdlm_ternary_if",
    "nmdlm_spike_attention_noalloc", "nmdlm_spike_attention_noalloc_max",
    "nmdlm_model_create", "nmdlm_model_destroy", "nmdlm_model_workspace_bytes",
    "nmdlm_layer_forward", "nmdlm_block_denoise_step", "nmdlm_block_commit",
]


class NmdlmError(RuntimeError):
    def __init__(self, status, what=""):
        self.status = status
        msg = status_string(status)
        if status == ERR_CUDA:
            try:
                msg += " [" + load(build_if_missing=False).nmdlm_last_cuda_error().decode() + "]"
            except Exception:
                pass
        super().__init__(f"{what}: {msg} (status {status})" if what else msg)


class Spikes(C.Structure):
    _fields_ = [("row_bits", _p), ("col_masks", _p), ("active_mask", _p), ("active_idx", _p),
                ("n_active", _p), ("BT", C.c_int32), ("T", C.c_int32), ("D", C.c_int32)]


class IfEpilogue(C.Structure):
    _fields_ = [("kind", C.c_int32), ("threshold_i", C.c_int32), ("threshold_f", C.c_float),
                ("residual_in", _p), ("gate_bits", _p), ("current_out", _p),
                ("spikes_out", _p), ("col_masks_out", _p), ("active_mask_out", _p)]


class ModelDesc(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("d_head", C.c_int32), ("d_mlp", C.c_int32), ("gated", C.c_int32),
                ("vocab", C.c_int32), ("T", C.c_int32), ("theta", C.c_float),
                ("B", C.c_int32), ("S", C.c_int32), ("max_ctx", C.c_int32),
                ("n_enc_layers", C.c_int32)]


class LinearW(C.Structure):
    _fields_ = [("wT", _p), ("scale", _p)]


class LayerW(C.Structure):
    _fields_ = [(n, LinearW) for n in ("q", "k", "v", "o", "gate", "up", "down")]


class LayerIO(C.Structure):
    _fields_ = [("x_bits", _p), ("x_col_masks", _p), ("x_active_mask", _p), ("u_in", _p),
                ("k_cache", _p), ("v_cache", _p), ("ctx_len", C.c_int32),
                ("x_bits_out", _p), ("x_col_masks_out", _p), ("x_active_mask_out", _p),
                ("u_out", _p), ("q_bits", _p), ("attn_current", _p), ("attn_bits", _p),
                ("u1", _p), ("x1_bits", _p), ("g_bits", _p), ("h_bits", _p),
                ("attn_bits_in", _p), ("attn_col_masks_in", _p), ("attn_active_mask_in", _p)]


class BlockState(C.Structure):
    _fields_ = [("tokens", _p), ("mask", _p), ("k_cache", _p), ("v_cache", _p),
                ("ctx_len", C.c_int32), ("step", C.c_int32)]


_lib = None


def lib_path():
    return _build.LIB_PATH


def load(build_if_missing=True):
    """Load libnmdlm.so (building it first if it is missing or stale)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.build() if build_if_missing else _build.LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"libnmdlm.so not found at {path}; run build() first")
    L = C.CDLL(path)
    _declare(L)
    _lib = L
    return L


def _declare(L):
    sig = {
        "nmdlm_status_string": ([_i], C.c_char_p),
        "nmdlm_abi_version": ([], _i),
        "nmdlm_launch_count": ([], _u64),
        "nmdlm_last_cuda_error": ([], C.c_char_p),
        "nmdlm_ctx_create": ([C.POINTER(_p), _i, C.c_size_t], _i),
        "nmdlm_ctx_destroy": ([_p], _i),
        "nmdlm_ctx_sync_status": ([_p, _p], _i),
        "nmdlm_ctx_set_impl": ([_p, _i], _i),
        "nmdlm_ctx_set_wait_limit": ([_p, _u64], _i),
        "nmdlm_debug_wait_test": ([_p, _u64, _p], _i),
        "nmdlm_ctx_set_profiling": ([_p, _i], _i),
        "nmdlm_ctx_profile_read": ([_p, C.POINTER(_u64), C.POINTER(C.c_double),
                                    C.POINTER(C.c_double), C.POINTER(C.c_double)], _i),
        "nmdlm_ctx_profile_launches": ([_p, _i, _p, C.POINTER(_i)], _i),
        "nmdlm_pack_spikes": ([_p, _p, _i, _i, _p, _p, _p, _p, _p, _p], _i),
        "nmdlm_if_neuron": ([_p, _p, _i, _i, _i, _i, C.c_int32, C.c_float, _p, _p, _p, _p, _p],
                            _i),
        "nmdlm_spike_linear": ([_p, C.POINTER(Spikes), _p, _p, _i, _i, _i, _p,
                                C.POINTER(IfEpilogue), _p, _p], _i),
        "nmdlm_ternary_encode": ([_p, _p, _i, _i, C.c_float, _i, _p, _p, _p, _p, _p], _i),
        "nmdlm_ternary_combine": ([_p, _p, _p, _i, _i, _i, _p, _p], _i),
        "nmdlm_ternary_linear": ([_p, _p, _i, _i, C.c_float, _i, _p, _i, _i, _p, _p, _p, _p],
                                 _i),
        "nmdlm_spike_attention": ([_p, _p, _p, _p, _i, _i, _i, _i, _i, _i, C.c_float, C.c_float,
                                   _p, _p, _p, _p, _p], _i),
        "nmdlm_spike_attention_noalloc": ([_p, _p, _p, _i, _i, _i, _i, _i, _i, C.c_float,
                                           C.c_float, _p, _p, _p, _p], _i),
        "nmdlm_spike_attention_noalloc_max": ([], C.c_size_t),
        "nmdlm_model_create": ([_p, C.POINTER(ModelDesc), C.POINTER(LayerW), _p, _p, LinearW,
                                C.POINTER(_p)], _i),
        "nmdlm_model_destroy": ([_p], _i),
        "nmdlm_model_workspace_bytes": ([C.POINTER(ModelDesc)], C.c_size_t),
        "nmdlm_layer_forward": ([_p, _p, _i, C.POINTER(LayerIO), _p], _i),
        "nmdlm_block_denoise_step": ([_p, _p, C.POINTER(BlockState), _p, _p, _p], _i),
        "nmdlm_block_commit": ([_p, _p, C.POINTER(BlockState), _p], _i),
        "nmdlm_debug_set": ([_p, _i, _i], _i),
        "nmdlm_debug_probe_rate": ([_p, _i, _i, _i, _i, _i, _i, C.POINTER(C.c_double)], _i),
        "nmdlm_debug_probe_stream": ([_p, _i, _i, _i, _i, _i, _i, C.POINTER(C.c_double)], _i),
    }
    for name, (args, res) in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = res


def status_string(status):
    try:
        return load(build_if_missing=False).nmdlm_status_string(int(status)).decode()
    except Exception:
        return f"status {status}"


def check(status, what=""):
    if status != OK:
        raise NmdlmError(status, what)
