"""Host-side checks of the C ABI: the library builds, loads and exports every symbol
that include/nmdlm.h declares (no compute calls, no GPU needed)."""
import os
import re
import subprocess

import pytest

from conftest import ROOT


def _declared():
    src = open(os.path.join(ROOT, "include", "nmdlm.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(nmdlm_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_five_paper_calls():
    names = _declared()
    for n in ("nmdlm_pack_spikes", "nmdlm_spike_linear", "nmdlm_if_neuron",
              "nmdlm_spike_attention", "nmdlm_block_denoise_step"):
        assert n in names


def test_library_exports_every_declared_symbol():
    from paper_2607_24841_gb300 import _lib
    path = _lib.load().__dict__.get("_name") or _lib.lib_path()
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\s[TW]\s+(nmdlm_[a-z0-9_]+)$", out, flags=re.M))
    missing = [n for n in _declared() if n not in exported]
    assert not missing, missing
    assert set(_lib.EXPORTS) <= exported


def test_status_strings_and_version():
    from paper_2607_24841_gb300 import _lib
    L = _lib.load()
    assert L.nmdlm_abi_version() == 2
    assert L.nmdlm_status_string(0) == b"ok"
    assert L.nmdlm_status_string(4) == b"device wait timed out"


def test_invalid_arguments_rejected_without_gpu():
    import ctypes as C
    from paper_2607_24841_gb300 import _lib
    L = _lib.load()
    assert L.nmdlm_ctx_create(None, 0, 0) == _lib.ERR_INVALID_ARG
    assert L.nmdlm_ctx_destroy(None) == _lib.ERR_INVALID_ARG
    assert L.nmdlm_pack_spikes(None, None, 1, 1, None, None, None, None, None, None) == \
        _lib.ERR_INVALID_ARG
    assert L.nmdlm_ternary_encode(None, None, 1, 1, 1.0, 1, None, None, None, None, None) == \
        _lib.ERR_INVALID_ARG
    assert L.nmdlm_ternary_combine(None, None, None, 1, 1, 1, None, None) == _lib.ERR_INVALID_ARG
    assert L.nmdlm_ternary_linear(None, None, 1, 1, 1.0, 1, None, 1, 0, None, None, None,
                                  None) == _lib.ERR_INVALID_ARG
    assert L.nmdlm_model_workspace_bytes(None) == 0
    d = _lib.ModelDesc(2, 64, 2, 32, 96, 0, 50, 4, 1.0, 4, 3, 10)  # B % S != 0
    assert L.nmdlm_model_workspace_bytes(C.byref(d)) == 0
    d.S = 2
    assert L.nmdlm_model_workspace_bytes(C.byref(d)) > 0


@pytest.mark.skipif(os.path.exists("/dev/nvidia0"),
                    reason="host-only check: with a GPU present a size check that failed to "
                           "reject would launch on placeholder pointers")
def test_attention_noalloc_size_limits_without_gpu():
    # The context-free attention entry checks its sizes before any CUDA call, and checks
    # B*T <= 256 and H*d_head <= 2^20 without forming products that overflow int.
    import ctypes as C
    from paper_2607_24841_gb300 import _lib
    L = _lib.load()
    q = C.c_void_p(256)  # placeholder: every case below is rejected before any use

    def call(T, B, H, d_head):
        return L.nmdlm_spike_attention_noalloc(q, q, q, T, B, 8, 8, H, d_head, 0.1, 1.0, q,
                                               None, None, None)
    assert call(32, 1 << 27, 1, 32) == _lib.ERR_UNSUPPORTED   # B*T is 2^32
    assert call(4, 65, 1, 32) == _lib.ERR_UNSUPPORTED         # B*T = 260
    assert call(4, 8, 1 << 26, 64) == _lib.ERR_UNSUPPORTED    # H*d_head is 2^32
    assert call(4, 8, 1, 48) == _lib.ERR_UNSUPPORTED          # d_head not a multiple of 32
    assert call(0, 8, 1, 32) == _lib.ERR_INVALID_ARG
    assert call(4, 8, 0, 32) == _lib.ERR_INVALID_ARG


def _ptxas_accepts(kind, tmp_path):
    import shutil
    import subprocess
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc) and shutil.which(nvcc) is None:
        pytest.skip("nvcc not available")
    src = tmp_path / f"mma_{kind}.cu"
    src.write_text(
        "#include <cstdint>\n"
        "__global__ void k(uint32_t d, uint64_t a, uint64_t b, uint32_t i) {\n"
        "  asm volatile(\"{\\n\\t.reg .pred p;\\n\\tsetp.ne.b32 p, 1, 0;\\n\\t\"\n"
        f"    \"tcgen05.mma.cta_group::1.kind::{kind} [%0], %1, %2, %3, p;\\n\\t}}\"\n"
        "    :: \"r\"(d), \"l\"(a), \"l\"(b), \"r\"(i));\n}\n")
    r = subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-c", str(src),
                        "-o", str(tmp_path / f"mma_{kind}.o")], capture_output=True, text=True)
    return r.returncode == 0, r.stdout + r.stderr


def test_sm103a_has_no_int8_tensor_core_mma(tmp_path):
    # The dense path multiplies int8 weights by 0/1 spikes as exact fp16 x fp16 products
    # (kind::f16) because GB300's sm_103a has no tcgen05.mma kind::i8 form at all: ptxas
    # rejects it for this target while accepting kind::f16 and kind::f8f6f4.
    ok16, _ = _ptxas_accepts("f16", tmp_path)
    ok8, _ = _ptxas_accepts("f8f6f4", tmp_path)
    oki8, log = _ptxas_accepts("i8", tmp_path)
    assert ok16 and ok8
    assert not oki8 and "not supported" in log
