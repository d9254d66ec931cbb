// noalloc.cu -- spike attention for callers that cannot allocate device memory.
//
// nmdlm_spike_attention stages its fp32 attention currents in the context workspace,
// which nmdlm_ctx_create obtains with cudaMalloc.  Some callers cannot call cudaMalloc
// at all -- for example a host framework whose own allocator owns every byte of device
// memory, or an embedded runtime with a fixed device-memory budget -- so they cannot
// create a context.  This entry point runs the same kernels without a context: the
// currents live in the file-scope array below, which every GPU that loads the library
// holds until the process exits.
#include <mutex>

#include "internal.h"

namespace {

// Largest B * T * H * d_head the array holds: 1,048,576 floats (4 MiB per device).
constexpr size_t kNoAllocMaxCurrents = size_t(1) << 20;
constexpr int kMaxDevices = 64;

__device__ __align__(256) float g_attn_currents[kNoAllocMaxCurrents];

// Device address of the array, resolved once per device with that device current.
float* g_scratch_ptr[kMaxDevices] = {nullptr};
std::mutex g_scratch_mutex;

nmdlm_status scratch_for_current_device(float** out) {
    int dev = 0;
    if (nmdlm::cuda_status(cudaGetDevice(&dev)) != NMDLM_OK) return NMDLM_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return NMDLM_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        if (nmdlm::cuda_status(cudaGetSymbolAddress(&p, g_attn_currents)) != NMDLM_OK)
            return NMDLM_ERR_CUDA;
        g_scratch_ptr[dev] = static_cast<float*>(p);
    }
    *out = g_scratch_ptr[dev];
    return NMDLM_OK;
}

}  // namespace

extern "C" size_t nmdlm_spike_attention_noalloc_max(void) { return kNoAllocMaxCurrents; }

extern "C" nmdlm_status nmdlm_spike_attention_noalloc(
    const uint32_t* q_bits, const uint32_t* k_bits, const uint32_t* v_bits, int T, int B,
    int L_keys, int L_stride, int H, int d_head, float alpha, float theta,
    uint32_t* spikes_out, uint32_t* col_masks_out, uint32_t* active_mask_out, void* stream) {
    using namespace nmdlm;
    if (!q_bits || !k_bits || !v_bits || !spikes_out) return NMDLM_ERR_INVALID_ARG;
    if (T < 1 || B < 1 || H < 1 || d_head < 1 || L_keys < 1 || L_stride < L_keys)
        return NMDLM_ERR_INVALID_ARG;
    // B T <= 256 and H d_head <= 2^20, checked without overflowing int
    if (d_head % 32 || T > 32 || B > 256 / T || H > (1 << 20) / d_head)
        return NMDLM_ERR_UNSUPPORTED;
    if ((size_t)B * T * H * d_head > kNoAllocMaxCurrents) return NMDLM_ERR_UNSUPPORTED;
    float* cur = nullptr;
    nmdlm_status st = scratch_for_current_device(&cur);
    if (st != NMDLM_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    // Every element of the array this call reads is first written by this call, so
    // nothing has to be cleared between calls.
    AttnArgs aa{q_bits, k_bits, v_bits, T, B, L_keys, L_stride, H, d_head, alpha, cur, nullptr};
    st = launch_attention_best(aa, s);
    if (st != NMDLM_OK) return st;
    IfArgs ia{};
    ia.B = B;
    ia.T = T;
    ia.N = H * d_head;
    ia.src_kind = 0;
    ia.cur_f = cur;
    ia.theta_f = theta;
    ia.bits = spikes_out;
    ia.cm = col_masks_out;
    ia.mask = active_mask_out;
    ia.err = nullptr;
    return launch_if(nullptr, ia, s);
}
