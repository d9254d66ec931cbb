// api.cu -- the C ABI (include/nmdlm.h): context, argument checks, composition of
// the kernels into a layer, a denoising step and a context (commit) pass.
#include <algorithm>
#include <atomic>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <tuple>
#include <vector>

#include "internal.h"

using namespace nmdlm;

namespace nmdlm {
nmdlm_status launch_fill_i32(int* p, int n, int v, cudaStream_t stream);
static std::atomic<unsigned long long> g_launches{0};
void count_launch(unsigned n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
static thread_local const char* g_last_cuda_error = "no error";
void note_cuda_error(cudaError_t e) {
    g_last_cuda_error = cudaGetErrorString(e);
    cudaGetLastError();
}

static std::mutex g_attr_mutex;
static std::map<std::pair<const void*, int>, size_t> g_dyn_smem;
static std::map<std::tuple<const void*, int, size_t>, std::vector<int>> g_clusters;

nmdlm_status ensure_dyn_smem(const void* func, size_t bytes) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return NMDLM_ERR_CUDA;
    }
    std::lock_guard<std::mutex> lock(g_attr_mutex);
    size_t& granted = g_dyn_smem[{func, dev}];
    if (bytes <= granted) return NMDLM_OK;
    if (cuda_status(cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)bytes)) != NMDLM_OK)
        return NMDLM_ERR_CUDA;
    granted = bytes;
    return NMDLM_OK;
}

nmdlm_status cluster_capacity(const void* func, int threads, size_t smem, int sm_count,
                              int out[9]) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return NMDLM_ERR_CUDA;
    }
    std::lock_guard<std::mutex> lock(g_attr_mutex);
    auto key = std::make_tuple(func, dev, smem);
    auto it = g_clusters.find(key);
    if (it == g_clusters.end()) {
        std::vector<int> caps(9, 0);
        for (int n = 1; n <= 8; ++n) {
            cudaLaunchConfig_t q = {};
            q.gridDim = dim3(1, n, 1);
            q.blockDim = dim3(threads, 1, 1);
            q.dynamicSmemBytes = smem;
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = 1;
            at[0].val.clusterDim.y = n;
            at[0].val.clusterDim.z = 1;
            q.attrs = at;
            q.numAttrs = 1;
            int c = 0;
            if (cudaOccupancyMaxActiveClusters(&c, func, &q) != cudaSuccess) {
                cudaGetLastError();
                c = n == 1 ? sm_count : 0;
            }
            caps[n] = c;
        }
        it = g_clusters.emplace(key, caps).first;
    }
    for (int n = 0; n <= 8; ++n) out[n] = it->second[n];
    return NMDLM_OK;
}
}

struct nmdlm_model {
    nmdlm_ctx* ctx;
    nmdlm_model_desc d;
    std::vector<nmdlm_layer_w> layers;
    const float* tok_emb;
    const float* pos_emb;
    nmdlm_linear_w head;
};

namespace {

constexpr size_t kDefaultWorkspace = size_t(512) << 20;
constexpr size_t kCounters = 1 << 16;
// split-K partial sums of the spiking linear: 128 rows x 131072 (splits x output
// channels) of int32
constexpr size_t kAccBytes = size_t(128) * 131072 * sizeof(int32_t);
constexpr size_t kProfSlots = 1 << 14;

struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) cudaSetDevice(dev);
    }
    ~DeviceGuard() {
        int cur;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

inline cudaStream_t S(void* s) { return reinterpret_cast<cudaStream_t>(s); }


// Profiling: bracket one spiking-linear launch with events and record its shape.
struct ProfScope {
    nmdlm_ctx* c;
    cudaStream_t s;
    size_t slot = (size_t)-1;
    ProfScope(nmdlm_ctx* ctx, cudaStream_t st) : c(ctx), s(st) {
        if (!c->profiling || c->ev_used + 2 > c->ev_pool.size()) return;
        slot = c->ev_used / 2;
        cudaEventRecord(c->ev_pool[c->ev_used], s);
    }
    void finish(const LinArgs& a) {
        if (slot == (size_t)-1) return;
        cudaEventRecord(c->ev_pool[c->ev_used + 1], s);
        c->ev_used += 2;
        long long dout = 0;
        double extra = 0;
        for (int i = 0; i < a.nseg; ++i) {
            dout += a.seg[i].n_out;
            extra += 4.0 * a.seg[i].n_out;  // scales
            if (a.seg[i].res) extra += 4.0 * a.BT * a.seg[i].n_out;
            if (a.seg[i].cur) extra += 4.0 * (a.kind == EPI_KIND_LOGITS ? a.B : a.BT) * a.seg[i].n_out;
            if (a.seg[i].acc_out) extra += 4.0 * a.BT * a.seg[i].n_out;
            if (a.kind != EPI_KIND_LOGITS && a.seg[i].bits)
                extra += a.BT * (double)a.seg[i].n_out / 8.0;
        }
        extra += (double)a.d_in * a.BTW * 4.0 + words_of(a.d_in) * 4.0;  // spike block in
        c->prof_bytes_static.push_back(extra);
        c->prof_dout.push_back(dout);
        c->prof_din.push_back(a.d_in);
        c->prof_bt.push_back(a.BT);
        unsigned long long* st = c->prof_stats + 2 * slot;
        cudaMemsetAsync(st, 0, 16, s);
        launch_linear_stats(a.in_cm, a.in_mask, a.d_in, a.BTW, a.dense, (unsigned long long)dout,
                            st, s);
        if (std::find(c->prof_streams.begin(), c->prof_streams.end(), s) == c->prof_streams.end())
            c->prof_streams.push_back(s);
    }
};

nmdlm_status run_linear(nmdlm_ctx* c, LinArgs& a, WsCursor ws, cudaStream_t s) {
    ProfScope p(c, s);
    nmdlm_status st = launch_linear(c, a, c->impl, ws, s);
    if (st == NMDLM_OK) p.finish(a);
    return st;
}

void fill_seg_defaults(LinSeg& g) { std::memset(&g, 0, sizeof(g)); }

}  // namespace

// ===================================================================== basics
extern "C" const char* nmdlm_status_string(nmdlm_status s) {
    switch (s) {
        case NMDLM_OK: return "ok";
        case NMDLM_ERR_INVALID_ARG: return "invalid argument";
        case NMDLM_ERR_UNSUPPORTED: return "unsupported size";
        case NMDLM_ERR_CUDA: return "CUDA error";
        case NMDLM_ERR_TIMEOUT: return "device wait timed out";
        case NMDLM_ERR_WORKSPACE: return "workspace too small";
    }
    return "unknown status";
}

extern "C" int nmdlm_abi_version(void) { return NMDLM_ABI_VERSION; }

extern "C" uint64_t nmdlm_launch_count(void) { return g_launches.load(); }

extern "C" const char* nmdlm_last_cuda_error(void) { return g_last_cuda_error; }

extern "C" nmdlm_status nmdlm_ctx_create(nmdlm_ctx** out, int device, size_t workspace_bytes) {
    if (!out) return NMDLM_ERR_INVALID_ARG;
    *out = nullptr;
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev)
        return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(device);
    nmdlm_ctx* c = new (std::nothrow) nmdlm_ctx();
    if (!c) return NMDLM_ERR_CUDA;
    c->device = device;
    cudaDeviceGetAttribute(&c->sm_count, cudaDevAttrMultiProcessorCount, device);
    c->ws_bytes = workspace_bytes ? workspace_bytes : kDefaultWorkspace;
    bool ok = cudaMalloc(&c->ws, c->ws_bytes) == cudaSuccess &&
              cudaMalloc(&c->err, sizeof(int)) == cudaSuccess &&
              cudaMalloc(&c->counters, kCounters * sizeof(unsigned)) == cudaSuccess &&
              cudaMalloc(&c->prof_stats, 2 * kProfSlots * sizeof(unsigned long long)) == cudaSuccess &&
              cudaMalloc(&c->dbg, 4096 * sizeof(unsigned long long)) == cudaSuccess &&
              cudaMalloc(&c->acc, kAccBytes) == cudaSuccess;
    c->acc_bytes = kAccBytes;
    if (ok) {
        c->n_counters = kCounters;
        ok = cudaMemset(c->err, 0, sizeof(int)) == cudaSuccess &&
             cudaMemset(c->counters, 0, kCounters * sizeof(unsigned)) == cudaSuccess &&
             cudaDeviceSynchronize() == cudaSuccess;
    }
    if (!ok) {
        nmdlm_ctx_destroy(c);
        return NMDLM_ERR_CUDA;
    }
    *out = c;
    return NMDLM_OK;
}

extern "C" nmdlm_status nmdlm_ctx_destroy(nmdlm_ctx* c) {
    if (!c) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    cudaDeviceSynchronize();
    for (cudaEvent_t e : c->ev_pool) cudaEventDestroy(e);
    cudaFree(c->ws);
    cudaFree(c->err);
    cudaFree(c->counters);
    cudaFree(c->prof_stats);
    cudaFree(c->dbg);
    cudaFree(c->acc);
    delete c;
    return NMDLM_OK;
}

extern "C" nmdlm_status nmdlm_ctx_sync_status(nmdlm_ctx* c, void* stream) {
    if (!c) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    if (cuda_status(cudaStreamSynchronize(S(stream))) != NMDLM_OK) return NMDLM_ERR_CUDA;
    int e = 0;
    if (cudaMemcpy(&e, c->err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
        return NMDLM_ERR_CUDA;
    if (e && cudaMemset(c->err, 0, sizeof(int)) != cudaSuccess) return NMDLM_ERR_CUDA;
    if (e & ERRBIT_TIMEOUT) return NMDLM_ERR_TIMEOUT;
    if (e & ERRBIT_VALUE) return NMDLM_ERR_INVALID_ARG;
    return NMDLM_OK;
}

extern "C" nmdlm_status nmdlm_ctx_set_impl(nmdlm_ctx* c, nmdlm_impl impl) {
    if (!c || impl < NMDLM_IMPL_AUTO || impl > NMDLM_IMPL_TC) return NMDLM_ERR_INVALID_ARG;
    c->impl = impl;
    return NMDLM_OK;
}

extern "C" nmdlm_status nmdlm_ctx_set_wait_limit(nmdlm_ctx* c, uint64_t ns) {
    if (!c) return NMDLM_ERR_INVALID_ARG;
    c->wait_ns = ns;
    return NMDLM_OK;
}

// Not part of the public header: debug knob for tests of the MMA descriptor layout.
extern "C" nmdlm_status nmdlm_debug_set(nmdlm_ctx* c, int key, int value) {
    if (!c) return NMDLM_ERR_INVALID_ARG;
    if (key == 1) c->desc_swap = value;
    else if (key == 2) {
        c->dbg_on = value;
        if (value) {  // a fresh record
            DeviceGuard g(c->device);
            if (cudaMemset(c->dbg, 0, 4096 * sizeof(unsigned long long)) != cudaSuccess)
                return NMDLM_ERR_CUDA;
        }
    }
    else if (key == 4) { c->dbg_shape = value; c->dbg_count = 0; }
    else if (key == 5) { c->dbg_nth = value; c->dbg_count = 0; }
    else if (key == 3) c->split_force = value;
    else if (key == 6) c->plan_tile = value;
    else if (key == 7) c->plan_ns = value;
    else if (key == 8) c->mode_force = value;
    else return NMDLM_ERR_INVALID_ARG;
    return NMDLM_OK;
}

// Not part of the public header: copy the debug timestamps to the host.
extern "C" nmdlm_status nmdlm_debug_read(nmdlm_ctx* c, unsigned long long* host, int n) {
    if (!c || !host || n < 0 || n > 4096) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    return cuda_status(cudaMemcpy(host, c->dbg, n * sizeof(unsigned long long),
                                  cudaMemcpyDeviceToHost));
}

extern "C" nmdlm_status nmdlm_debug_wait_test(nmdlm_ctx* c, uint64_t ns, void* stream) {
    if (!c) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    return launch_wait_test(c, ns, S(stream));
}

extern "C" nmdlm_status nmdlm_ctx_set_profiling(nmdlm_ctx* c, int enable) {
    if (!c) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    if (enable && c->ev_pool.empty()) {
        c->ev_pool.resize(2 * kProfSlots);
        for (auto& e : c->ev_pool)
            if (cudaEventCreate(&e) != cudaSuccess) return NMDLM_ERR_CUDA;
    }
    c->profiling = enable ? 1 : 0;
    return NMDLM_OK;
}

extern "C" nmdlm_status nmdlm_ctx_profile_read(nmdlm_ctx* c, uint64_t* launches,
                                               double* total_ms, double* total_bytes,
                                               double* rows_fetched) {
    if (!c) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    for (cudaStream_t s : c->prof_streams)
        if (cudaStreamSynchronize(s) != cudaSuccess) return NMDLM_ERR_CUDA;
    const size_t n = c->ev_used / 2;
    std::vector<unsigned long long> st(2 * std::max<size_t>(n, 1));
    if (n && cudaMemcpy(st.data(), c->prof_stats, 2 * n * sizeof(unsigned long long),
                        cudaMemcpyDeviceToHost) != cudaSuccess)
        return NMDLM_ERR_CUDA;
    double ms = 0, bytes = 0, rows = 0;
    for (size_t i = 0; i < n; ++i) {
        float t = 0;
        if (cudaEventElapsedTime(&t, c->ev_pool[2 * i], c->ev_pool[2 * i + 1]) != cudaSuccess)
            return NMDLM_ERR_CUDA;
        ms += t;
        bytes += (double)st[2 * i] * (double)c->prof_dout[i] + c->prof_bytes_static[i];
        rows += (double)st[2 * i];
    }
    if (launches) *launches = n;
    if (total_ms) *total_ms = ms;
    if (total_bytes) *total_bytes = bytes;
    if (rows_fetched) *rows_fetched = rows;
    c->ev_used = 0;
    c->prof_bytes_static.clear();
    c->prof_dout.clear();
    c->prof_din.clear();
    c->prof_bt.clear();
    c->prof_streams.clear();
    return NMDLM_OK;
}

extern "C" nmdlm_status nmdlm_ctx_profile_launches(nmdlm_ctx* c, int max_launches,
                                                   double* out, int* n_out) {
    if (!c || !n_out || max_launches < 0 || (max_launches > 0 && !out))
        return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    for (cudaStream_t s : c->prof_streams)
        if (cudaStreamSynchronize(s) != cudaSuccess) return NMDLM_ERR_CUDA;
    const size_t n = std::min<size_t>(c->ev_used / 2, (size_t)max_launches);
    std::vector<unsigned long long> st(2 * std::max<size_t>(n, 1));
    if (n && cudaMemcpy(st.data(), c->prof_stats, 2 * n * sizeof(unsigned long long),
                        cudaMemcpyDeviceToHost) != cudaSuccess)
        return NMDLM_ERR_CUDA;
    for (size_t i = 0; i < n; ++i) {
        float t = 0;
        if (cudaEventElapsedTime(&t, c->ev_pool[2 * i], c->ev_pool[2 * i + 1]) != cudaSuccess)
            return NMDLM_ERR_CUDA;
        double* r = out + 6 * i;
        r[0] = t;
        r[1] = (double)st[2 * i];
        r[2] = (double)st[2 * i + 1];
        r[3] = c->prof_din[i];
        r[4] = (double)c->prof_dout[i];
        r[5] = c->prof_bt[i];
    }
    *n_out = (int)n;
    return NMDLM_OK;
}

// ===================================================================== pack / IF
extern "C" nmdlm_status nmdlm_pack_spikes(nmdlm_ctx* c, const uint8_t* spikes, int BT, int D,
                                          uint32_t* row_bits, uint32_t* col_masks,
                                          uint32_t* active_mask, int32_t* active_idx,
                                          int32_t* n_active, void* stream) {
    if (!c || !spikes || !row_bits || BT < 1 || D < 1) return NMDLM_ERR_INVALID_ARG;
    if (BT > 256) return NMDLM_ERR_UNSUPPORTED;
    if ((active_idx || n_active) && !active_mask) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    return launch_pack(c, spikes, BT, D, row_bits, col_masks, active_mask, active_idx, n_active,
                       S(stream));
}

extern "C" nmdlm_status nmdlm_if_neuron(nmdlm_ctx* c, const void* current, nmdlm_dtype dt,
                                        int B, int T, int N, int32_t threshold_i,
                                        float threshold_f, void* v_state, uint32_t* spikes_out,
                                        uint32_t* col_masks_out, uint32_t* active_mask_out,
                                        void* stream) {
    if (!c || !current || !spikes_out || B < 1 || T < 1 || N < 1) return NMDLM_ERR_INVALID_ARG;
    if (dt != NMDLM_I32 && dt != NMDLM_F32) return NMDLM_ERR_INVALID_ARG;
    if (T > 32 || B > 256 / T) return NMDLM_ERR_UNSUPPORTED;  // B T <= 256, without overflow
    DeviceGuard g(c->device);
    IfArgs a{};
    a.B = B; a.T = T; a.N = N;
    a.src_kind = dt == NMDLM_I32 ? 1 : 0;
    a.cur_f = (const float*)current;
    a.cur_i = (const int32_t*)current;
    a.theta_f = threshold_f;
    a.theta_i = threshold_i;
    a.v_state = v_state;
    a.bits = spikes_out;
    a.cm = col_masks_out;
    a.mask = active_mask_out;
    a.err = c->err;
    return launch_if(c, a, S(stream));
}

// ===================================================================== linear
// The spiking linear after argument checks; `ws` is the workspace still free (a
// caller that carved buffers out of the workspace passes its advanced cursor).
static nmdlm_status spike_linear_impl(nmdlm_ctx* c, const nmdlm_spikes* in, const int8_t* wT,
                                      const float* scale, int d_in, int d_out,
                                      nmdlm_mode mode, int32_t* acc_out,
                                      const nmdlm_if_epilogue* epi, uint64_t* stats,
                                      WsCursor ws, cudaStream_t stream);

extern "C" nmdlm_status nmdlm_spike_linear(nmdlm_ctx* c, const nmdlm_spikes* in,
                                           const int8_t* wT, const float* scale, int d_in,
                                           int d_out, nmdlm_mode mode, int32_t* acc_out,
                                           const nmdlm_if_epilogue* epi, uint64_t* stats,
                                           void* stream) {
    if (!c || !in || !wT || d_in < 1 || d_out < 1) return NMDLM_ERR_INVALID_ARG;
    if (!in->col_masks || !in->active_mask || in->D != d_in) return NMDLM_ERR_INVALID_ARG;
    if (in->BT < 1 || in->T < 1 || in->BT % in->T) return NMDLM_ERR_INVALID_ARG;
    if (in->T > 32 || in->BT > 256) return NMDLM_ERR_UNSUPPORTED;
    if (!acc_out && !epi) return NMDLM_ERR_INVALID_ARG;
    if (mode < NMDLM_MODE_AUTO || mode > NMDLM_MODE_DENSE) return NMDLM_ERR_INVALID_ARG;
    if (epi) {
        if (!epi->spikes_out) return NMDLM_ERR_INVALID_ARG;
        if (epi->kind != NMDLM_IF_INT && epi->kind != NMDLM_IF_FP32) return NMDLM_ERR_INVALID_ARG;
        if ((epi->kind == NMDLM_IF_FP32 || epi->current_out) && !scale) return NMDLM_ERR_INVALID_ARG;
        if (epi->kind == NMDLM_IF_INT && (epi->residual_in || epi->gate_bits))
            return NMDLM_ERR_INVALID_ARG;
    }
    DeviceGuard g(c->device);
    return spike_linear_impl(c, in, wT, scale, d_in, d_out, mode, acc_out, epi, stats, WsCursor(c),
                             S(stream));
}

static nmdlm_status spike_linear_impl(nmdlm_ctx* c, const nmdlm_spikes* in, const int8_t* wT,
                                      const float* scale, int d_in, int d_out,
                                      nmdlm_mode mode, int32_t* acc_out,
                                      const nmdlm_if_epilogue* epi, uint64_t* stats,
                                      WsCursor ws, cudaStream_t stream) {
    uint32_t* tmp_bits = nullptr;
    LinArgs a;
    std::memset(&a, 0, sizeof(a));
    a.in_cm = in->col_masks;
    a.in_mask = in->active_mask;
    a.in_rows = in->row_bits;
    a.d_in = d_in;
    a.BT = in->BT;
    a.T = in->T;
    a.B = in->BT / in->T;
    a.BTW = words_of(in->BT);
    a.nseg = 1;
    a.dense = mode == NMDLM_MODE_DENSE;
    a.auto_dense = mode == NMDLM_MODE_AUTO;
    LinSeg& s = a.seg[0];
    fill_seg_defaults(s);
    s.wT = wT;
    s.scale = scale;
    s.ld_w = d_out;
    s.n_out = d_out;
    s.acc_out = acc_out;
    s.sb = (long long)a.T * words_of(d_out);
    s.st = words_of(d_out);
    if (epi) {
        a.kind = epi->kind == NMDLM_IF_INT ? EPI_KIND_INT : EPI_KIND_F32;
        a.theta_i = epi->threshold_i;
        a.theta_f = epi->threshold_f;
        s.bits = epi->spikes_out;
        s.cm = epi->col_masks_out;
        s.mask = epi->active_mask_out;
        s.cur = epi->current_out;
        s.res = epi->residual_in;
        s.gate = epi->gate_bits;
    } else {
        // integer sums only: spikes of an (unused) integer IF go to scratch
        a.kind = EPI_KIND_INT;
        a.theta_i = 0x7fffffff;
        tmp_bits = ws.take<uint32_t>((size_t)a.BT * words_of(d_out));
        if (!tmp_bits) return NMDLM_ERR_WORKSPACE;
        s.bits = tmp_bits;
    }
    nmdlm_status st = run_linear(c, a, ws, stream);
    if (st == NMDLM_OK && stats)
        st = launch_linear_stats(a.in_cm, a.in_mask, d_in, a.BTW, a.dense,
                                 (unsigned long long)d_out, (unsigned long long*)stats,
                                 stream);
    return st;
}

// ===================================================================== ternary coding
static bool ternary_args_ok(float K, int T) {
    return K > 0.0f && K < INFINITY && T >= 1 && T <= 24;
}

extern "C" nmdlm_status nmdlm_ternary_encode(nmdlm_ctx* c, const float* a, int N, int D,
                                             float K, int T, uint8_t* plus_out,
                                             uint8_t* minus_out, int32_t* ahat_out,
                                             float* vth_out, void* stream) {
    if (!c || !a || !plus_out || !minus_out || N < 1 || D < 1 || !ternary_args_ok(K, T))
        return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    return launch_ternary_encode(a, N, D, K, T, T, plus_out, minus_out, ahat_out, vth_out,
                                 S(stream));
}

extern "C" nmdlm_status nmdlm_ternary_combine(nmdlm_ctx* c, const int32_t* acc_plus,
                                              const int32_t* acc_minus, int N, int T,
                                              int d_out, int32_t* y_out, void* stream) {
    if (!c || !acc_plus || !acc_minus || !y_out || N < 1 || d_out < 1 || T < 1 || T > 24)
        return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    return launch_ternary_combine(acc_plus, acc_minus, N, T, T, d_out, y_out, S(stream));
}

extern "C" nmdlm_status nmdlm_ternary_if(nmdlm_ctx* c, const int32_t* y, int N, int d_out,
                                         int T, int theta, int8_t* spikes_out,
                                         int32_t* v_out, void* stream) {
    if (!c || !y || !spikes_out || N < 1 || d_out < 1 || T < 1 || T > 24 || theta < 1)
        return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    return launch_ternary_if(y, N, d_out, T, theta, spikes_out, v_out, S(stream));
}

extern "C" nmdlm_status nmdlm_ternary_linear(nmdlm_ctx* c, const float* a, int N, int D,
                                             float K, int T, const int8_t* wT, int d_out,
                                             nmdlm_mode mode, int32_t* y_out,
                                             int32_t* ahat_out, float* vth_out, void* stream) {
    if (!c || !a || !wT || !y_out || N < 1 || D < 1 || d_out < 1 || !ternary_args_ok(K, T))
        return NMDLM_ERR_INVALID_ARG;
    if (mode < NMDLM_MODE_AUTO || mode > NMDLM_MODE_DENSE) return NMDLM_ERR_INVALID_ARG;
    if (N > 256) return NMDLM_ERR_UNSUPPORTED;  // before N * T can overflow
    const int BT = N * T;
    if (BT > 256 || 127.0 * (double)((1 << T) - 1) * (double)D >= 2147483648.0)
        return NMDLM_ERR_UNSUPPORTED;
    DeviceGuard g(c->device);
    cudaStream_t s = S(stream);
    WsCursor ws(c);
    const int DW = words_of(D);
    // One block of 2 N T rows: row n * 2T + t-1 the +1 spikes of plane t, row
    // n * 2T + T + t-1 the -1 spikes, so one launch of the spiking linear streams the
    // weights once for both planes (a row of W^T is fetched when either plane spikes in
    // it).  The stacked block must fit the tensor-memory kernel's 128 rows: a 256-row
    // block on the older 256-row kernel measured 115 us against 88 us for two 128-row
    // launches (16 x 4096 -> 11008, T 8), so larger blocks take the planes as two.
    if (2 * BT <= 128) {
        const int R = 2 * BT, RW = words_of(R);
        uint8_t* planes = ws.take<uint8_t>((size_t)R * D);
        uint32_t* rb = ws.take<uint32_t>((size_t)R * DW);
        uint32_t* cm = ws.take<uint32_t>((size_t)D * RW);
        uint32_t* am = ws.take<uint32_t>((size_t)DW);
        int32_t* acc = ws.take<int32_t>((size_t)R * d_out);
        if (!planes || !rb || !cm || !am || !acc) return NMDLM_ERR_WORKSPACE;
        nmdlm_status st = launch_ternary_encode(a, N, D, K, T, 2 * T, planes,
                                                planes + (size_t)T * D, ahat_out, vth_out, s);
        if (st == NMDLM_OK) st = launch_pack(c, planes, R, D, rb, cm, am, nullptr, nullptr, s);
        if (st == NMDLM_OK) {
            nmdlm_spikes in{rb, cm, am, nullptr, nullptr, R, 1, D};
            st = spike_linear_impl(c, &in, wT, nullptr, D, d_out, mode, acc, nullptr, nullptr,
                                   ws, s);
        }
        if (st == NMDLM_OK)
            st = launch_ternary_combine(acc, acc + (size_t)T * d_out, N, T, 2 * T, d_out, y_out,
                                        s);
        return st;
    }
    const int BTW = words_of(BT);
    uint8_t* planes[2];
    uint32_t *rb[2], *cm[2], *am[2];
    int32_t* acc[2];
    for (int p = 0; p < 2; ++p) {
        planes[p] = ws.take<uint8_t>((size_t)BT * D);
        rb[p] = ws.take<uint32_t>((size_t)BT * DW);
        cm[p] = ws.take<uint32_t>((size_t)D * BTW);
        am[p] = ws.take<uint32_t>((size_t)DW);
        acc[p] = ws.take<int32_t>((size_t)BT * d_out);
        if (!planes[p] || !rb[p] || !cm[p] || !am[p] || !acc[p]) return NMDLM_ERR_WORKSPACE;
    }
    nmdlm_status st = launch_ternary_encode(a, N, D, K, T, T, planes[0], planes[1], ahat_out,
                                            vth_out, s);
    for (int p = 0; p < 2 && st == NMDLM_OK; ++p)
        st = launch_pack(c, planes[p], BT, D, rb[p], cm[p], am[p], nullptr, nullptr, s);
    for (int p = 0; p < 2 && st == NMDLM_OK; ++p) {
        nmdlm_spikes in{rb[p], cm[p], am[p], nullptr, nullptr, BT, T, D};
        st = spike_linear_impl(c, &in, wT, nullptr, D, d_out, mode, acc[p], nullptr, nullptr, ws,
                               s);
    }
    if (st == NMDLM_OK) st = launch_ternary_combine(acc[0], acc[1], N, T, T, d_out, y_out, s);
    return st;
}

// ===================================================================== attention
extern "C" nmdlm_status nmdlm_spike_attention(nmdlm_ctx* c, const uint32_t* q_bits,
                                              const uint32_t* k_bits, const uint32_t* v_bits,
                                              int T, int B, int L_keys, int L_stride, int H,
                                              int d_head, float alpha, float theta,
                                              float* current_out, uint32_t* spikes_out,
                                              uint32_t* col_masks_out,
                                              uint32_t* active_mask_out, void* stream) {
    if (!c || !q_bits || !k_bits || !v_bits || !spikes_out) return NMDLM_ERR_INVALID_ARG;
    if (T < 1 || B < 1 || H < 1 || d_head < 1 || L_keys < 1 || L_stride < L_keys)
        return NMDLM_ERR_INVALID_ARG;
    // B T <= 256 and H d_head <= 2^20, checked without overflowing int
    if (d_head % 32 || T > 32 || B > 256 / T || H > (1 << 20) / d_head)
        return NMDLM_ERR_UNSUPPORTED;
    DeviceGuard g(c->device);
    WsCursor ws(c);
    const int D = H * d_head;
    float* cur = current_out ? current_out : ws.take<float>((size_t)B * T * D);
    if (!cur) return NMDLM_ERR_WORKSPACE;
    AttnArgs aa{q_bits, k_bits, v_bits, T, B, L_keys, L_stride, H, d_head, alpha, cur, c->err};
    aa.wait_ns = c->wait_ns;
    aa.dbg = c->dbg_on ? c->dbg : nullptr;
    nmdlm_status st = launch_attention_best(aa, S(stream));
    if (st != NMDLM_OK) return st;
    IfArgs ia{};
    ia.B = B; ia.T = T; ia.N = D;
    ia.src_kind = 0;
    ia.cur_f = cur;
    ia.theta_f = theta;
    ia.bits = spikes_out;
    ia.cm = col_masks_out;
    ia.mask = active_mask_out;
    ia.err = c->err;
    return launch_if(c, ia, S(stream));
}

// ===================================================================== model
static bool desc_ok(const nmdlm_model_desc* d) {
    return d && d->n_layers >= 1 && d->n_enc_layers >= 0 && d->d_model >= 32 && d->n_heads >= 1 &&
           d->d_head * d->n_heads == d->d_model && d->d_head % 32 == 0 && d->d_mlp >= 1 &&
           d->vocab >= 1 && d->T >= 1 && d->T <= 32 && d->B >= 1 && d->S >= 1 &&
           d->B % d->S == 0 && d->B * d->T <= 256 && d->max_ctx >= d->B && d->B <= 64 &&
           d->d_model % 32 == 0;
}

struct StepBufs {
    float* u[2];
    uint32_t* xb[2];
    uint32_t* xc[2];
    uint32_t* xm[2];
    uint32_t *q, *ab, *ac, *am, *x1b, *x1c, *x1m, *g, *hb, *hc, *hm;
    float *acur, *u1, *logits;
};

static bool carve_step(WsCursor& ws, const nmdlm_model_desc& d, StepBufs& b) {
    const size_t BT = (size_t)d.B * d.T, D = d.d_model, F = d.d_mlp;
    const size_t DW = words_of((int)D), FW = words_of((int)F), BTW = words_of((int)BT);
    bool ok = true;
    for (int i = 0; i < 2; ++i) {
        ok &= (b.u[i] = ws.take<float>(BT * D)) != nullptr;
        ok &= (b.xb[i] = ws.take<uint32_t>(BT * DW)) != nullptr;
        ok &= (b.xc[i] = ws.take<uint32_t>(D * BTW)) != nullptr;
        ok &= (b.xm[i] = ws.take<uint32_t>(DW)) != nullptr;
    }
    ok &= (b.q = ws.take<uint32_t>(BT * DW)) != nullptr;
    ok &= (b.ab = ws.take<uint32_t>(BT * DW)) != nullptr;
    ok &= (b.ac = ws.take<uint32_t>(D * BTW)) != nullptr;
    ok &= (b.am = ws.take<uint32_t>(DW)) != nullptr;
    ok &= (b.x1b = ws.take<uint32_t>(BT * DW)) != nullptr;
    ok &= (b.x1c = ws.take<uint32_t>(D * BTW)) != nullptr;
    ok &= (b.x1m = ws.take<uint32_t>(DW)) != nullptr;
    ok &= (b.g = ws.take<uint32_t>(BT * FW)) != nullptr;
    ok &= (b.hb = ws.take<uint32_t>(BT * FW)) != nullptr;
    ok &= (b.hc = ws.take<uint32_t>(F * BTW)) != nullptr;
    ok &= (b.hm = ws.take<uint32_t>(FW)) != nullptr;
    ok &= (b.acur = ws.take<float>(BT * D)) != nullptr;
    ok &= (b.u1 = ws.take<float>(BT * D)) != nullptr;
    ok &= (b.logits = ws.take<float>((size_t)d.B * d.vocab)) != nullptr;
    return ok;
}

extern "C" size_t nmdlm_model_workspace_bytes(const nmdlm_model_desc* d) {
    if (!desc_ok(d)) return 0;
    nmdlm_ctx fake;
    fake.ws = (void*)(uintptr_t)256;
    fake.ws_bytes = (size_t)1 << 60;
    WsCursor ws(&fake);
    StepBufs b;
    carve_step(ws, *d, b);
    ws.take<double>(d->B);
    ws.take<int>(d->B);
    // split-K partials of the largest linear (up to 32 splits of 128 x 256 tiles)
    const size_t maxout = std::max<size_t>({(size_t)d->d_model, (size_t)d->d_mlp, (size_t)d->vocab});
    const size_t tiles = (maxout + 127) / 128 * 3;
    const size_t np = d->B * d->T <= 128 ? 128 : 256;
    size_t part = std::min<size_t>(32, std::max<size_t>(1, 2 * 152 / std::max<size_t>(1, tiles / 3) + 1));
    part = part * tiles * np * 128 * 4;
    return ws.off + part + (1 << 20);
}

extern "C" nmdlm_status nmdlm_model_create(nmdlm_ctx* c, const nmdlm_model_desc* desc,
                                           const nmdlm_layer_w* layers, const float* tok_emb,
                                           const float* pos_emb, nmdlm_linear_w head,
                                           nmdlm_model** out) {
    if (!out) return NMDLM_ERR_INVALID_ARG;
    *out = nullptr;
    if (!c || !desc_ok(desc) || !layers || !tok_emb || !pos_emb || !head.wT || !head.scale)
        return NMDLM_ERR_INVALID_ARG;
    const int n_all = desc->n_enc_layers + desc->n_layers;
    for (int l = 0; l < n_all; ++l) {
        const nmdlm_layer_w& w = layers[l];
        if (!w.q.wT || !w.k.wT || !w.v.wT || !w.o.wT || !w.up.wT || !w.down.wT ||
            !w.q.scale || !w.k.scale || !w.v.scale || !w.o.scale || !w.up.scale ||
            !w.down.scale)
            return NMDLM_ERR_INVALID_ARG;
        if (desc->gated && (!w.gate.wT || !w.gate.scale)) return NMDLM_ERR_INVALID_ARG;
    }
    nmdlm_model* m = new (std::nothrow) nmdlm_model();
    if (!m) return NMDLM_ERR_CUDA;
    m->ctx = c;
    m->d = *desc;
    m->layers.assign(layers, layers + n_all);
    m->tok_emb = tok_emb;
    m->pos_emb = pos_emb;
    m->head = head;
    *out = m;
    return NMDLM_OK;
}

extern "C" nmdlm_status nmdlm_model_destroy(nmdlm_model* m) {
    if (!m) return NMDLM_ERR_INVALID_ARG;
    delete m;
    return NMDLM_OK;
}

// One linear of the layer with a single output segment.
static LinArgs layer_linear(const nmdlm_model_desc& d, const uint32_t* in_cm,
                            const uint32_t* in_mask, int d_in, const nmdlm_linear_w& w,
                            int d_out, uint32_t* bits, uint32_t* cm, uint32_t* mask,
                            const float* res, float* cur, const uint32_t* gate) {
    LinArgs a;
    std::memset(&a, 0, sizeof(a));
    a.in_cm = in_cm;
    a.in_mask = in_mask;
    a.d_in = d_in;
    a.BT = d.B * d.T;
    a.T = d.T;
    a.B = d.B;
    a.BTW = words_of(a.BT);
    a.nseg = 1;
    a.kind = EPI_KIND_F32;
    a.theta_f = d.theta;
    a.auto_dense = 1;
    LinSeg& s = a.seg[0];
    fill_seg_defaults(s);
    s.wT = w.wT;
    s.scale = w.scale;
    s.ld_w = d_out;
    s.n_out = d_out;
    s.bits = bits;
    s.sb = (long long)d.T * words_of(d_out);
    s.st = words_of(d_out);
    s.cm = cm;
    s.mask = mask;
    s.res = res;
    s.cur = cur;
    s.gate = gate;
    return a;
}

static nmdlm_status layer_forward_impl(nmdlm_ctx* c, const nmdlm_model* m, int l,
                                       const nmdlm_layer_io& io, const StepBufs& b,
                                       WsCursor ws, cudaStream_t s) {
    const nmdlm_model_desc& d = m->d;
    const nmdlm_layer_w& w = m->layers[l];
    const int D = d.d_model, F = d.d_mlp, T = d.T, B = d.B;
    const int DW = words_of(D);
    nmdlm_status st;
    uint32_t* q = io.q_bits ? io.q_bits : b.q;
    // Q, K, V: one launch, three output segments.  K and V spikes land in the caches
    // at positions ctx_len..ctx_len+B-1.
    {
        LinArgs a = layer_linear(d, io.x_col_masks, io.x_active_mask, D, w.q, D, q, nullptr,
                                 nullptr, nullptr, nullptr, nullptr);
        a.in_rows = io.x_bits;
        a.nseg = 3;
        const nmdlm_linear_w* kv[2] = {&w.k, &w.v};
        uint32_t* cache[2] = {io.k_cache, io.v_cache};
        for (int i = 0; i < 2; ++i) {
            LinSeg& g = a.seg[1 + i];
            g = a.seg[0];
            g.wT = kv[i]->wT;
            g.scale = kv[i]->scale;
            g.bits = cache[i] + (size_t)io.ctx_len * DW;
            g.sb = DW;
            g.st = (long long)d.max_ctx * DW;
        }
        if ((st = run_linear(c, a, ws, s)) != NMDLM_OK) return st;
    }
    float* acur = io.attn_current ? io.attn_current : b.acur;
    const uint32_t* ab = io.attn_bits ? io.attn_bits : b.ab;
    const uint32_t* acm = b.ac;
    const uint32_t* aam = b.am;
    if (io.attn_bits_in) {  // teacher-forced attention spikes
        ab = io.attn_bits_in;
        acm = io.attn_col_masks_in;
        aam = io.attn_active_mask_in;
    } else {
        const int L = io.ctx_len + B;
        AttnArgs aa{q, io.k_cache, io.v_cache, T, B, L, d.max_ctx, d.n_heads, d.d_head,
                    1.0f / sqrtf((float)d.d_head), acur, c->err};
        aa.wait_ns = c->wait_ns;
        if ((st = launch_attention_best(aa, s)) != NMDLM_OK) return st;
        IfArgs ia{};
        ia.B = B; ia.T = T; ia.N = D;
        ia.cur_f = acur;
        ia.theta_f = d.theta;
        ia.bits = io.attn_bits ? io.attn_bits : b.ab;
        ia.cm = b.ac;
        ia.mask = b.am;
        ia.err = c->err;
        if ((st = launch_if(c, ia, s)) != NMDLM_OK) return st;
    }
    float* u1 = io.u1 ? io.u1 : b.u1;
    uint32_t* x1b = io.x1_bits ? io.x1_bits : b.x1b;
    {
        LinArgs a = layer_linear(d, acm, aam, D, w.o, D, x1b, b.x1c, b.x1m, io.u_in, u1,
                                 nullptr);
        a.in_rows = ab;
        if ((st = run_linear(c, a, ws, s)) != NMDLM_OK) return st;
    }
    uint32_t* hb = io.h_bits ? io.h_bits : b.hb;
    bool mlp_done = false;
    if (d.gated) {
        // Gate and up in one launch when the tensor-core kernel can pair them: the gate's
        // spikes gate the up current inside the epilogue and are written only if traced.
        LinArgs a = layer_linear(d, b.x1c, b.x1m, D, w.up, F, hb, b.hc, b.hm, nullptr, nullptr,
                                 nullptr);
        a.nseg = 2;
        a.paired = 1;
        a.in_rows = x1b;
        a.seg[1] = a.seg[0];
        LinSeg& g = a.seg[0];
        fill_seg_defaults(g);
        g.wT = w.gate.wT;
        g.scale = w.gate.scale;
        g.ld_w = F;
        g.n_out = F;
        g.bits = io.g_bits;
        g.sb = (long long)d.T * words_of(F);
        g.st = words_of(F);
        st = run_linear(c, a, ws, s);
        if (st == NMDLM_OK) mlp_done = true;
        else if (st != NMDLM_ERR_UNSUPPORTED) return st;
    }
    if (!mlp_done) {
        const uint32_t* gate = nullptr;
        if (d.gated) {
            uint32_t* gb = io.g_bits ? io.g_bits : b.g;
            LinArgs a = layer_linear(d, b.x1c, b.x1m, D, w.gate, F, gb, nullptr, nullptr, nullptr,
                                     nullptr, nullptr);
            a.in_rows = x1b;
            if ((st = run_linear(c, a, ws, s)) != NMDLM_OK) return st;
            gate = gb;
        }
        LinArgs a = layer_linear(d, b.x1c, b.x1m, D, w.up, F, hb, b.hc, b.hm, nullptr, nullptr,
                                 gate);
        a.in_rows = x1b;
        if ((st = run_linear(c, a, ws, s)) != NMDLM_OK) return st;
    }
    {
        LinArgs a = layer_linear(d, b.hc, b.hm, F, w.down, D, io.x_bits_out, io.x_col_masks_out,
                                 io.x_active_mask_out, u1, io.u_out, nullptr);
        a.in_rows = hb;
        if ((st = run_linear(c, a, ws, s)) != NMDLM_OK) return st;
    }
    return NMDLM_OK;
}

extern "C" nmdlm_status nmdlm_layer_forward(nmdlm_ctx* c, const nmdlm_model* m, int layer,
                                            const nmdlm_layer_io* io, void* stream) {
    if (!c || !m || !io || layer < 0 || layer >= m->d.n_enc_layers + m->d.n_layers)
        return NMDLM_ERR_INVALID_ARG;
    if (!io->x_col_masks || !io->x_active_mask || !io->u_in || !io->k_cache || !io->v_cache ||
        !io->x_bits_out || !io->x_col_masks_out || !io->x_active_mask_out || !io->u_out)
        return NMDLM_ERR_INVALID_ARG;
    if (io->ctx_len < 0 || io->ctx_len + m->d.B > m->d.max_ctx) return NMDLM_ERR_INVALID_ARG;
    if (io->attn_bits_in && (!io->attn_col_masks_in || !io->attn_active_mask_in))
        return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    WsCursor ws(c);
    StepBufs b;
    if (!carve_step(ws, m->d, b)) return NMDLM_ERR_WORKSPACE;
    return layer_forward_impl(c, m, layer, *io, b, ws, S(stream));
}

static nmdlm_status run_block_pass(nmdlm_ctx* c, const nmdlm_model* m, nmdlm_block_state* st,
                                   bool commit, int32_t* unmasked_out, float* logits_out,
                                   cudaStream_t s) {
    const nmdlm_model_desc& d = m->d;
    WsCursor ws(c);
    StepBufs b;
    if (!carve_step(ws, d, b)) return NMDLM_ERR_WORKSPACE;
    const int D = d.d_model, DW = words_of(D);
    const size_t layer_cache = (size_t)d.T * d.max_ctx * DW;
    nmdlm_status r;
    // embedding currents (constant over T) -> IF -> the first layer's input block
    IfArgs ia{};
    ia.B = d.B; ia.T = d.T; ia.N = D;
    ia.src_kind = 2;
    ia.tokens = st->tokens;
    ia.tok_emb = m->tok_emb;
    ia.pos_emb = m->pos_emb;
    ia.pos0 = st->ctx_len;
    ia.vocab = d.vocab;
    ia.theta_f = d.theta;
    ia.bits = b.xb[0];
    ia.cm = b.xc[0];
    ia.mask = b.xm[0];
    ia.cur_out = b.u[0];
    ia.err = c->err;
    if ((r = launch_if(c, ia, s)) != NMDLM_OK) return r;
    int cur = 0;
    // Sec. III-A: a shared-layer model runs every layer in both passes; an
    // encoder-decoder model its encoders on the context pass, its decoders on the steps.
    int first = 0, count = d.n_layers;
    if (d.n_enc_layers > 0 && commit) count = d.n_enc_layers;
    if (d.n_enc_layers > 0 && !commit) first = d.n_enc_layers;
    for (int l = first; l < first + count; ++l) {
        nmdlm_layer_io io{};
        io.x_bits = b.xb[cur];
        io.x_col_masks = b.xc[cur];
        io.x_active_mask = b.xm[cur];
        io.u_in = b.u[cur];
        io.k_cache = st->k_cache + l * layer_cache;
        io.v_cache = st->v_cache + l * layer_cache;
        io.ctx_len = st->ctx_len;
        io.x_bits_out = b.xb[cur ^ 1];
        io.x_col_masks_out = b.xc[cur ^ 1];
        io.x_active_mask_out = b.xm[cur ^ 1];
        io.u_out = b.u[cur ^ 1];
        if ((r = layer_forward_impl(c, m, l, io, b, ws, s)) != NMDLM_OK) return r;
        cur ^= 1;
    }
    if (commit && d.n_enc_layers > 0) {
        // Eq. (5): h^b = the encoder's output for the block; each decoder layer's K and V
        // spikes of it, one two-segment launch per decoder layer, into the decoder caches
        for (int l = 0; l < d.n_layers; ++l) {
            const int ld = d.n_enc_layers + l;
            const nmdlm_layer_w& w = m->layers[ld];
            LinArgs a = layer_linear(d, b.xc[cur], b.xm[cur], D, w.k, D,
                                     st->k_cache + ld * layer_cache + (size_t)st->ctx_len * DW,
                                     nullptr, nullptr, nullptr, nullptr, nullptr);
            a.in_rows = b.xb[cur];
            a.nseg = 2;
            LinSeg& g = a.seg[1];
            g = a.seg[0];
            g.wT = w.v.wT;
            g.scale = w.v.scale;
            g.bits = st->v_cache + ld * layer_cache + (size_t)st->ctx_len * DW;
            for (int i = 0; i < 2; ++i) {
                a.seg[i].sb = DW;
                a.seg[i].st = (long long)d.max_ctx * DW;
            }
            if ((r = run_linear(c, a, ws, s)) != NMDLM_OK) return r;
        }
    }
    if (commit) return NMDLM_OK;
    float* logits = logits_out ? logits_out : b.logits;
    {
        LinArgs a = layer_linear(d, b.xc[cur], b.xm[cur], D, m->head, d.vocab, nullptr, nullptr,
                                 nullptr, nullptr, logits, nullptr);
        a.kind = EPI_KIND_LOGITS;
        a.in_rows = b.xb[cur];
        if ((r = run_linear(c, a, ws, s)) != NMDLM_OK) return r;
    }
    return launch_head_unmask(c, logits, d.B, d.vocab, d.B / d.S, st->tokens, st->mask,
                              unmasked_out, ws, s);
}

extern "C" nmdlm_status nmdlm_block_denoise_step(nmdlm_ctx* c, const nmdlm_model* m,
                                                 nmdlm_block_state* st, int32_t* unmasked_out,
                                                 float* logits_out, void* stream) {
    if (!c || !m || !st || !st->tokens || !st->mask || !st->k_cache || !st->v_cache)
        return NMDLM_ERR_INVALID_ARG;
    if (st->step < 0 || st->step >= m->d.S) return NMDLM_ERR_INVALID_ARG;
    if (st->ctx_len < 0 || st->ctx_len + m->d.B > m->d.max_ctx) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    nmdlm_status r = run_block_pass(c, m, st, false, unmasked_out, logits_out, S(stream));
    if (r == NMDLM_OK) st->step += 1;
    return r;
}

extern "C" nmdlm_status nmdlm_block_commit(nmdlm_ctx* c, const nmdlm_model* m,
                                           nmdlm_block_state* st, void* stream) {
    if (!c || !m || !st || !st->tokens || !st->mask || !st->k_cache || !st->v_cache)
        return NMDLM_ERR_INVALID_ARG;
    if (st->ctx_len < 0 || st->ctx_len + m->d.B > m->d.max_ctx) return NMDLM_ERR_INVALID_ARG;
    DeviceGuard g(c->device);
    nmdlm_status r = run_block_pass(c, m, st, true, nullptr, nullptr, S(stream));
    if (r != NMDLM_OK) return r;
    if ((r = launch_fill_i32(st->tokens, m->d.B, m->d.vocab, S(stream))) != NMDLM_OK) return r;
    if ((r = launch_fill_i32(st->mask, m->d.B, 1, S(stream))) != NMDLM_OK) return r;
    st->ctx_len += m->d.B;
    st->step = 0;
    return NMDLM_OK;
}
