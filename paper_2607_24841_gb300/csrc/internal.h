// internal.h -- host-side declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>

#include <vector>

#include "common.cuh"

// counters[kLinTicketBase, kLinTicketBase + 2 * tiles): the spiking linear's per-tile
// arrival / departure counters of the slot split-K (below: the head's counters).
constexpr size_t kLinTicketBase = 8192;

struct nmdlm_ctx {
    int device = 0;
    int sm_count = 0;
    void* ws = nullptr;            // general workspace
    size_t ws_bytes = 0;
    int* err = nullptr;            // device error word
    unsigned int* counters = nullptr;  // split-K arrival counters (zero between launches)
    size_t n_counters = 0;
    unsigned long long* prof_stats = nullptr;  // device {rows, sops} for profiling
    int32_t* acc = nullptr;        // split-K partial sums of the spiking linear
    size_t acc_bytes = 0;
    unsigned long long wait_ns = 1000000000ull;
    nmdlm_impl impl = NMDLM_IMPL_AUTO;
    int desc_swap = 0;
    int split_force = 0;           // tests: 0 auto, 1 cluster split-K, 2 L2 slots summed by
                                   // the separate epilogue kernel, 3 L2 slots summed in the
                                   // kernel by the tile's splits after meeting at a counter
    struct TmapEntry {
        const void* ptr;
        int d_in, n_out, ld, box_rows, box_w;
        CUtensorMap map;
    };
    std::vector<TmapEntry> tmaps;
    int plan_tile = 0;             // debug: spiking-linear tile width / split count to use
    int plan_ns = 0;               // (0: the launcher's choice)
    int mode_force = 0;            // debug: 1 gather active rows, 2 stream every row
    int dbg_on = 0;
    int dbg_shape = 0;             // debug: stamp only linears of d_in * 65536 + d_out ...
    int dbg_nth = 0;               // ... and of those only the nth launched since it was set
    int dbg_count = 0;
    unsigned long long* dbg = nullptr;  // 4096 debug timestamps (device)
    // profiling
    int profiling = 0;
    std::vector<cudaEvent_t> ev_pool;
    size_t ev_used = 0;
    std::vector<double> prof_bytes_static;  // per launch: scale/spike bytes known on host
    std::vector<long long> prof_dout;       // per launch: d_out (active rows * d_out bytes)
    std::vector<int> prof_din, prof_bt;     // per launch: d_in, block rows BT
    std::vector<void*> prof_stats_ptr;
    std::vector<cudaStream_t> prof_streams;
};

namespace nmdlm {

// Host-side count of kernel launches issued by the library (all contexts).
void count_launch(unsigned n = 1);

// Workspace carve-out helper: bump allocator over the context workspace.
struct WsCursor {
    char* base;
    size_t cap, off = 0;
    WsCursor(nmdlm_ctx* c) : base((char*)c->ws), cap(c->ws_bytes) {}
    template <class T>
    T* take(size_t n) {
        size_t bytes = (n * sizeof(T) + 255) & ~size_t(255);
        if (off + bytes > cap) return nullptr;
        T* p = (T*)(base + off);
        off += bytes;
        return p;
    }
};

// 2-D TMA descriptor of an int8 W^T block [d_in][n_out] (row stride ld bytes): box of
// 128 channels x box_rows rows, 128-byte swizzle.  Cached per (pointer, shape) in the context.
nmdlm_status weight_tensor_map(nmdlm_ctx* ctx, const int8_t* wT, int d_in, int n_out, int ld,
                               int box_rows, CUtensorMap* out, int box_w = 128);

// Launch a spiking linear (SIMT or tcgen05 by impl/shape).  `ws` provides split-K
// scratch.  Returns a status; sets up per-kernel attributes on first use.
nmdlm_status launch_linear(nmdlm_ctx* ctx, LinArgs& a, nmdlm_impl impl, WsCursor& ws,
                           cudaStream_t stream);

// Pack uint8 spikes; optional compaction.
nmdlm_status launch_pack(nmdlm_ctx* ctx, const uint8_t* spikes, int BT, int D,
                         uint32_t* row_bits, uint32_t* col_masks, uint32_t* active_mask,
                         int32_t* active_idx, int32_t* n_active, cudaStream_t stream);

// Compact an active mask into ascending indices.
nmdlm_status launch_compact(nmdlm_ctx* ctx, const uint32_t* mask, int D, int32_t* idx,
                            int32_t* n_active, cudaStream_t stream);

// IF encode: current source -> spike block.
struct IfArgs {
    int B, T, N;
    int src_kind;              // 0 fp32 dense, 1 int32 dense, 2 embedding gather
    const float* cur_f;        // [B][T][N]
    const int32_t* cur_i;
    const int32_t* tokens;     // embedding: [B]
    const float* tok_emb;      // [V+1][N]
    const float* pos_emb;      // [Lmax][N]
    int pos0, vocab;
    float theta_f;
    int theta_i;
    void* v_state;             // [B][N] or null
    uint32_t* bits;            // [BT][words(N)]
    uint32_t* cm;              // [N][words(BT)] or null
    uint32_t* mask;            // [words(N)] or null
    float* cur_out;            // [BT][N] or null (embedding: the residual stream)
    int* err;
};
nmdlm_status launch_if(nmdlm_ctx* ctx, const IfArgs& a, cudaStream_t stream);

// Attention currents (before the attention IF).
struct AttnArgs {
    const uint32_t* q;   // [B*T][WD]
    const uint32_t* k;   // [T][Ls][WD]
    const uint32_t* v;
    int T, B, L, Ls, H, dh;
    float alpha;
    float* out;          // [B*T][H*dh]
    int* err;
    unsigned long long wait_ns = 1000000000ull;  // bound of every device wait
    unsigned long long* dbg = nullptr;           // debug: phase timestamps of CTA 0, or null
};
nmdlm_status launch_attention(nmdlm_ctx* ctx, const AttnArgs& a, cudaStream_t stream);
// Tensor-core attention (d_head in {32, 64, 96, 128}, B <= 64) else launch_attention.
nmdlm_status launch_attention_best(const AttnArgs& a, cudaStream_t stream);
// Scores and mixture on tcgen05 (kind::f8f6f4, d_head 128); UNSUPPORTED otherwise.
nmdlm_status launch_attention_tc(const AttnArgs& a, cudaStream_t stream);

// Head statistics and unmasking.
nmdlm_status launch_head_unmask(nmdlm_ctx* ctx, const float* logits, int B, int V, int k,
                                int32_t* tokens, int32_t* mask, int32_t* unmasked_out,
                                WsCursor& ws, cudaStream_t stream);

// Bitwise ternary coding (ternary.cu).
nmdlm_status launch_ternary_encode(const float* a, int N, int D, float K, int T, int rs,
                                   uint8_t* plus, uint8_t* minus, int32_t* ahat, float* vth,
                                   cudaStream_t stream);
nmdlm_status launch_ternary_combine(const int32_t* accp, const int32_t* accm, int N, int T,
                                    int rs, int d_out, int32_t* y, cudaStream_t stream);
nmdlm_status launch_ternary_if(const int32_t* y, int N, int d_out, int T, int theta,
                               int8_t* s_out, int32_t* v_out, cudaStream_t stream);

nmdlm_status launch_linear_stats(const uint32_t* cm, const uint32_t* mask, int d_in, int BTW,
                                 int dense, unsigned long long dout,
                                 unsigned long long* stats, cudaStream_t stream);

nmdlm_status launch_wait_test(nmdlm_ctx* ctx, unsigned long long ns, cudaStream_t stream);

// Record a failed CUDA call (its message is returned by nmdlm_last_cuda_error) and
// clear the runtime's sticky last-error state so later launches are not blamed.
void note_cuda_error(cudaError_t e);
// Launch `kernel` as a programmatic dependent of the previous work on `stream`
// (cluster of cluster_y CTAs along y when > 1).
template <class... KArgs, class... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, int cluster_y, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute at[2];
    int n = 0;
    at[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
    if (cluster_y > 1) {
        at[n].id = cudaLaunchAttributeClusterDimension;
        at[n].val.clusterDim.x = 1;
        at[n].val.clusterDim.y = cluster_y;
        at[n].val.clusterDim.z = 1;
        ++n;
    }
    cfg.attrs = at;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// Make sure `func` may use `bytes` of dynamic shared memory on the current device.  The
// attribute belongs to the device, so the size already granted is remembered per
// (kernel, device) under a lock; a larger request raises it.
nmdlm_status ensure_dyn_smem(const void* func, size_t bytes);

// Thread-block clusters of 1..8 CTAs (along y, `threads` threads and `smem` bytes of
// dynamic shared memory each) that fit on the current device at once (occupancy API),
// cached per (kernel, device, smem); out[n] for n = 1..8, out[0] = 0.
nmdlm_status cluster_capacity(const void* func, int threads, size_t smem, int sm_count,
                              int out[9]);

inline nmdlm_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return NMDLM_OK;
    note_cuda_error(e);
    return NMDLM_ERR_CUDA;
}

}  // namespace nmdlm
