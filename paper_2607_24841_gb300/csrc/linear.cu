// linear.cu -- QBSM spiking linear layers with the IF epilogue fused in.
//
// acc[bt][o] = sum over active input channels d of x[bt][d] * W^T[d][o]  (Sec. IV-A):
// a row of W^T is fetched only when its input channel spiked in some row of the
// block (assumption (ii)).  Two kernel families compute the same exact int32 sums:
//   k_linear_simt  CUDA-core accumulation (small blocks, any shape);
//   k_linear_tc    gather-then-MMA on the 5th-generation tensor cores: the active
//                  rows of W^T are gathered into shared memory as the K dimension,
//                  converted int8 -> fp16 (exact), multiplied by the 0/1 spike operand
//                  with tcgen05.mma kind::f16 into fp32 TMEM accumulators.  Products
//                  are exact and every partial sum is an integer below 2^24
//                  (|acc| <= 127 * d_in), so the fp32 result equals the int32 sum.
// Both end in the same IF epilogue (Sec. II-B, Eq. (3)-(4)), so spikes leave the
// kernel packed and never round-trip through memory as integers.
#include <algorithm>
#include <cstdio>

#include "internal.h"

namespace nmdlm {

// ------------------------------------------------------------------ SIMT ----
// grid.x: groups of 32 output channels; block (32, BY).  Thread (lane, ty) owns
// channel lo0 + lane for tokens ty, ty + BY, ...
template <int MAXT, int MAXW>
__global__ void k_linear_simt(LinArgs a) {
    const int g = blockIdx.x;
    const int si = seg_of_tile(a, g);
    const LinSeg& s = a.seg[si];
    const int lane = threadIdx.x, ty = threadIdx.y, BY = blockDim.y;
    const int lo = (g - s.tile_begin) * 32 + lane;
    const bool valid = lo < s.n_out;
    __shared__ uint32_t cm_s[32][MAXW];
    __shared__ int any_s[32];
    for (int i = threadIdx.y * 32 + lane; i < 32 * MAXW; i += 32 * BY) cm_s[i / MAXW][i % MAXW] = 0;
    if (ty == 0) any_s[lane] = 0;
    __syncthreads();

    uint32_t cmw[MAXW];
#pragma unroll
    for (int w = 0; w < MAXW; ++w) cmw[w] = 0;
    bool any = false;
    const int DW = words_of(a.d_in);
    const int T = a.T, BTW = a.BTW;
    for (int b = ty; b < a.B; b += BY) {
        int acc[MAXT];
#pragma unroll
        for (int t = 0; t < MAXT; ++t) acc[t] = 0;
        const int bt0 = b * T, w0 = bt0 >> 5, sh = bt0 & 31;
        for (int w = 0; w < DW; ++w) {
            uint32_t m;
            if (a.dense) {
                const int rem = a.d_in - w * 32;
                m = rem >= 32 ? 0xffffffffu : ((1u << rem) - 1u);
            } else {
                m = a.in_mask[w];
            }
            while (m) {
                const int d = w * 32 + __ffs(m) - 1;
                m &= m - 1;
                const int wv = valid ? (int)s.wT[(size_t)d * s.ld_w + lo] : 0;
                const uint32_t* c = a.in_cm + (size_t)d * BTW;
                uint64_t win = c[w0];
                if (w0 + 1 < BTW) win |= (uint64_t)c[w0 + 1] << 32;
                const uint32_t bits = (uint32_t)(win >> sh);
#pragma unroll
                for (int t = 0; t < MAXT; ++t)
                    if (t < T) acc[t] += ((bits >> t) & 1u) ? wv : 0;
            }
        }
        epi_token<MAXT, MAXW>(a, s, lo, valid, b, [&](int t) { return acc[t]; }, cmw, any);
    }
#pragma unroll
    for (int w = 0; w < MAXW; ++w)
        if (w < BTW && cmw[w]) atomicOr(&cm_s[lane][w], cmw[w]);
    if (any) any_s[lane] = 1;
    __syncthreads();
    if (ty == 0) {
        if (valid && s.cm)
            for (int w = 0; w < BTW; ++w) s.cm[(size_t)lo * BTW + w] = cm_s[lane][w];
        const uint32_t mw = __ballot_sync(0xffffffffu, valid && any_s[lane]);
        if (lane == 0 && s.mask) s.mask[lo >> 5] = mw;
    }
}

// ------------------------------------------------------- block scan (256) ----
// Exclusive prefix sum over the words of the active mask (or all channels when
// dense) into prefix[0..DW]; prefix[DW] is the number of active rows.
__device__ void active_prefix(const LinArgs& a, uint32_t* mask_s, int* prefix, int DW) {
    const int tid = threadIdx.x;
    const int per = (DW + blockDim.x - 1) / blockDim.x;
    const int beg = tid * per, end = min(beg + per, DW);
    int local = 0;
    for (int w = beg; w < end; ++w) {
        uint32_t m;
        if (a.dense) {
            const int rem = a.d_in - w * 32;
            m = rem >= 32 ? 0xffffffffu : ((1u << rem) - 1u);
        } else {
            m = a.in_mask[w];
        }
        mask_s[w] = m;
        local += __popc(m);
    }
    // inclusive scan of `local` across the block
    __shared__ int warp_tot[32];
    const int lane = tid & 31, warp = tid >> 5;
    int x = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        int y = lane < nw ? warp_tot[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int z = __shfl_up_sync(0xffffffffu, y, o);
            if (lane >= o) y += z;
        }
        if (lane < nw) warp_tot[lane] = y;  // inclusive warp totals
    }
    __syncthreads();
    int run = x - local + (warp > 0 ? warp_tot[warp - 1] : 0);  // exclusive prefix
    for (int w = beg; w < end; ++w) {
        prefix[w] = run;
        run += __popc(mask_s[w]);
    }
    if (tid == blockDim.x - 1) prefix[DW] = run;  // last thread holds the total
    __syncthreads();
}

// Row of W^T (input channel) holding compacted position p, or -1 past the end.
__device__ __forceinline__ int active_row(const uint32_t* mask_s, const int* prefix, int DW,
                                          int p) {
    if (p >= prefix[DW]) return -1;
    int lo = 0, hi = DW;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (prefix[mid] <= p) lo = mid; else hi = mid;
    }
    return lo * 32 + (int)__fns(mask_s[lo], 0, p - prefix[lo] + 1);
}

// ---------------------------------------------------------------- tcgen05 ----
namespace tcl {
constexpr int M = 128;       // output channels per tile (TMEM lanes)
constexpr int KC = 64;       // rows of W^T per pipeline stage
constexpr int NSTAGE = 3;
constexpr int NTHREADS = 256;
constexpr int A_BYTES = M * KC * 2;
constexpr int SBO = (KC / 8) * 128;  // bytes between 8-wide MN core-matrix groups
constexpr int LBO = 128;             // bytes between K-adjacent core matrices

template <int NP>
struct Smem {
    static constexpr int B_BYTES = NP * KC * 2;
    static constexpr int STAGE = A_BYTES + B_BYTES;
    static constexpr int STAGES = NSTAGE * STAGE;
    static constexpr int ACC = NP * M * 4;  // accumulator staging (reuses the stages)
    static_assert(ACC <= STAGES, "staging must fit in the stage buffers");
    static constexpr int NCOL = NP <= 32 ? 32 : (NP <= 64 ? 64 : (NP <= 128 ? 128 : 256));
    static size_t bytes(int DW) {
        return STAGES + 8 * (NSTAGE + 1) + 16 + 4 * KC + 4 * (size_t)(2 * DW + 1) + 1024;
    }
};
}  // namespace tcl

template <int NP>
__global__ void __launch_bounds__(tcl::NTHREADS) k_linear_tc(LinArgs a) {
    using namespace tcl;
    using SM = Smem<NP>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = (uint64_t*)(smem + SM::STAGES);
    uint32_t* tmem_holder = (uint32_t*)(bars + NSTAGE + 1);
    int* idx_s = (int*)(tmem_holder + 4);
    const int DW = words_of(a.d_in);
    uint32_t* mask_s = (uint32_t*)(idx_s + KC);
    int* prefix = (int*)(mask_s + DW);
    float* accs = (float*)smem;  // [NP][M] after the main loop

    const int tile = blockIdx.x, split = blockIdx.y;
    const int si = seg_of_tile(a, tile);
    const LinSeg& s = a.seg[si];
    const int lo0 = (tile - s.tile_begin) * M;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int BTW = a.BTW;

    active_prefix(a, mask_s, prefix, DW);
    const int n_active = prefix[DW];
    const int nch = (n_active + KC - 1) / KC;
    const int c0 = (int)((long long)split * nch / a.nsplit);
    const int c1 = (int)((long long)(split + 1) * nch / a.nsplit);

    if (tid == 0) {
        for (int i = 0; i <= NSTAGE; ++i) mbar_init(&bars[i], 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        tmem_alloc(tmem_holder, SM::NCOL);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    const uint32_t idesc = idesc_f16_mn(M, NP);
    const uint32_t lbo = a.desc_swap ? SBO : LBO, sbo = a.desc_swap ? LBO : SBO;

    // W^T segment of this thread: 16 channels starting at lo0 + 16 * warp.
    const int och = lo0 + 16 * warp;
    const bool oval = och + 16 <= s.n_out;
    bool ok = true;
    int issued = 0;
    for (int c = c0; c < c1; ++c) {
        const int j = c - c0, st = j % NSTAGE, use = j / NSTAGE;
        if (tid < KC) {
            const int p = c * KC + tid;
            idx_s[tid] = a.dense ? (p < a.d_in ? p : -1) : active_row(mask_s, prefix, DW, p);
        }
        bool mine = true;
        if (use > 0) mine = mbar_wait_bounded(&bars[st], (use - 1) & 1, a.wait_ns);
        if (__syncthreads_or(!mine)) { ok = false; break; }
        uint8_t* A = smem + st * SM::STAGE;
        uint8_t* Bm = A + A_BYTES;
        // A operand: 64 gathered rows x 128 channels, int8 -> fp16, MN-major.
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int k = lane + 32 * h;
            const int d = idx_s[k];
            uint4 raw = make_uint4(0, 0, 0, 0);
            if (d >= 0 && oval) raw = __ldg(reinterpret_cast<const uint4*>(s.wT + (size_t)d * s.ld_w + och));
            uint4 f0, f1;
            i8x4_to_f16x4(raw.x, f0.x, f0.y);
            i8x4_to_f16x4(raw.y, f0.z, f0.w);
            i8x4_to_f16x4(raw.z, f1.x, f1.y);
            i8x4_to_f16x4(raw.w, f1.z, f1.w);
            uint8_t* dst = A + (2 * warp) * SBO + (k >> 3) * LBO + (k & 7) * 16;
            *reinterpret_cast<uint4*>(dst) = f0;
            *reinterpret_cast<uint4*>(dst + SBO) = f1;
        }
        // B operand: spikes of the gathered rows, 0/1 fp16, MN-major (n = bt).
        for (int e = tid; e < (NP / 8) * KC; e += NTHREADS) {
            const int k = e % KC, ng = e / KC;
            const int d = idx_s[k];
            uint32_t byte = 0;
            if (d >= 0 && (ng >> 2) < BTW) byte = (a.in_cm[(size_t)d * BTW + (ng >> 2)] >> (8 * (ng & 3))) & 0xFFu;
            uint4 v = make_uint4(bits2_to_f16x2(byte), bits2_to_f16x2(byte >> 2),
                                 bits2_to_f16x2(byte >> 4), bits2_to_f16x2(byte >> 6));
            *reinterpret_cast<uint4*>(Bm + ng * SBO + (k >> 3) * LBO + (k & 7) * 16) = v;
        }
        fence_proxy_async_smem();
        __syncthreads();
        if (tid == 0) {
            tc_fence_after();
            const uint32_t a0 = smem_u32(A), b0 = smem_u32(Bm);
#pragma unroll
            for (int kk = 0; kk < KC / 16; ++kk) {
                const uint64_t ad = smem_desc(a0 + kk * 2 * LBO, lbo, sbo);
                const uint64_t bd = smem_desc(b0 + kk * 2 * LBO, lbo, sbo);
                mma_f16(tmem, ad, bd, idesc, (j > 0 || kk > 0) ? 1u : 0u);
            }
            mma_commit(&bars[st]);
        }
        ++issued;
    }
    // Every MMA issued by thread 0 completes before the done barrier fires.
    if (issued > 0) {
        if (tid == 0) mma_commit(&bars[NSTAGE]);
        const bool done = mbar_wait_bounded(&bars[NSTAGE], 0,
                                            ok ? a.wait_ns : 1000000000ull);
        if (__syncthreads_or(!done)) ok = false;
    }
    if (!ok) {
        if (tid == 0) raise_error(a.err, ERRBIT_TIMEOUT);
        tc_fence_before();
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, SM::NCOL);
        return;
    }
    tc_fence_after();
    // TMEM -> shared staging accs[bt][m] (warps 0-3 own TMEM lanes 32w..32w+31).
    if (warp < 4) {
        const int m = warp * 32 + lane;
        for (int cb = 0; cb < NP / 8; ++cb) {
            uint32_t v[8];
            if (issued > 0) {
                tmem_ld8(tmem + ((uint32_t)(warp * 32) << 16) + cb * 8, v);
            } else {
#pragma unroll
                for (int i = 0; i < 8; ++i) v[i] = 0;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) accs[(cb * 8 + i) * M + m] = __uint_as_float(v[i]);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, SM::NCOL);

    // Split-K: publish the partial tile; the last CTA of the tile sums and finishes.
    if (a.nsplit > 1) {
        float* part = a.ws + ((size_t)split * a.n_tiles + tile) * NP * M;
        for (int i = tid; i < NP * M; i += NTHREADS) part[i] = accs[i];
        __threadfence();
        __syncthreads();
        __shared__ int s_last;
        if (tid == 0) {
            const unsigned prev = atomicAdd(&a.counters[tile], 1u);
            s_last = (prev == (unsigned)(a.nsplit - 1));
            if (s_last) a.counters[tile] = 0;  // ready for the next launch
        }
        __syncthreads();
        if (!s_last) return;
        __threadfence();
        for (int i = tid; i < NP * M; i += NTHREADS) {
            float sum = 0.0f;
            for (int q = 0; q < a.nsplit; ++q)
                sum += __ldcg(a.ws + ((size_t)q * a.n_tiles + tile) * NP * M + i);
            accs[i] = sum;
        }
        __syncthreads();
    }
    // Epilogue: warps 0-3, one output channel per lane, all tokens.
    if (warp < 4) {
        const int m = warp * 32 + lane;
        const int lo = lo0 + m;
        const bool valid = lo < s.n_out;
        uint32_t cmw[8];
#pragma unroll
        for (int w = 0; w < 8; ++w) cmw[w] = 0;
        bool any = false;
        for (int b = 0; b < a.B; ++b) {
            epi_token<32, 8>(a, s, lo, valid, b,
                             [&](int t) { return (int)accs[(b * a.T + t) * M + m]; }, cmw, any);
        }
        if (a.kind != EPI_KIND_LOGITS) {
            if (valid && s.cm)
                for (int w = 0; w < BTW; ++w) s.cm[(size_t)lo * BTW + w] = cmw[w];
            const uint32_t mw = __ballot_sync(0xffffffffu, valid && any);
            if (lane == 0 && s.mask && lo < s.n_out) s.mask[lo >> 5] = mw;
        }
    }
}

// ------------------------------------------------------------------ stats ----
__global__ void k_linear_stats(const uint32_t* cm, const uint32_t* mask, int d_in, int BTW,
                               int dense, unsigned long long dout, unsigned long long* stats) {
    unsigned long long rows = 0, nnz = 0;
    for (int d = blockIdx.x * blockDim.x + threadIdx.x; d < d_in; d += gridDim.x * blockDim.x) {
        const bool act = (mask[d >> 5] >> (d & 31)) & 1u;
        rows += (dense || act) ? 1 : 0;
        if (act)
            for (int w = 0; w < BTW; ++w) nnz += __popc(cm[(size_t)d * BTW + w]);
    }
    for (int o = 16; o > 0; o >>= 1) {
        rows += __shfl_down_sync(0xffffffffu, rows, o);
        nnz += __shfl_down_sync(0xffffffffu, nnz, o);
    }
    if ((threadIdx.x & 31) == 0) {
        if (rows) atomicAdd(&stats[0], rows);
        if (nnz) atomicAdd(&stats[1], nnz * dout);
    }
}

nmdlm_status launch_linear_stats(const uint32_t* cm, const uint32_t* mask, int d_in, int BTW,
                                 int dense, unsigned long long dout,
                                 unsigned long long* stats, cudaStream_t stream) {
    const int threads = 256;
    const int blocks = std::min(64, (d_in + threads - 1) / threads);
    k_linear_stats<<<blocks, threads, 0, stream>>>(cm, mask, d_in, BTW, dense, dout, stats);
    count_launch();
    return cuda_status(cudaGetLastError());
}

// ------------------------------------------------------------------ launch ----
template <int MAXT, int MAXW>
static nmdlm_status launch_simt_t(LinArgs& a, cudaStream_t stream) {
    int groups = 0;
    for (int i = 0; i < a.nseg; ++i) {
        a.seg[i].tile_begin = groups;
        groups += words_of(a.seg[i].n_out);
    }
    a.n_tiles = groups;
    int g = 1;
    while (g < 32 && (g * a.T) % 32 != 0) g <<= 1;  // tokens per 32-bit column word
    const int BY = std::max(1, std::min(a.B, std::max(g, 8)));
    dim3 block(32, BY);
    k_linear_simt<MAXT, MAXW><<<groups, block, 0, stream>>>(a);
    count_launch();
    return cuda_status(cudaGetLastError());
}

static nmdlm_status launch_simt(LinArgs& a, cudaStream_t stream) {
    if (a.T <= 4 && a.BTW <= 8) return launch_simt_t<4, 8>(a, stream);
    if (a.T <= 8 && a.BTW <= 8) return launch_simt_t<8, 8>(a, stream);
    return launch_simt_t<32, 8>(a, stream);
}

template <int NP>
static nmdlm_status launch_tc_t(nmdlm_ctx* ctx, LinArgs& a, WsCursor& ws,
                                cudaStream_t stream) {
    using SM = tcl::Smem<NP>;
    const size_t smem = SM::bytes(words_of(a.d_in));
    if (smem > 200 * 1024) return NMDLM_ERR_UNSUPPORTED;
    static size_t configured = 0;
    if (smem > configured) {
        if (cuda_status(cudaFuncSetAttribute(k_linear_tc<NP>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem)) != NMDLM_OK)
            return NMDLM_ERR_CUDA;
        configured = smem;
    }
    int tiles = 0;
    for (int i = 0; i < a.nseg; ++i) {
        a.seg[i].tile_begin = tiles;
        tiles += (a.seg[i].n_out + tcl::M - 1) / tcl::M;
    }
    a.n_tiles = tiles;
    const int max_chunks = std::max(1, (a.d_in + tcl::KC - 1) / tcl::KC);
    const int per_sm = smem <= 110 * 1024 ? 2 : 1;
    const int target = ctx->sm_count * per_sm;
    int nsplit = std::max(1, std::min((target + tiles - 1) / tiles, max_chunks));
    nsplit = std::min(nsplit, 32);
    if (nsplit > 1) {
        if ((size_t)tiles > ctx->n_counters) return NMDLM_ERR_WORKSPACE;
        a.ws = ws.take<float>((size_t)nsplit * tiles * NP * tcl::M);
        if (!a.ws) return NMDLM_ERR_WORKSPACE;
    }
    a.counters = ctx->counters;
    a.nsplit = nsplit;
    dim3 grid(tiles, nsplit);
    k_linear_tc<NP><<<grid, tcl::NTHREADS, smem, stream>>>(a);
    count_launch();
    return cuda_status(cudaGetLastError());
}

nmdlm_status launch_linear(nmdlm_ctx* ctx, LinArgs& a, nmdlm_impl impl, WsCursor& ws,
                           cudaStream_t stream) {
    a.err = ctx->err;
    a.wait_ns = ctx->wait_ns;
    a.desc_swap = ctx->desc_swap;
    bool tc_ok = a.BT <= 256 && a.T <= 32 && words_of(a.d_in) <= 4096;
    for (int i = 0; i < a.nseg; ++i) {
        const LinSeg& s = a.seg[i];
        if (s.n_out % 16 || s.ld_w % 16 || ((uintptr_t)s.wT & 15)) tc_ok = false;
        if (i + 1 < a.nseg && s.n_out % 128) tc_ok = false;
    }
    if (impl == NMDLM_IMPL_TC && !tc_ok) return NMDLM_ERR_UNSUPPORTED;
    bool use_tc = impl == NMDLM_IMPL_TC || (impl == NMDLM_IMPL_AUTO && tc_ok && a.BT > 8);
    if (!use_tc) {
        for (int i = 0; i + 1 < a.nseg; ++i)
            if (a.seg[i].n_out % 32) return NMDLM_ERR_UNSUPPORTED;
        return launch_simt(a, stream);
    }
    if (a.BT <= 16) return launch_tc_t<16>(ctx, a, ws, stream);
    if (a.BT <= 32) return launch_tc_t<32>(ctx, a, ws, stream);
    if (a.BT <= 64) return launch_tc_t<64>(ctx, a, ws, stream);
    if (a.BT <= 128) return launch_tc_t<128>(ctx, a, ws, stream);
    return launch_tc_t<256>(ctx, a, ws, stream);
}

}  // namespace nmdlm
