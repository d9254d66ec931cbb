// probe.cu -- tensor-core and tensor-memory rate probes (measurement only).
//
// The kernel design choices of the spiking linear and the spike attention rest on a
// few per-SM rates of the 5th-generation tensor cores: how long one tcgen05.mma of a
// given kind and shape occupies the pipe when issued back to back, with the A operand
// in shared memory or in tensor memory, and how fast warps move data into tensor
// memory.  These probes time them on one CTA with clock64.  Operands are zero (the
// values do not change the rate); every wait is bounded.
#include <type_traits>
#include <vector>

#include "internal.h"

namespace nmdlm {
namespace {

constexpr int kProbeThreads = 128;
constexpr uint32_t kProbeBuf = 65536;  // bytes of each shared-memory operand buffer

// Instruction descriptors (dense, no negation): D format at bits 4-5, A / B formats at
// 7-9 / 10-12, A / B major-ness at 15 / 16, N / 8 at 17-22, M / 16 at 24-28.
__device__ __forceinline__ uint32_t probe_idesc(int kind, int M, int N) {
    uint32_t d = ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
    if (kind == 0) d |= 1u << 4;  // f16 x f16 -> f32, both K-major
    if (kind == 1) d |= 1u << 4;  // e4m3 x e4m3 -> f32 (format code 0), both K-major
    if (kind == 2) d |= (1u << 4) | (1u << 15) | (1u << 16);  // e4m3, both MN-major
    if (kind == 3) d |= (1u << 4) | (1u << 16);               // e4m3, B MN-major
    return d;
}

__device__ __forceinline__ void mma_f8_ss(uint32_t td, uint64_t a, uint64_t b, uint32_t id,
                                          uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(td),
        "l"(a), "l"(b), "r"(id), "r"(acc)
        : "memory");
}

// kind 0: f16 (A in shared memory, or in tensor memory when a_tmem), kind 1: e4m3,
// kind 2: e4m3 with A and B MN-major, kind 3: e4m3 with B MN-major.
// MMA i accumulates into D region i % n_acc (N columns each from column 0), so n_acc > 1
// issues independent accumulation chains back to back.  out[0] = cycles from the first
// issue to the completion of the last MMA, out[1] = 1 when the completion was observed
// within wait_ns.
__global__ void __launch_bounds__(kProbeThreads, 1)
    k_probe_mma(int kind, int a_tmem, int M, int N, int n_acc, int n_mma, int per_commit,
                int handoff, unsigned long long wait_ns, unsigned long long* out) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    __shared__ uint64_t bar, pbar;
    __shared__ uint32_t tmem_holder;
    for (uint32_t i = threadIdx.x; i < 2 * kProbeBuf / 16; i += kProbeThreads)
        reinterpret_cast<uint4*>(smem)[i] = make_uint4(0, 0, 0, 0);
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_init(&pbar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    fence_proxy_async_smem();
    if (threadIdx.x < 32) {
        tmem_alloc(&tmem_holder, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_holder;
    if (a_tmem) {  // zero the A columns [448, 464) of every lane
        uint32_t z[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) z[i] = 0u;
        const int q = threadIdx.x >> 5;
        tmem_st16(tmem + ((uint32_t)(q * 32) << 16) + 448u, z);
        tmem_wait_st();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (threadIdx.x == 0) {
        const uint32_t id = probe_idesc(kind, M, N);
        // K-major, no swizzle: K-adjacent core matrices 128 B apart, 8-row groups 256 B
        // apart; an M = 128 operand spans 4 KB, an N = 256 one 8 KB, inside the buffers.
        const uint64_t ad = smem_desc(smem_u32(smem), 128, 256);
        const uint64_t bd = smem_desc(smem_u32(smem + kProbeBuf), 128, 256);
        const long long t0 = clock64();
        auto issue = [&](int i, int r) {
            const uint32_t acc = i >= n_acc ? 1u : 0u;
            const uint32_t td = tmem + (uint32_t)(r * N);
            if (kind >= 1) mma_f8_ss(td, ad, bd, id, acc);
            else if (a_tmem) mma_f16_ts(td, tmem + 448u, bd, id, acc);
            else mma_f16(td, ad, bd, id, acc);
        };
        // the hand-off a pipelined kernel makes per group of G MMAs (bit 0 of handoff: a
        // commit to a barrier, bit 1: a tcgen05 fence, bit 2: a non-blocking query of
        // another barrier), with the group unrolled so that nothing else runs between
        auto groups = [&](auto G) {
            for (int i = 0; i < n_mma; i += G.value) {
#pragma unroll
                for (int g = 0; g < G.value; ++g) issue(i + g, (i + g) % n_acc);
                if (handoff & 1) mma_commit(&pbar);
                if (handoff & 2) tc_fence_after();
                if (handoff & 4) (void)mbar_test_wait(&bar, 1);
            }
        };
        if (per_commit == 0) {
            int r = 0;
            for (int i = 0; i < n_mma; ++i) {
                issue(i, r);
                if (++r == n_acc) r = 0;
            }
        } else if (per_commit == 1) {
            groups(std::integral_constant<int, 1>());
        } else if (per_commit == 2) {
            groups(std::integral_constant<int, 2>());
        } else if (per_commit == 4) {
            groups(std::integral_constant<int, 4>());
        } else {
            groups(std::integral_constant<int, 8>());
        }
        mma_commit(&bar);
        bool ok = mbar_wait_bounded(&bar, 0, wait_ns);
        const long long t1 = clock64();
        if (!ok) mbar_wait_bounded(&bar, 0, wait_ns);  // let the MMAs drain before freeing
        out[0] = (unsigned long long)(t1 - t0);
        out[1] = ok ? 1ull : 0ull;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (threadIdx.x < 32) tmem_dealloc(tmem, 512);
}

// Tensor-memory store rate: each of the four warps writes its lane quarter, 16 columns
// per tcgen05.st, n_st times over 256 columns, then waits for the stores.
__global__ void __launch_bounds__(kProbeThreads, 1)
    k_probe_tmem_st(int n_st, unsigned long long* out) {
    __shared__ uint32_t tmem_holder;
    if (threadIdx.x < 32) {
        tmem_alloc(&tmem_holder, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_holder;
    const int q = threadIdx.x >> 5;
    uint32_t v[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = threadIdx.x * 16u + i;
    __syncthreads();
    const long long t0 = clock64();
    for (int i = 0; i < n_st; ++i)
        tmem_st16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)((i & 15) * 16), v);
    tmem_wait_st();
    const long long t1 = clock64();
    if (threadIdx.x == 0) {
        out[0] = (unsigned long long)(t1 - t0);
        out[1] = 1ull;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (threadIdx.x < 32) tmem_dealloc(tmem, 512);
}

// Weight streaming alone (no conversion, no MMA): CTA c reads tile c % tiles of a d_in x
// (tiles x 256) int8 matrix, rows [split x d_in / nsplit, ...), in the spiking linear's
// chunks (64 rows x 256 channels) through `stages` stages.  mode 0: the matrix row-major,
// a chunk as two 2-D TMA boxes of 128 channels with the 128-byte swizzle (64 pieces of
// 256 bytes, d_out bytes apart); 1: each tile's columns stored contiguously ([tile][row]
// [256]), the same boxes; 2: the contiguous layout, a chunk as one 16 KB 1-D bulk copy;
// 3 (k_probe_stream_ldg): the contiguous layout read with plain 16-byte loads.
constexpr int kStreamMaxStages = 8;
__global__ void __launch_bounds__(64, 1)
    k_probe_stream(const __grid_constant__ CUtensorMap map, const int8_t* w, int tiles, int d_in,
                   int nsplit, int mode, int stages, unsigned long long wait_ns,
                   unsigned long long* out) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    __shared__ uint64_t full[kStreamMaxStages], empty[kStreamMaxStages];
    if (threadIdx.x == 0) {
        for (int i = 0; i < stages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    const int tile = blockIdx.x % tiles, split = blockIdx.x / tiles;
    const int nch = d_in / 64 / nsplit, r0 = split * nch * 64;
    bool ok = true;
    if (threadIdx.x == 0) {
        for (int j = 0; j < nch && ok; ++j) {
            const int st = j % stages, u = j / stages;
            if (u > 0) ok = mbar_wait_bounded(&empty[st], (u - 1) & 1, wait_ns);
            if (!ok) break;
            mbar_arrive_expect_tx(&full[st], 16384u);
            const int row = r0 + j * 64;
            if (mode == 2) {
                bulk_load(smem + st * 16384, w + ((size_t)tile * d_in + row) * 256, 16384u, &full[st]);
            } else {
                for (int b = 0; b < 2; ++b)
                    tma_load_2d(smem + st * 16384 + b * 8192, &map, mode ? b * 128 : tile * 256 + b * 128,
                                mode ? tile * d_in + row : row, &full[st]);
            }
        }
    } else if (threadIdx.x == 32) {
        for (int j = 0; j < nch && ok; ++j) {
            const int st = j % stages, u = j / stages;
            ok = mbar_wait_bounded(&full[st], u & 1, wait_ns);
            if (ok) mbar_arrive(&empty[st]);
        }
    }
    if (!ok) out[1] = 1ull;  // a wait ran out (the host reports a timeout)
    __syncthreads();
}

// The same reads with plain 16-byte loads from 256 threads (no TMA, no shared memory):
// CTA c reads its tile's rows of the tile-contiguous layout, each thread four 16-byte
// pieces of a chunk, `depth` chunks in flight; the bytes are summed into out[2].
__global__ void __launch_bounds__(256)
    k_probe_stream_ldg(const int8_t* w, int tiles, int d_in, int nsplit, unsigned long long* out) {
    const int tile = blockIdx.x % tiles, split = blockIdx.x / tiles;
    const int nch = d_in / 64 / nsplit, r0 = split * nch * 64;
    const uint4* base = reinterpret_cast<const uint4*>(w + ((size_t)tile * d_in + r0) * 256);
    uint32_t acc = 0;
    constexpr int DEPTH = 4;  // chunks in flight per thread
    for (int j0 = 0; j0 < nch; j0 += DEPTH) {
        uint4 v[DEPTH][4];
#pragma unroll
        for (int d = 0; d < DEPTH; ++d)
#pragma unroll
            for (int i = 0; i < 4; ++i)
                v[d][i] = j0 + d < nch ? __ldcs(base + (size_t)(j0 + d) * 1024 + i * 256 + threadIdx.x)
                                       : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int d = 0; d < DEPTH; ++d)
#pragma unroll
            for (int i = 0; i < 4; ++i) acc ^= v[d][i].x ^ v[d][i].y ^ v[d][i].z ^ v[d][i].w;
    }
    if (acc == 0x9e3779b9u) out[2] = acc;  // keeps the loads
}

}  // namespace
}  // namespace nmdlm

// Not part of the public header (measurement): cycles per operation of one CTA.
//   op 0: tcgen05.mma kind::f16, A in shared memory;  op 1: the same with A in tensor
//   memory;  op 2: kind::f8f6f4 (e4m3), A in shared memory;  op 3: tcgen05.st of
//   32 lanes x 16 columns per warp (4 warps);  op 4: e4m3 with A and B MN-major;  op 5:
//   e4m3 with B MN-major.  M in {64, 128}, N a multiple of 16 up
//   to 256 (the MMA shapes of cta_group::1); n_acc independent accumulators
//   (n_acc * N <= 448 columns) taken in turn; per_commit = n | (h << 16), n in
//   {1, 2, 4, 8}, adds after every n MMAs the hand-off steps selected by the bits of h
//   (1: commit to a barrier, 2: tcgen05 fence, 4: non-blocking query of a barrier).
extern "C" nmdlm_status nmdlm_debug_probe_rate(nmdlm_ctx* ctx, int op, int M, int N,
                                               int n_acc, int per_commit, int count,
                                               double* cycles_per_op) {
    using namespace nmdlm;
    if (!ctx || !cycles_per_op || op < 0 || op > 5 || count < 1 || count > (1 << 16))
        return NMDLM_ERR_INVALID_ARG;
    const bool mma = op != 3;
    if (mma && (!(M == 64 || M == 128) || N < 16 || N > 256 || N % 16 || n_acc < 1 ||
                   n_acc * N > 448))
        return NMDLM_ERR_UNSUPPORTED;
    int prev = -1;
    cudaGetDevice(&prev);
    if (prev != ctx->device) cudaSetDevice(ctx->device);
    unsigned long long* d_out = ctx->dbg;  // the context's debug words
    cudaError_t e = cudaMemset(d_out, 0, 2 * sizeof(unsigned long long));
    if (e != cudaSuccess) {
    } else if (mma) {
        const size_t smem = 2 * kProbeBuf + 1024;
        e = cudaFuncSetAttribute(k_probe_mma, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e == cudaSuccess) {
            const int kind = op == 2 ? 1 : op == 4 ? 2 : op == 5 ? 3 : 0;
            k_probe_mma<<<1, kProbeThreads, smem>>>(kind, op == 1 ? 1 : 0, M, N,
                                                    n_acc, count, per_commit & 0xffff,
                                                    per_commit >> 16, 1000000000ull, d_out);
            e = cudaGetLastError();
        }
    } else {
        k_probe_tmem_st<<<1, kProbeThreads>>>(count, d_out);
        e = cudaGetLastError();
    }
    unsigned long long h[2] = {0, 0};
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e == cudaSuccess) e = cudaMemcpy(h, d_out, sizeof(h), cudaMemcpyDeviceToHost);
    if (prev >= 0 && prev != ctx->device) cudaSetDevice(prev);
    if (e != cudaSuccess) return cuda_status(e);
    if (!h[1]) return NMDLM_ERR_TIMEOUT;
    *cycles_per_op = (double)h[0] / (double)count;
    return NMDLM_OK;
}

// Not part of the public header (measurement): microseconds per launch of k_probe_stream
// over a d_in x (tiles x 256) int8 matrix, `copies` copies rotated (more than L2), `reps`
// launches each; mode_stages = mode | (stages << 8) (stages 0: 4).
extern "C" nmdlm_status nmdlm_debug_probe_stream(nmdlm_ctx* ctx, int mode_stages, int tiles,
                                                 int d_in, int nsplit, int copies, int reps,
                                                 double* us_per_launch) {
    using namespace nmdlm;
    const int mode = mode_stages & 0xff, stages = mode_stages >> 8 ? mode_stages >> 8 : 4;
    const int tiled = mode != 0;
    if (!ctx || !us_per_launch || tiles < 1 || tiles > 256 || nsplit < 1 || d_in < 64 ||
        d_in % (64 * nsplit) || mode > 3 || stages < 2 || stages > kStreamMaxStages || copies < 1 ||
        copies > 16 || reps < 1 || reps > 1000)
        return NMDLM_ERR_INVALID_ARG;
    int prev = -1;
    cudaGetDevice(&prev);
    if (prev != ctx->device) cudaSetDevice(ctx->device);
    const size_t bytes = (size_t)tiles * 256 * d_in;
    std::vector<int8_t*> w(copies, nullptr);
    nmdlm_status st = NMDLM_OK;
    for (int c = 0; c < copies && st == NMDLM_OK; ++c)
        if (cudaMalloc(&w[c], bytes) != cudaSuccess || cudaMemset(w[c], c, bytes) != cudaSuccess)
            st = NMDLM_ERR_CUDA;
    std::vector<CUtensorMap> maps(copies);
    for (int c = 0; c < copies && st == NMDLM_OK; ++c)
        st = tiled ? weight_tensor_map(ctx, w[c], tiles * d_in, 256, 256, 64, &maps[c], 128)
                   : weight_tensor_map(ctx, w[c], d_in, tiles * 256, tiles * 256, 64, &maps[c], 128);
    unsigned long long* d_out = ctx->dbg;
    const size_t smem = (size_t)stages * 16384 + 1024;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    if (st == NMDLM_OK && (cudaMemset(d_out, 0, 2 * sizeof(unsigned long long)) != cudaSuccess ||
                           cudaFuncSetAttribute(k_probe_stream, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                (int)smem) != cudaSuccess ||
                           cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess))
        st = NMDLM_ERR_CUDA;
    if (st == NMDLM_OK) {
        auto launch = [&](int c) {
            if (mode == 3)
                k_probe_stream_ldg<<<tiles * nsplit, 256>>>(w[c], tiles, d_in, nsplit, d_out);
            else
                k_probe_stream<<<tiles * nsplit, 64, smem>>>(maps[c], w[c], tiles, d_in, nsplit, mode,
                                                             stages, 1000000000ull, d_out);
        };
        for (int c = 0; c < copies; ++c) launch(c);  // warm-up
        cudaEventRecord(e0);
        for (int r = 0; r < reps; ++r) launch(r % copies);
        cudaEventRecord(e1);
        if (cudaEventSynchronize(e1) != cudaSuccess) st = NMDLM_ERR_CUDA;
        float ms = 0.0f;
        cudaEventElapsedTime(&ms, e0, e1);
        unsigned long long h[2] = {0, 0};
        if (st == NMDLM_OK && cudaMemcpy(h, d_out, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess)
            st = NMDLM_ERR_CUDA;
        if (st == NMDLM_OK && h[1]) st = NMDLM_ERR_TIMEOUT;
        *us_per_launch = 1000.0 * ms / reps;
    }
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    for (int c = 0; c < copies; ++c)
        if (w[c]) cudaFree(w[c]);
    ctx->tmaps.clear();  // the maps named freed memory
    if (prev >= 0 && prev != ctx->device) cudaSetDevice(prev);
    return st;
}
