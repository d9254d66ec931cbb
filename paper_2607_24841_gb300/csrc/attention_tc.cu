// attention_tc.cu -- spike attention with the mixture on the 5th-generation tensor cores.
//
// One CTA per (head h, timestep t, tile of up to 32 queries), d_head = 128 (the reading
// of the paper's binary-binary attention, Fig. 1, is the one of attention.cu):
//   score[n][j] = popcount(q_n AND k_j)                            (CUDA cores)
//   p[n][j]     = exp(alpha * (score[n][j] - c_n)) / Z_n,  Z_n = sum_j exp(...)
//   out[n][d]   = sum_j p[n][j] * v_j[d]                           (tcgen05.mma)
// Softmax is invariant to the shift c_n; this kernel takes c_n = popcount(q_n), the
// largest score query n can reach, so every exponent is <= 0 and no running maximum or
// rescaling is needed: keys are visited once, in tiles of 128, and the partial sums of
// every tile add into one accumulator.  The exponentials of the d_head + 1 possible
// values of score - c_n come from a table (computed in fp64, rounded to fp32, scaled by
// 2^15 so that the smallest, e^{-alpha d_head} 2^15 >= 0.4, stays a normal fp16 number);
// each weight is split into two fp16 halves, hi + lo, so the mixture keeps ~2^-22
// relative precision.
//
// The mixture O^T = V^T P^T per tile: M = 128 (the head's channels), N = 64 (P hi of
// the 32 queries, then P lo), K = 128 keys in 8 steps of 16, fp32 accumulation in tensor
// memory.  Both operands are MN-major fp16 core matrices in shared memory: A = V^T
// written by 4 warps with one key per thread (a key's V word already runs along the
// channels, so no transpose is needed; spikes as fp16 2^-16, removed at the end), and
// B = P^T written by 16 scoring warps, one key and 8 queries per thread.  Scores cost
// three popcounts per key and query (a carry-save sum of the four AND words).  One
// warp issues the MMAs; two stages of A and B.  Every wait is bounded.
#include <algorithm>

#include "internal.h"

namespace nmdlm {
// Debug timestamp of CTA (0, 0, 0), thread `th` (when a.dbg is set).
#define NMDLM_ASTAMP(a, th, slot)                                                    \
    do {                                                                             \
        if ((a).dbg && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0 &&       \
            threadIdx.x == (th) && (slot) < 4096)                                    \
            (a).dbg[(slot)] = clock64();                                             \
    } while (0)
namespace attn3 {
constexpr int DH = 128;                       // head width: the mixture's M
constexpr int NQ = 32;                        // queries per CTA
constexpr int KT = 128;                       // keys per tile
constexpr int NVW = 4;                        // V^T warps: one key per thread
constexpr int NSCORE = 16;                    // scoring warps: 128 keys x 4 query quarters
constexpr int QQ = 8;                         // queries per scoring thread
constexpr int WARP_MMA = NVW + NSCORE;        // 20
constexpr int NTHREADS = (WARP_MMA + 1) * 32; // 672
constexpr int LOADERS = (NVW + NSCORE) * 32;
constexpr int NP = 2 * NQ;                    // MMA N: P hi then P lo
constexpr int LBO = 128;                      // bytes between K-adjacent core matrices
constexpr int SBO = (KT / 8) * 128;           // bytes between 8-row groups (channels / queries)
constexpr int A_BYTES = DH * KT * 2;          // 32 KB per stage
constexpr int P_BYTES = NP * KT * 2;          // 16 KB per stage
constexpr int NCOL = 64;                      // D: NP columns of tensor memory
constexpr int PSCALE_LOG2 = 15;
// shared memory: NST stages of A and P, K and V words of every key, Q, table, sums,
// per-query normalisers, barriers (3 per stage + 1)
template <int NST>
struct Lay {
    static constexpr int OFF_A = 0;
    static constexpr int OFF_P = NST * A_BYTES;
    static constexpr int OFF_KV = OFF_P + NST * P_BYTES;
    static __host__ __device__ constexpr size_t off_q(int L) { return OFF_KV + (size_t)32 * L; }
    static __host__ __device__ constexpr size_t off_lut(int L) { return off_q(L) + NQ * 16; }
    static __host__ __device__ constexpr size_t off_z(int L) { return off_lut(L) + (DH + 1) * 8; }
    static __host__ __device__ constexpr size_t off_zq(int L) { return off_z(L) + NSCORE * QQ * 4; }
    static __host__ __device__ constexpr size_t off_bar(int L) { return off_zq(L) + NQ * 4; }
    static __host__ __device__ constexpr size_t smem_bytes(int L) {
        return off_bar(L) + 8 * (3 * NST + 1) + 16 + 1024;
    }
};
static_assert(NP <= NCOL, "tensor memory budget");
}  // namespace attn3

// popcount(w0) + popcount(w1) + popcount(w2) + popcount(w3) with three popcounts: a
// carry-save sum of the four words per bit position (a full adder, then a half adder).
__device__ __forceinline__ int popc4(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3) {
    const uint32_t s1 = w0 ^ w1 ^ w2, c1 = (w0 & w1) | (w2 & (w0 ^ w1));
    const uint32_t s2 = s1 ^ w3, c2 = s1 & w3;
    return __popc(s2) + 2 * (__popc(c1) + __popc(c2));
}

template <int NST>
__global__ void __launch_bounds__(attn3::NTHREADS, 1) k_attention_tc(const __grid_constant__ AttnArgs a) {
    using namespace attn3;
    using Y = Lay<NST>;
    constexpr int OFF_A = Y::OFF_A, OFF_P = Y::OFF_P, OFF_KV = Y::OFF_KV;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const int L = a.L;
    uint4* kv_s = (uint4*)(smem + OFF_KV);                 // [L] K words, then [L] V words
    uint4* q_s = (uint4*)(smem + Y::off_q(L));             // [NQ]
    uint2* lut = (uint2*)(smem + Y::off_lut(L));           // [DH + 1] {hi|lo fp16, p fp32}
    float* z_s = (float*)(smem + Y::off_z(L));             // [NSCORE][QQ] per-warp sums
    float* zq_s = (float*)(smem + Y::off_zq(L));           // [NQ] normaliser per query
    uint64_t* bar = (uint64_t*)(smem + Y::off_bar(L));
    uint64_t* a_full = bar;           // [NST] V^T written (NVW arrivals)
    uint64_t* p_full = bar + NST;     // [NST] P written (NSCORE arrivals)
    uint64_t* st_free = bar + 2 * NST;  // [NST] the MMAs reading the stage completed
    uint64_t* done = bar + 3 * NST;   // every MMA completed
    uint32_t* tmem_holder = (uint32_t*)(bar + 3 * NST + 1);
    volatile int* abort_flag = (volatile int*)(bar + 3 * NST + 1) + 1;

    const int h = blockIdx.x, t = blockIdx.y, q0 = blockIdx.z * NQ;
    const int nq = min(NQ, a.B - q0);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int WD = words_of(a.H * DH);
    const int ntile = (L + KT - 1) / KT;

    // ---- setup that reads nothing another kernel writes
    for (int x = tid; x <= DH; x += NTHREADS) {
        // weight of score - c = -x, scaled by 2^15, split into fp16 hi + lo
        const float p = (float)(exp(-(double)a.alpha * (double)x) * (double)(1 << PSCALE_LOG2));
        const __half hi = __float2half_rn(p);
        const __half lo = __float2half_rn(p - __half2float(hi));
        lut[DH - x] = make_uint2((uint32_t)__half_as_ushort(hi) | ((uint32_t)__half_as_ushort(lo) << 16),
                                 __float_as_uint(p));
    }
    if (tid == 0) {
        *abort_flag = 0;
        for (int s = 0; s < NST; ++s) {
            mbar_init(&a_full[s], NVW);
            mbar_init(&p_full[s], NSCORE);
            mbar_init(&st_free[s], 1);
        }
        mbar_init(done, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == WARP_MMA) {
        tmem_alloc(tmem_holder, NCOL);
        tmem_relinquish();
    }
    pdl_wait();
    NMDLM_ASTAMP(a, 0, 40);
    // ---- queries of this tile and every key's K and V words of this head and timestep
    if (tid < NQ) {
        uint4 qv = make_uint4(0u, 0u, 0u, 0u);
        if (tid < nq) qv = *reinterpret_cast<const uint4*>(a.q + (size_t)((q0 + tid) * a.T + t) * WD + h * 4);
        q_s[tid] = qv;
    }
    if (warp < WARP_MMA) {
        const uint32_t* kb = a.k + (size_t)t * a.Ls * WD + h * 4;
        const uint32_t* vb = a.v + (size_t)t * a.Ls * WD + h * 4;
        for (int j = tid; j < L; j += LOADERS) {
            cp_async16(kv_s + j, kb + (size_t)j * WD, 16u);
            cp_async16(kv_s + L + j, vb + (size_t)j * WD, 16u);
        }
        cp_async_commit();
        cp_async_wait<0>();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    NMDLM_ASTAMP(a, 0, 41);

    if (warp < NVW) {
        // ---------------------------------------- V^T: key k's channels as fp16 2^-16 / 0
        const int k = tid;  // key row of the tile
        for (int kt = 0; kt < ntile; ++kt) {
            const int s = kt % NST, u = kt / NST;
            const int key = kt * KT + k;
            const uint4 v = key < L ? kv_s[L + key] : make_uint4(0u, 0u, 0u, 0u);
            uint32_t e[4][16];
            bits_to_e16_pairs(v.x, e[0]);
            bits_to_e16_pairs(v.y, e[1]);
            bits_to_e16_pairs(v.z, e[2]);
            bits_to_e16_pairs(v.w, e[3]);
            if (u > 0) {
                const bool ok = mbar_wait_bounded(&st_free[s], (u - 1) & 1, a.wait_ns);
                if (!__all_sync(0xffffffffu, ok) || *abort_flag) {
                    if (lane == 0) { *abort_flag = 1; raise_error(a.err, ERRBIT_TIMEOUT); }
                    break;
                }
            }
            // channel group g (8 channels, 16 bytes) of key k: A + g*SBO + (k/8)*LBO + (k%8)*16
            uint8_t* A = smem + OFF_A + s * A_BYTES + (k >> 3) * LBO + (k & 7) * 16;
#pragma unroll
            for (int w = 0; w < 4; ++w)
#pragma unroll
                for (int g = 0; g < 4; ++g)
                    *reinterpret_cast<uint4*>(A + (4 * w + g) * SBO) =
                        make_uint4(e[w][4 * g], e[w][4 * g + 1], e[w][4 * g + 2], e[w][4 * g + 3]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&a_full[s]);
            NMDLM_ASTAMP(a, 0, 100 + kt);
        }
    } else if (warp < WARP_MMA) {
        // ------------------------------------------ scores, weights, P^T in shared memory
        const int ts = tid - NVW * 32;
        const int k = ts % KT, qq = ts / KT;  // key row of the tile, query eighth-group
        uint4 qw[QQ];
        int cq[QQ];
        float z[QQ];
#pragma unroll
        for (int i = 0; i < QQ; ++i) {
            qw[i] = q_s[qq * QQ + i];
            cq[i] = popc4(qw[i].x, qw[i].y, qw[i].z, qw[i].w);
            z[i] = 0.0f;
        }
        for (int kt = 0; kt < ntile; ++kt) {
            const int s = kt % NST, u = kt / NST;
            const int key = kt * KT + k;
            const bool valid = key < L;
            const uint4 kw = valid ? kv_s[key] : make_uint4(0u, 0u, 0u, 0u);
            uint32_t hl[QQ];
#pragma unroll
            for (int i = 0; i < QQ; ++i) {
                const int sc = popc4(qw[i].x & kw.x, qw[i].y & kw.y, qw[i].z & kw.z, qw[i].w & kw.w);
                const uint2 e = lut[DH + sc - cq[i]];
                hl[i] = valid ? e.x : 0u;
                z[i] = __fadd_rn(z[i], valid ? __uint_as_float(e.y) : 0.0f);
            }
            uint4 vh, vl;
            vh.x = (hl[0] & 0xffffu) | (hl[1] << 16);
            vh.y = (hl[2] & 0xffffu) | (hl[3] << 16);
            vh.z = (hl[4] & 0xffffu) | (hl[5] << 16);
            vh.w = (hl[6] & 0xffffu) | (hl[7] << 16);
            vl.x = (hl[0] >> 16) | (hl[1] & 0xffff0000u);
            vl.y = (hl[2] >> 16) | (hl[3] & 0xffff0000u);
            vl.z = (hl[4] >> 16) | (hl[5] & 0xffff0000u);
            vl.w = (hl[6] >> 16) | (hl[7] & 0xffff0000u);
            if (u > 0) {
                const bool ok = mbar_wait_bounded(&st_free[s], (u - 1) & 1, a.wait_ns);
                if (!__all_sync(0xffffffffu, ok) || *abort_flag) {
                    if (lane == 0) { *abort_flag = 1; raise_error(a.err, ERRBIT_TIMEOUT); }
                    break;
                }
            }
            // key row k of P^T: query group qq (hi) in column group qq, lo in NQ/8 + qq
            uint8_t* P = smem + OFF_P + s * P_BYTES + (k >> 3) * LBO + (k & 7) * 16;
            *reinterpret_cast<uint4*>(P + qq * SBO) = vh;
            *reinterpret_cast<uint4*>(P + (NQ / 8 + qq) * SBO) = vl;
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_full[s]);
            NMDLM_ASTAMP(a, NVW * 32, 200 + kt);
        }
        // Z per query: warp sums in a fixed order, then the 4 warps of a query group in order
#pragma unroll
        for (int i = 0; i < QQ; ++i) {
            float v = z[i];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
            if (lane == 0) z_s[(warp - NVW) * QQ + i] = v;
        }
    } else {
        // -------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16_mn(DH, NP);
            const uint64_t ad0 = smem_desc(smem_u32(smem + OFF_A), LBO, SBO);
            const uint64_t bd0 = smem_desc(smem_u32(smem + OFF_P), LBO, SBO);
            constexpr uint64_t KSTEP = 2 * LBO / 16;  // 16 keys = two core matrices
            for (int kt = 0; kt < ntile; ++kt) {
                const int s = kt % NST, u = kt / NST;
                NMDLM_ASTAMP(a, WARP_MMA * 32, 300 + 2 * kt);
                const bool ok = !*abort_flag && mbar_wait_bounded(&a_full[s], u & 1, a.wait_ns) &&
                                mbar_wait_bounded(&p_full[s], u & 1, a.wait_ns);
                if (!ok) {
                    *abort_flag = 1;
                    raise_error(a.err, ERRBIT_TIMEOUT);
                    break;
                }
                tc_fence_after();
                const uint64_t ad = ad0 + (uint64_t)(s * (A_BYTES >> 4));
                const uint64_t bd = bd0 + (uint64_t)(s * (P_BYTES >> 4));
#pragma unroll
                for (int kk = 0; kk < KT / 16; ++kk)
                    mma_f16(tmem, ad + kk * KSTEP, bd + kk * KSTEP, idesc, (kt > 0 || kk > 0) ? 1u : 0u);
                mma_commit(&st_free[s]);
                NMDLM_ASTAMP(a, WARP_MMA * 32, 301 + 2 * kt);
            }
            mma_commit(done);
        }
        __syncwarp();
    }
    __syncthreads();
    bool ok = !*abort_flag;
    if (ntile > 0) {
        const bool fin = mbar_wait_bounded(done, 0, ok ? a.wait_ns : 1000000000ull);
        if (!fin) ok = false;
    }
    // the normaliser of each query: its 4 scoring warps' sums, in order
    if (tid < NQ) {
        const int g = tid / QQ, i = tid % QQ;
        float zs = 0.0f;
        for (int w = 0; w < KT / 32; ++w) zs = __fadd_rn(zs, z_s[(g * (KT / 32) + w) * QQ + i]);
        zq_s[tid] = zs;
    }
    const bool aborted = __syncthreads_or(!ok);
    tc_fence_after();
    NMDLM_ASTAMP(a, 0, 42);
    if (!aborted && warp < 16) {
        // ------------------------------- epilogue: out = 2^16 (hi + lo) / Z (V was 2^-16)
        // warp w reads lanes 32 (w % 4) .. + 31 (channels) and queries 8 (w / 4) .. + 7
        const int q = warp & 3, n0 = (warp >> 2) * 8, d = q * 32 + lane;
        uint32_t vh[8], vl[8];
        tmem_ld8(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)n0, vh);
        tmem_ld8(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(NQ + n0), vl);
        const int D = a.H * DH;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int n = n0 + j;
            if (n < nq) {
                const float o = __fmul_rn(__fadd_rn(__uint_as_float(vh[j]), __uint_as_float(vl[j])), 65536.0f);
                a.out[(size_t)((q0 + n) * a.T + t) * D + h * DH + d] = __fdiv_rn(o, zq_s[n]);
            }
        }
    }
    if (aborted && tid == 0) raise_error(a.err, ERRBIT_TIMEOUT);
    tc_fence_before();
    __syncthreads();
    NMDLM_ASTAMP(a, 0, 43);
    if (warp == WARP_MMA) tmem_dealloc(tmem, NCOL);
}

// UNSUPPORTED unless d_head is 128 and every key's words fit in shared memory: three
// operand stages where they fit (the scoring, V^T and MMA roles then overlap instead of
// pacing each other tile by tile), else two.
nmdlm_status launch_attention_tc(const AttnArgs& a, cudaStream_t stream) {
    using namespace attn3;
    if (a.dh != DH || a.L < 1 || a.B < 1) return NMDLM_ERR_UNSUPPORTED;
    const dim3 grid(a.H, a.T, (a.B + NQ - 1) / NQ);
    cudaError_t le;
    if (Lay<3>::smem_bytes(a.L) <= 225 * 1024) {
        const size_t smem = Lay<3>::smem_bytes(a.L);
        if (ensure_dyn_smem((const void*)k_attention_tc<3>, smem) != NMDLM_OK) return NMDLM_ERR_CUDA;
        le = launch_pdl(k_attention_tc<3>, grid, dim3(NTHREADS), smem, stream, 1, a);
    } else {
        const size_t smem = Lay<2>::smem_bytes(a.L);
        if (smem > 225 * 1024) return NMDLM_ERR_UNSUPPORTED;
        if (ensure_dyn_smem((const void*)k_attention_tc<2>, smem) != NMDLM_OK) return NMDLM_ERR_CUDA;
        le = launch_pdl(k_attention_tc<2>, grid, dim3(NTHREADS), smem, stream, 1, a);
    }
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

}  // namespace nmdlm
