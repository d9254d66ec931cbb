// attention.cu -- binary-binary (BBM) spike attention currents.
//
// For one timestep t and head h (the paper names binary-binary multiplication and a
// spiking attention in every layer, Fig. 1, without an equation; reading):
//   score[b][j] = popcount(q_b AND k_j)        integer in [0, d_head]
//   p[b][j]     = softmax_j(alpha * score)     (fp32)
//   out[b][c]   = sum_j p[b][j] * v_j[c]
// Because v is binary, out[b][c] = (1/Z_b) * sum over keys j with v_j[c] = 1 of
// exp(alpha * (score[b][j] - max_b)), so the mixture only visits the set bits of the
// transposed V spikes.  Scores are small integers, so exp is a table of d_head + 1
// entries shared by every query.  The IF that turns these currents into spikes runs
// in the IF-encode kernel.
#include <algorithm>

#include "internal.h"

namespace nmdlm {

namespace attn {
constexpr int NTHREADS = 512;
constexpr int KCH = 256;  // keys per mixture chunk
constexpr int QT = 64;    // queries per CTA (grid.z covers larger blocks)
}  // namespace attn

// grid (H, T, ceil(B / QT)); one CTA owns up to QT queries of one (timestep, head).
__global__ void __launch_bounds__(attn::NTHREADS) k_attention(AttnArgs a) {
    pdl_wait();
    using namespace attn;
    extern __shared__ __align__(16) uint8_t sm[];
    const int h = blockIdx.x, t = blockIdx.y, q0 = blockIdx.z * QT;
    const int B = min(QT, a.B - q0), L = a.L, dh = a.dh, DW = dh >> 5;
    const int WD = words_of(a.H * dh);
    const int LW = words_of(L);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = NTHREADS / 32;

    uint32_t* q_s = (uint32_t*)sm;                 // [B][DW]
    float* e_s = (float*)(q_s + B * DW);           // [dh + 1]
    int* mx_s = (int*)(e_s + dh + 1);              // [B]
    float* z_s = (float*)(mx_s + B);               // [B]
    uint32_t* vt_s = (uint32_t*)(z_s + B);         // [dh][LW]  V^T bits over keys
    float* w_s = (float*)(vt_s + (size_t)dh * LW); // [KCH][32] weights of 32 queries
    uint8_t* sc_s = (uint8_t*)(w_s + (size_t)KCH * 32); // [B][L]

    for (int i = tid; i < B * DW; i += NTHREADS) {
        const int b = i / DW, w = i % DW;
        q_s[i] = a.q[(size_t)((q0 + b) * a.T + t) * WD + h * DW + w];
    }
    for (int g = tid; g <= dh; g += NTHREADS) e_s[g] = expf(-__fmul_rn(a.alpha, (float)g));
    __syncthreads();

    // Scores (one key per thread) and V^T (one warp transposes 32 keys at a time).
    const uint32_t* kbase = a.k + (size_t)t * a.Ls * WD + h * DW;
    const uint32_t* vbase = a.v + (size_t)t * a.Ls * WD + h * DW;
    for (int j0 = warp * 32; j0 < L; j0 += nwarp * 32) {
        const int j = j0 + lane;
        const bool jv = j < L;
        uint32_t kw[8], vw[8];
#pragma unroll
        for (int w = 0; w < 8; ++w) {
            kw[w] = (w < DW && jv) ? kbase[(size_t)j * WD + w] : 0u;
            vw[w] = (w < DW && jv) ? vbase[(size_t)j * WD + w] : 0u;
        }
        if (jv) {
            for (int b = 0; b < B; ++b) {
                int s = 0;
#pragma unroll
                for (int w = 0; w < 8; ++w)
                    if (w < DW) s += __popc(q_s[b * DW + w] & kw[w]);
                sc_s[(size_t)b * L + j] = (uint8_t)s;
            }
        }
#pragma unroll
        for (int w = 0; w < 8; ++w)
            if (w < DW) vt_s[(size_t)(w * 32 + lane) * LW + (j0 >> 5)] = warp_transpose32(vw[w]);
    }
    __syncthreads();

    // Per-query max score and softmax normaliser (one warp per query).
    for (int b = warp; b < B; b += nwarp) {
        int m = 0;
        for (int j = lane; j < L; j += 32) m = max(m, (int)sc_s[(size_t)b * L + j]);
        for (int o = 16; o > 0; o >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
        float z = 0.0f;
        for (int j = lane; j < L; j += 32) z += e_s[m - sc_s[(size_t)b * L + j]];
        for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
        if (lane == 0) {
            mx_s[b] = m;
            z_s[b] = z;
        }
    }
    __syncthreads();

    // Mixture: a warp owns channels c = warp, warp + 16, ...; lane = query.  For each
    // channel the warp walks the set bits of V^T[c] (uniform across the warp) and adds
    // the key's softmax weight w[j][lane], a conflict-free row read.
    constexpr int CPW = 16;  // channels per warp for d_head <= 256
    float acc[CPW];
#pragma unroll
    for (int i = 0; i < CPW; ++i) acc[i] = 0.0f;
    for (int b0 = 0; b0 < B; b0 += 32) {
        const int qb = b0 + lane;
#pragma unroll
        for (int i = 0; i < CPW; ++i) acc[i] = 0.0f;
        for (int k0 = 0; k0 < L; k0 += KCH) {
            const int kn = min(KCH, L - k0);
            for (int i = tid; i < kn * 32; i += NTHREADS) {
                const int jj = i >> 5, q = b0 + (i & 31);
                w_s[i] = q < B ? e_s[mx_s[q] - sc_s[(size_t)q * L + k0 + jj]] : 0.0f;
            }
            __syncthreads();
#pragma unroll
            for (int i = 0; i < CPW; ++i) {
                const int c = warp + i * nwarp;
                if (c < dh) {
                    for (int w = 0; w < (kn + 31) / 32; ++w) {
                        uint32_t m = vt_s[(size_t)c * LW + (k0 >> 5) + w];
                        while (m) {
                            const int jj = w * 32 + __ffs(m) - 1;
                            m &= m - 1;
                            acc[i] += w_s[jj * 32 + lane];
                        }
                    }
                }
            }
            __syncthreads();
        }
        const int D = a.H * dh;
        if (qb < B) {
#pragma unroll
            for (int i = 0; i < CPW; ++i) {
                const int c = warp + i * nwarp;
                if (c < dh)
                    a.out[(size_t)((q0 + qb) * a.T + t) * D + h * dh + c] =
                        __fdiv_rn(acc[i], z_s[qb]);
            }
        }
    }
}

size_t attention_smem_bytes(int B, int L, int dh) {
    const int DW = dh / 32, LW = (L + 31) / 32;
    return (size_t)4 * B * DW + 4 * (dh + 1) + 8 * B + (size_t)4 * dh * LW +
           (size_t)4 * attn::KCH * 32 + (size_t)B * L + 64;
}

nmdlm_status launch_attention(nmdlm_ctx*, const AttnArgs& a, cudaStream_t stream) {
    if (a.dh % 32 || a.dh > 256) return NMDLM_ERR_UNSUPPORTED;
    if (a.B < 1 || a.L < 1) return NMDLM_ERR_UNSUPPORTED;
    const size_t smem = attention_smem_bytes(std::min(a.B, attn::QT), a.L, a.dh);
    if (smem > 220 * 1024) return NMDLM_ERR_UNSUPPORTED;
    if (ensure_dyn_smem((const void*)k_attention, smem) != NMDLM_OK) return NMDLM_ERR_CUDA;
    dim3 grid(a.H, a.T, (a.B + attn::QT - 1) / attn::QT);
    const cudaError_t le = launch_pdl(k_attention, dim3(grid), dim3(attn::NTHREADS), smem,
                                      stream, 1, a);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

}  // namespace nmdlm

// ----------------------------------------------------------- tensor cores ----
// The same attention with both contractions on the tensor cores (mma.sync m16n8k16,
// fp32 accumulation):
//   S = Q K^T   (queries x keys; 0/1 spikes enter as fp16 2^-16 (subnormal 0x0100,
//                multiplied exactly), so the sums are exact multiples of 2^-32 and the
//                integer scores are recovered exactly),
//   O = P V     (P = exp(alpha (S - max)) split into two fp16 halves, hi + lo, so the
//                mixture keeps ~2^-22 relative precision; V as 2^-16, removed at the end).
// A warp owns one range of keys for every query of the CTA's tile (one or two 16-row
// m-tiles), so each key's bits are expanded once; it keeps a running (flash-style)
// maximum, normaliser and output, and the warps merge through shared memory at the end.
namespace nmdlm {
namespace attn2 {
constexpr int QT = 64;  // queries per CTA (grid.z covers larger blocks)
}  // namespace attn2

// bits 0 and 1 of x -> fp16x2 {bit0 ? 2^-16 : 0, bit1 ? 2^-16 : 0}
__device__ __forceinline__ uint32_t bitpair_e16(uint32_t x) {
    return ((x & 3u) * 0x00800100u) & 0x01000100u;
}
// the bit pair at byte `byte` of xs (bit 0) and xs1 = xs >> 1 (bit 0) -> fp16x2 of 2^-16 / 0
__device__ __forceinline__ uint32_t bytepair_e16(uint32_t xs, uint32_t xs1, int byte) {
    return __byte_perm(xs, xs1, (byte << 4) | ((4 + byte) << 12)) & 0x01000100u;
}

__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
    __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}

// K rows and V^T of head h at timestep t into shared memory.  Every key's slice is
// requested at once with asynchronous copies (a loop of plain loads waits one memory
// latency per iteration); V lands in a staging area and each warp then transposes 32
// keys x 32 channels at a time: bit j % 32 of vt_s[c][j / 32] is v[j][c].
template <int DH, int NTHREADS>
__device__ __forceinline__ void load_head_kv(const AttnArgs& a, int t, int h, int L, int LW,
                                             uint32_t* k_s, uint32_t* vt_s, uint32_t* vst) {
    constexpr int DW = DH / 32;
    const int WD = words_of(a.H * DH);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint32_t* kbase = a.k + (size_t)t * a.Ls * WD + h * DW;
    const uint32_t* vbase = a.v + (size_t)t * a.Ls * WD + h * DW;
    const bool wide = DW == 4 && (WD & 3) == 0 &&
                      ((((uintptr_t)kbase) | ((uintptr_t)vbase) | ((uintptr_t)k_s) | ((uintptr_t)vst)) & 15) == 0;
    if (wide) {
        for (int j = tid; j < L; j += NTHREADS) {
            cp_async16(k_s + (size_t)j * DW, kbase + (size_t)j * WD, 16u);
            cp_async16(vst + (size_t)j * DW, vbase + (size_t)j * WD, 16u);
        }
    } else {
        for (int i = tid; i < L * DW; i += NTHREADS) {
            const int j = i / DW, w = i % DW;
            cp_async4(k_s + i, kbase + (size_t)j * WD + w, 4u);
            cp_async4(vst + i, vbase + (size_t)j * WD + w, 4u);
        }
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    for (int j0 = warp * 32; j0 < L; j0 += NTHREADS) {
        const int j = j0 + lane;
        uint32_t vw[DW];
#pragma unroll
        for (int w = 0; w < DW; ++w) vw[w] = j < L ? vst[(size_t)j * DW + w] : 0u;
#pragma unroll
        for (int w = 0; w < DW; ++w)
            vt_s[(size_t)(w * 32 + lane) * LW + (j0 >> 5)] = warp_transpose32(vw[w]);
    }
}

// grid (H, T, ceil(B / QT)); MW = 16-query m-tiles per warp (1 or 2).  Warp w takes
// m-tile group w % MG and key range w / MG.
template <int DH, int WARPS, int MW>
__global__ void __launch_bounds__(WARPS * 32, 1) k_attention_mma(AttnArgs a) {
    pdl_wait();
    using namespace attn2;
    constexpr int NTHREADS = WARPS * 32;
    constexpr int DW = DH / 32;    // words per key row of this head
    constexpr int NKS = DH / 16;   // k steps of the score product
    constexpr int NNT = DH / 8;    // n tiles of the output product
    extern __shared__ __align__(16) uint8_t sm[];
    const int h = blockIdx.x, t = blockIdx.y, q0 = blockIdx.z * QT;
    const int B = min(QT, a.B - q0), L = a.L;
    const int WD = words_of(a.H * DH);
    const int LW = words_of(L);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g = lane >> 2, c = lane & 3;
    const int MT = ((B + 15) / 16 + MW - 1) / MW * MW;  // m-tiles, padded to a multiple of MW
    const int MG = MT / MW;                               // m-tile groups
    const int KR = WARPS / MG;                            // key ranges

    float* e_s = (float*)sm;                                  // [DH + 1]
    uint32_t* q_s = (uint32_t*)(e_s + DH + 1 + 3);            // [QT][DW]
    uint4* qf_s = (uint4*)(q_s + QT * DW);                    // [QT/16][NKS][32] A fragments
    uint32_t* k_s = (uint32_t*)(qf_s + (QT / 16) * NKS * 32);  // [L][DW]
    uint32_t* vt_s = k_s + (size_t)L * DW;                    // [DH][LW]
    // merge area (reuses k_s/vt_s after the key loop): [WARPS][16 MW][DH] + m, l
    float* o_s = (float*)k_s;
    float* m_s = o_s + (size_t)WARPS * 16 * MW * DH;
    float* l_s = m_s + WARPS * 16 * MW;

    for (int gg = tid; gg <= DH; gg += NTHREADS) e_s[gg] = expf(-__fmul_rn(a.alpha, (float)gg));
    for (int i = tid; i < MT * 16 * DW; i += NTHREADS) {
        const int b = i / DW, w = i % DW;
        q_s[i] = b < B ? a.q[(size_t)((q0 + b) * a.T + t) * WD + h * DW + w] : 0u;
    }
    load_head_kv<DH, NTHREADS>(a, t, h, L, LW, k_s, vt_s, vt_s + (size_t)DH * LW);
    __syncthreads();
    // Q as fp16 A fragments (rows 16 mt + g and + 8; channels 16 ks + 2c, +1 and + 8, + 9)
    for (int i = tid; i < MT * NKS * 32; i += NTHREADS) {
        const int ln = i & 31, ks = (i >> 5) % NKS, mt_ = i / (NKS * 32);
        const int gg = ln >> 2, ch = 16 * ks + 2 * (ln & 3);
        const uint32_t* r0 = q_s + (mt_ * 16 + gg) * DW;
        const uint32_t* r1 = q_s + (mt_ * 16 + gg + 8) * DW;
        qf_s[i] = make_uint4(bitpair_e16(r0[ch >> 5] >> (ch & 31)),
                             bitpair_e16(r1[ch >> 5] >> (ch & 31)),
                             bitpair_e16(r0[(ch + 8) >> 5] >> ((ch + 8) & 31)),
                             bitpair_e16(r1[(ch + 8) >> 5] >> ((ch + 8) & 31)));
    }
    __syncthreads();

    const int mg = warp % MG, kr = warp / MG;
    const bool active = kr < KR;
    const int nblk = (L + 31) / 32;
    const int kb0 = active ? kr * nblk / KR : 0, kb1 = active ? (kr + 1) * nblk / KR : 0;
    const uint4* qf = qf_s + (size_t)(mg * MW) * NKS * 32 + lane;

    float o[MW][NNT][4];
#pragma unroll
    for (int u = 0; u < MW; ++u)
#pragma unroll
        for (int n = 0; n < NNT; ++n) o[u][n][0] = o[u][n][1] = o[u][n][2] = o[u][n][3] = 0.0f;
    int mrow[MW][2];      // running maximum score of rows g and g + 8 (-1: none yet)
    float lrow[MW][2];    // this thread's part of the running normaliser
#pragma unroll
    for (int u = 0; u < MW; ++u) { mrow[u][0] = mrow[u][1] = -1; lrow[u][0] = lrow[u][1] = 0.f; }

    for (int kb = kb0; kb < kb1; ++kb) {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int key0 = kb * 32 + half * 16;
            // scores of 16 keys: n tile 0 = keys key0..key0+7, n tile 1 = key0+8..key0+15
            float sacc[MW][2][4];
#pragma unroll
            for (int u = 0; u < MW; ++u)
#pragma unroll
                for (int nt = 0; nt < 2; ++nt) sacc[u][nt][0] = sacc[u][nt][1] = sacc[u][nt][2] = sacc[u][nt][3] = 0.f;
            const uint32_t* kr0 = k_s + (size_t)min(key0 + g, L - 1) * DW;
            const uint32_t* kr1 = k_s + (size_t)min(key0 + 8 + g, L - 1) * DW;
            const bool kv0 = key0 + g < L, kv1 = key0 + 8 + g < L;
            // channels 16 ks + 2c, +1 and +8, +9 of a key sit at bytes 2 (ks & 1) and + 1 of
            // its word (ks / 2) shifted right by 2c
#pragma unroll
            for (int wi = 0; wi < DW; ++wi) {
                const uint32_t w0 = kv0 ? kr0[wi] : 0u, w1 = kv1 ? kr1[wi] : 0u;
                const uint32_t w0s = w0 >> (2 * c), w0s1 = w0 >> (2 * c + 1);
                const uint32_t w1s = w1 >> (2 * c), w1s1 = w1 >> (2 * c + 1);
#pragma unroll
                for (int hk = 0; hk < 2; ++hk) {
                    const int ks = 2 * wi + hk;
                    const uint32_t b00 = bytepair_e16(w0s, w0s1, 2 * hk);
                    const uint32_t b01 = bytepair_e16(w0s, w0s1, 2 * hk + 1);
                    const uint32_t b10 = bytepair_e16(w1s, w1s1, 2 * hk);
                    const uint32_t b11 = bytepair_e16(w1s, w1s1, 2 * hk + 1);
#pragma unroll
                    for (int u = 0; u < MW; ++u) {
                        const uint4 qv = qf[(u * NKS + ks) * 32];
                        const uint32_t qa[4] = {qv.x, qv.y, qv.z, qv.w};
                        mma16816(sacc[u][0], qa, b00, b01);
                        mma16816(sacc[u][1], qa, b10, b11);
                    }
                }
            }
            bool kv[2][2];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                kv[nt][0] = key0 + nt * 8 + 2 * c < L;
                kv[nt][1] = key0 + nt * 8 + 2 * c + 1 < L;
            }
            uint32_t ph[MW][4], pl[MW][4];
#pragma unroll
            for (int u = 0; u < MW; ++u) {
                int sc[2][4];
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        sc[nt][e] = __float2int_rn(__fmul_rn(sacc[u][nt][e], 4294967296.0f));
                // block maximum of each row (4 lanes of a group share a row)
#pragma unroll
                for (int r = 0; r < 2; ++r) {
                    int bm = -1;
#pragma unroll
                    for (int nt = 0; nt < 2; ++nt) {
                        if (kv[nt][0]) bm = max(bm, sc[nt][2 * r]);
                        if (kv[nt][1]) bm = max(bm, sc[nt][2 * r + 1]);
                    }
                    bm = max(bm, __shfl_xor_sync(0xffffffffu, bm, 1));
                    bm = max(bm, __shfl_xor_sync(0xffffffffu, bm, 2));
                    if (bm > mrow[u][r]) {
                        if (mrow[u][r] >= 0) {
                            const float f = e_s[bm - mrow[u][r]];
                            lrow[u][r] *= f;
#pragma unroll
                            for (int n = 0; n < NNT; ++n) {
                                o[u][n][2 * r] *= f;
                                o[u][n][2 * r + 1] *= f;
                            }
                        }
                        mrow[u][r] = bm;
                    }
                }
                float p[2][4];
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int r = e >> 1;
                        p[nt][e] = kv[nt][e & 1] ? e_s[mrow[u][r] - sc[nt][e]] : 0.0f;
                        lrow[u][r] += p[nt][e];
                    }
                // P = P_hi + P_lo, both fp16: the two products give P V to ~2^-22 relative
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float x0 = p[q >> 1][2 * (q & 1)], x1 = p[q >> 1][2 * (q & 1) + 1];
                    const __half2 hi = __floats2half2_rn(x0, x1);
                    const float2 hf = __half22float2(hi);
                    ph[u][q] = *reinterpret_cast<const uint32_t*>(&hi);
                    pl[u][q] = pack_f16x2(x0 - hf.x, x1 - hf.y);
                }
            }
            // O += P V: B fragment of n tile = keys (2c, 2c+1 | 2c+8, 2c+9) at channel 8 n + g
#pragma unroll
            for (int n = 0; n < NNT; ++n) {
                const uint32_t vw = vt_s[(size_t)(8 * n + g) * LW + kb];
                const uint32_t vs = vw >> (2 * c), vs1 = vw >> (2 * c + 1);
                const uint32_t b0 = bytepair_e16(vs, vs1, 2 * half);
                const uint32_t b1 = bytepair_e16(vs, vs1, 2 * half + 1);
#pragma unroll
                for (int u = 0; u < MW; ++u) {
                    mma16816(o[u][n], ph[u], b0, b1);
                    mma16816(o[u][n], pl[u], b0, b1);
                }
            }
        }
    }
    // normaliser of each row summed over the 4 lanes of its group
#pragma unroll
    for (int u = 0; u < MW; ++u)
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            lrow[u][r] += __shfl_xor_sync(0xffffffffu, lrow[u][r], 1);
            lrow[u][r] += __shfl_xor_sync(0xffffffffu, lrow[u][r], 2);
        }
    __syncthreads();  // k_s / vt_s are reused as the merge area
    if (active) {
#pragma unroll
        for (int u = 0; u < MW; ++u) {
            float* ow = o_s + ((size_t)warp * MW + u) * 16 * DH;
#pragma unroll
            for (int n = 0; n < NNT; ++n) {
                const int ch = 8 * n + 2 * c;
                *reinterpret_cast<float2*>(ow + g * DH + ch) = make_float2(o[u][n][0], o[u][n][1]);
                *reinterpret_cast<float2*>(ow + (g + 8) * DH + ch) = make_float2(o[u][n][2], o[u][n][3]);
            }
            if (c == 0) {
                m_s[(warp * MW + u) * 16 + g] = (float)mrow[u][0];
                m_s[(warp * MW + u) * 16 + g + 8] = (float)mrow[u][1];
                l_s[(warp * MW + u) * 16 + g] = lrow[u][0];
                l_s[(warp * MW + u) * 16 + g + 8] = lrow[u][1];
            }
        }
    }
    __syncthreads();
    // merge the key ranges of each query row; undo the 2^-16 of V; write the currents
    const int D = a.H * DH;
    for (int i = tid; i < B * DH; i += NTHREADS) {
        const int b = i / DH, ch = i % DH;
        const int mt = b / 16, row = b % 16;
        const int grp = mt / MW, u = mt % MW;
        int mstar = -1;
        for (int k2 = 0; k2 < KR; ++k2)
            mstar = max(mstar, (int)m_s[((k2 * MG + grp) * MW + u) * 16 + row]);
        float num = 0.0f, den = 0.0f;
        for (int k2 = 0; k2 < KR; ++k2) {
            const int w = (k2 * MG + grp) * MW + u;
            const int mw = (int)m_s[w * 16 + row];
            if (mw < 0) continue;  // this range held no key
            const float f = e_s[mstar - mw];
            num += o_s[((size_t)w * 16 + row) * DH + ch] * f;
            den += l_s[w * 16 + row] * f;
        }
        a.out[(size_t)((q0 + b) * a.T + t) * D + h * DH + ch] =
            __fdiv_rn(__fmul_rn(num, 65536.0f), den);
    }
}

// Warp-pair form for tiles of more than 16 queries.  A pair of warps owns two m-tiles
// (32 queries) and one range of keys: warp r computes the scores and the softmax of
// m-tile r, the pair swaps the fp16 P fragments and rescale factors through shared
// memory (double-buffered, one named barrier per 16 keys), and warp r then forms the
// mixture for channel half r of both m-tiles.  Each warp keeps half the output
// registers of the one-warp form, so twice the warps fit.
template <int DH, int WARPS>
__global__ void __launch_bounds__(WARPS * 32, 1) k_attention_pair(AttnArgs a) {
    pdl_wait();
    using namespace attn2;
    constexpr int NTHREADS = WARPS * 32, PAIRS = WARPS / 2;
    constexpr int DW = DH / 32, NKS = DH / 16, NNT = DH / 8, NNH = NNT / 2;
    // exchange words per lane: P hi (4), P lo (4), factors (2), padding (2) -- a multiple
    // of 4 so every lane's 16-byte accesses stay aligned
    constexpr int XW = 12;
    extern __shared__ __align__(16) uint8_t sm[];
    const int h = blockIdx.x, t = blockIdx.y, q0 = blockIdx.z * QT;
    const int B = min(QT, a.B - q0), L = a.L;
    const int WD = words_of(a.H * DH);
    const int LW = words_of(L);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g = lane >> 2, c = lane & 3;
    const int MT = ((B + 15) / 16 + 1) / 2 * 2;  // m-tiles, padded to pairs
    const int MG = MT / 2;                        // m-tile pairs
    const int KR = PAIRS / MG;                    // key ranges

    float* e_s = (float*)sm;                                   // [DH + 1]
    uint32_t* q_s = (uint32_t*)(e_s + DH + 1 + 3);             // [QT][DW]
    uint4* qf_s = (uint4*)(q_s + QT * DW);                     // [QT/16][NKS][32]
    uint32_t* xbuf = (uint32_t*)(qf_s + (QT / 16) * NKS * 32);  // [PAIRS][2][2][32][XW]
    uint32_t* k_s = xbuf + PAIRS * 2 * 2 * 32 * XW;            // [L][DW]
    uint32_t* vt_s = k_s + (size_t)L * DW;                     // [DH][LW]
    float* o_s = (float*)k_s;                  // merge: [PAIRS][2][16][DH] over k_s / vt_s
    float* m_s = o_s + (size_t)PAIRS * 2 * 16 * DH;
    float* l_s = m_s + PAIRS * 2 * 16;

    for (int gg = tid; gg <= DH; gg += NTHREADS) e_s[gg] = expf(-__fmul_rn(a.alpha, (float)gg));
    for (int i = tid; i < MT * 16 * DW; i += NTHREADS) {
        const int b = i / DW, w = i % DW;
        q_s[i] = b < B ? a.q[(size_t)((q0 + b) * a.T + t) * WD + h * DW + w] : 0u;
    }
    load_head_kv<DH, NTHREADS>(a, t, h, L, LW, k_s, vt_s, vt_s + (size_t)DH * LW);
    __syncthreads();
    for (int i = tid; i < MT * NKS * 32; i += NTHREADS) {
        const int ln = i & 31, ks = (i >> 5) % NKS, mt_ = i / (NKS * 32);
        const int gg = ln >> 2, ch = 16 * ks + 2 * (ln & 3);
        const uint32_t* r0 = q_s + (mt_ * 16 + gg) * DW;
        const uint32_t* r1 = q_s + (mt_ * 16 + gg + 8) * DW;
        qf_s[i] = make_uint4(bitpair_e16(r0[ch >> 5] >> (ch & 31)),
                             bitpair_e16(r1[ch >> 5] >> (ch & 31)),
                             bitpair_e16(r0[(ch + 8) >> 5] >> ((ch + 8) & 31)),
                             bitpair_e16(r1[(ch + 8) >> 5] >> ((ch + 8) & 31)));
    }
    __syncthreads();

    const int pr = warp >> 1, role = warp & 1;
    const int mg = pr % MG, kr = pr / MG;
    const bool active = kr < KR;
    const int nblk = (L + 31) / 32;
    const int kb0 = active ? kr * nblk / KR : 0, kb1 = active ? (kr + 1) * nblk / KR : 0;
    const uint4* qf = qf_s + (size_t)(mg * 2 + role) * NKS * 32 + lane;
    uint32_t* xmine = xbuf + ((size_t)(pr * 2) * 2 + role) * 32 * XW + lane * XW;   // + buf * 2*32*XW
    uint32_t* xpeer = xbuf + ((size_t)(pr * 2) * 2 + (role ^ 1)) * 32 * XW + lane * XW;

    // output of this warp's channel half: own m-tile (`role`) and the partner's
    float oo[NNH][4], op[NNH][4];
#pragma unroll
    for (int n = 0; n < NNH; ++n) {
        oo[n][0] = oo[n][1] = oo[n][2] = oo[n][3] = 0.0f;
        op[n][0] = op[n][1] = op[n][2] = op[n][3] = 0.0f;
    }
    int mrow[2] = {-1, -1};      // own m-tile: running maximum of rows g, g + 8
    float lrow[2] = {0.f, 0.f};  // own m-tile: this thread's part of the normaliser
    int buf = 0;

    for (int kb = kb0; kb < kb1; ++kb) {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int key0 = kb * 32 + half * 16;
            float sacc[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) sacc[nt][0] = sacc[nt][1] = sacc[nt][2] = sacc[nt][3] = 0.f;
            const uint32_t* kr0 = k_s + (size_t)min(key0 + g, L - 1) * DW;
            const uint32_t* kr1 = k_s + (size_t)min(key0 + 8 + g, L - 1) * DW;
            const bool kv0 = key0 + g < L, kv1 = key0 + 8 + g < L;
#pragma unroll
            for (int wi = 0; wi < DW; ++wi) {
                const uint32_t w0 = kv0 ? kr0[wi] : 0u, w1 = kv1 ? kr1[wi] : 0u;
                const uint32_t w0s = w0 >> (2 * c), w0s1 = w0 >> (2 * c + 1);
                const uint32_t w1s = w1 >> (2 * c), w1s1 = w1 >> (2 * c + 1);
#pragma unroll
                for (int hk = 0; hk < 2; ++hk) {
                    const uint4 qv = qf[(2 * wi + hk) * 32];
                    const uint32_t qa[4] = {qv.x, qv.y, qv.z, qv.w};
                    mma16816(sacc[0], qa, bytepair_e16(w0s, w0s1, 2 * hk), bytepair_e16(w0s, w0s1, 2 * hk + 1));
                    mma16816(sacc[1], qa, bytepair_e16(w1s, w1s1, 2 * hk), bytepair_e16(w1s, w1s1, 2 * hk + 1));
                }
            }
            bool kv[2][2];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                kv[nt][0] = key0 + nt * 8 + 2 * c < L;
                kv[nt][1] = key0 + nt * 8 + 2 * c + 1 < L;
            }
            int sc[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    sc[nt][e] = __float2int_rn(__fmul_rn(sacc[nt][e], 4294967296.0f));
            float fac[2] = {1.0f, 1.0f};
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                int bm = -1;
#pragma unroll
                for (int nt = 0; nt < 2; ++nt) {
                    if (kv[nt][0]) bm = max(bm, sc[nt][2 * r]);
                    if (kv[nt][1]) bm = max(bm, sc[nt][2 * r + 1]);
                }
                bm = max(bm, __shfl_xor_sync(0xffffffffu, bm, 1));
                bm = max(bm, __shfl_xor_sync(0xffffffffu, bm, 2));
                if (bm > mrow[r]) {
                    if (mrow[r] >= 0) fac[r] = e_s[bm - mrow[r]];
                    mrow[r] = bm;
                }
                lrow[r] *= fac[r];
            }
            float p[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int r = e >> 1;
                    p[nt][e] = kv[nt][e & 1] ? e_s[mrow[r] - sc[nt][e]] : 0.0f;
                    lrow[r] += p[nt][e];
                }
            uint32_t ph[4], pl[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float x0 = p[q >> 1][2 * (q & 1)], x1 = p[q >> 1][2 * (q & 1) + 1];
                const __half2 hi = __floats2half2_rn(x0, x1);
                const float2 hf = __half22float2(hi);
                ph[q] = *reinterpret_cast<const uint32_t*>(&hi);
                pl[q] = pack_f16x2(x0 - hf.x, x1 - hf.y);
            }
            // swap with the partner warp: its m-tile's P fragments and rescale factors
            uint32_t* mine = xmine + buf * 2 * 32 * XW;
            const uint32_t* peer = xpeer + buf * 2 * 32 * XW;
            *reinterpret_cast<uint4*>(mine) = make_uint4(ph[0], ph[1], ph[2], ph[3]);
            *reinterpret_cast<uint4*>(mine + 4) = make_uint4(pl[0], pl[1], pl[2], pl[3]);
            *reinterpret_cast<float2*>(mine + 8) = make_float2(fac[0], fac[1]);
            asm volatile("bar.sync %0, 64;" ::"r"(1 + pr) : "memory");
            const uint4 qh = *reinterpret_cast<const uint4*>(peer);
            const uint4 ql = *reinterpret_cast<const uint4*>(peer + 4);
            const float2 pf = *reinterpret_cast<const float2*>(peer + 8);
            const uint32_t pph[4] = {qh.x, qh.y, qh.z, qh.w}, ppl[4] = {ql.x, ql.y, ql.z, ql.w};
            buf ^= 1;
            // rescale where a running maximum grew (rare after the first keys)
            if (__any_sync(0xffffffffu, fac[0] != 1.0f || fac[1] != 1.0f || pf.x != 1.0f || pf.y != 1.0f)) {
#pragma unroll
                for (int n = 0; n < NNH; ++n) {
                    oo[n][0] *= fac[0];
                    oo[n][1] *= fac[0];
                    oo[n][2] *= fac[1];
                    oo[n][3] *= fac[1];
                    op[n][0] *= pf.x;
                    op[n][1] *= pf.x;
                    op[n][2] *= pf.y;
                    op[n][3] *= pf.y;
                }
            }
            // O += P V for this warp's channel half, both m-tiles
#pragma unroll
            for (int n = 0; n < NNH; ++n) {
                const uint32_t vw = vt_s[(size_t)(8 * (role * NNH + n) + g) * LW + kb];
                const uint32_t vs = vw >> (2 * c), vs1 = vw >> (2 * c + 1);
                const uint32_t b0 = bytepair_e16(vs, vs1, 2 * half);
                const uint32_t b1 = bytepair_e16(vs, vs1, 2 * half + 1);
                mma16816(oo[n], ph, b0, b1);
                mma16816(oo[n], pl, b0, b1);
                mma16816(op[n], pph, b0, b1);
                mma16816(op[n], ppl, b0, b1);
            }
        }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
        lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
    }
    __syncthreads();  // k_s / vt_s are reused as the merge area
    if (active) {
        float* wo = o_s + ((size_t)pr * 2 + role) * 16 * DH + role * (DH / 2);
        float* wp = o_s + ((size_t)pr * 2 + (role ^ 1)) * 16 * DH + role * (DH / 2);
#pragma unroll
        for (int n = 0; n < NNH; ++n) {
            const int ch = 8 * n + 2 * c;
            *reinterpret_cast<float2*>(wo + g * DH + ch) = make_float2(oo[n][0], oo[n][1]);
            *reinterpret_cast<float2*>(wo + (g + 8) * DH + ch) = make_float2(oo[n][2], oo[n][3]);
            *reinterpret_cast<float2*>(wp + g * DH + ch) = make_float2(op[n][0], op[n][1]);
            *reinterpret_cast<float2*>(wp + (g + 8) * DH + ch) = make_float2(op[n][2], op[n][3]);
        }
        if (c == 0) {  // the score owner of m-tile `role` holds its maximum and normaliser
            m_s[(pr * 2 + role) * 16 + g] = (float)mrow[0];
            m_s[(pr * 2 + role) * 16 + g + 8] = (float)mrow[1];
            l_s[(pr * 2 + role) * 16 + g] = lrow[0];
            l_s[(pr * 2 + role) * 16 + g + 8] = lrow[1];
        }
    }
    __syncthreads();
    const int D = a.H * DH;
    for (int i = tid; i < B * DH; i += NTHREADS) {
        const int b = i / DH, ch = i % DH;
        const int mt = b / 16, row = b % 16;
        const int grp = mt / 2, u = mt % 2;
        int mstar = -1;
        for (int k2 = 0; k2 < KR; ++k2)
            mstar = max(mstar, (int)m_s[((k2 * MG + grp) * 2 + u) * 16 + row]);
        float num = 0.0f, den = 0.0f;
        for (int k2 = 0; k2 < KR; ++k2) {
            const int sl = (k2 * MG + grp) * 2 + u;
            const int mw = (int)m_s[sl * 16 + row];
            if (mw < 0) continue;
            const float f = e_s[mstar - mw];
            num += o_s[((size_t)sl * 16 + row) * DH + ch] * f;
            den += l_s[sl * 16 + row] * f;
        }
        a.out[(size_t)((q0 + b) * a.T + t) * D + h * DH + ch] =
            __fdiv_rn(__fmul_rn(num, 65536.0f), den);
    }
}

size_t attention_pair_smem_bytes(int L, int dh, int warps) {
    const int DW = dh / 32, LW = (L + 31) / 32, pairs = warps / 2;
    const size_t head = 4 * (size_t)(dh + 4) + 4 * (size_t)attn2::QT * DW +
                        16 * (size_t)(attn2::QT / 16) * (dh / 16) * 32 +
                        4 * (size_t)pairs * 2 * 2 * 32 * 12;
    const size_t kv = 8 * (size_t)L * DW + 4 * (size_t)dh * LW;  // K, V^T, staged V rows
    const size_t merge = 4 * (size_t)pairs * 2 * 16 * dh + 8 * (size_t)pairs * 2 * 16;
    return head + std::max(kv, merge) + 64;
}

template <int DH, int WARPS>
static nmdlm_status launch_attention_pair_t(const AttnArgs& a, cudaStream_t stream) {
    const size_t smem = attention_pair_smem_bytes(a.L, DH, WARPS);
    if (smem > 220 * 1024) return launch_attention(nullptr, a, stream);
    if (ensure_dyn_smem((const void*)k_attention_pair<DH, WARPS>, smem) != NMDLM_OK)
        return NMDLM_ERR_CUDA;
    dim3 grid(a.H, a.T, (a.B + attn2::QT - 1) / attn2::QT);
    const cudaError_t le = launch_pdl(k_attention_pair<DH, WARPS>, grid, dim3(WARPS * 32), smem,
                                      stream, 1, a);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

size_t attention_mma_smem_bytes(int B, int L, int dh, int warps, int mw) {
    const int DW = dh / 32, LW = (L + 31) / 32;
    const size_t head = 4 * (size_t)(dh + 4) + 4 * (size_t)attn2::QT * DW +
                        16 * (size_t)(attn2::QT / 16) * (dh / 16) * 32;
    const size_t kv = 8 * (size_t)L * DW + 4 * (size_t)dh * LW;  // K, V^T, staged V rows
    const size_t merge = 4 * (size_t)warps * 16 * mw * dh + 8 * (size_t)warps * 16 * mw;
    (void)B;
    return head + std::max(kv, merge) + 64;
}

template <int DH, int WARPS, int MW>
static nmdlm_status launch_attention_mma_t(const AttnArgs& a, cudaStream_t stream) {
    const size_t smem = attention_mma_smem_bytes(std::min(a.B, attn2::QT), a.L, DH, WARPS, MW);
    if (smem > 220 * 1024) return launch_attention(nullptr, a, stream);
    if (ensure_dyn_smem((const void*)k_attention_mma<DH, WARPS, MW>, smem) != NMDLM_OK)
        return NMDLM_ERR_CUDA;
    dim3 grid(a.H, a.T, (a.B + attn2::QT - 1) / attn2::QT);
    const cudaError_t le = launch_pdl(k_attention_mma<DH, WARPS, MW>, grid, dim3(WARPS * 32),
                                      smem, stream, 1, a);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

// Tensor-core attention when the head width allows, else CUDA cores.  Tiles of more
// than 16 queries let every warp take two m-tiles.
nmdlm_status launch_attention_best(const AttnArgs& a, cudaStream_t stream) {
    if (a.B < 1 || a.L < 1) return launch_attention(nullptr, a, stream);
    const bool two = std::min(a.B, attn2::QT) > 16;
    switch (a.dh) {
        case 32: return two ? launch_attention_mma_t<32, 16, 2>(a, stream)
                            : launch_attention_mma_t<32, 16, 1>(a, stream);
        case 64: return two ? launch_attention_mma_t<64, 12, 2>(a, stream)
                            : launch_attention_mma_t<64, 16, 1>(a, stream);
        case 96: return two ? launch_attention_mma_t<96, 8, 2>(a, stream)
                            : launch_attention_mma_t<96, 12, 1>(a, stream);
        case 128: {
            const nmdlm_status st = launch_attention_tc(a, stream);
            if (st != NMDLM_ERR_UNSUPPORTED) return st;
            return two ? launch_attention_pair_t<128, 12>(a, stream)
                       : launch_attention_mma_t<128, 12, 1>(a, stream);
        }
        default: return launch_attention(nullptr, a, stream);
    }
}

}  // namespace nmdlm
