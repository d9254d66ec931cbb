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
    static size_t configured = 0;
    if (smem > configured) {
        if (cuda_status(cudaFuncSetAttribute(
                k_attention, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != NMDLM_OK)
            return NMDLM_ERR_CUDA;
        configured = smem;
    }
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
// fp16 operands holding exact 0/1 spikes, fp32 accumulation):
//   S = Q K^T   (queries x keys; the scores are exact integers),
//   O = P V     (P = exp(alpha (S - max)) rounded to fp16, relative error <= 2^-11).
// A warp owns 16 queries and one range of keys and keeps a running (flash-style)
// maximum, normaliser and output; the warps of one query tile merge at the end.
namespace nmdlm {
namespace attn2 {
constexpr int QT = 64;  // queries per CTA (grid.z covers larger blocks)
}  // namespace attn2

__device__ __forceinline__ uint32_t bitpair_f16x2(uint32_t x) {
    // bits 0 and 1 of x -> fp16x2 {bit0 ? 1 : 0, bit1 ? 1 : 0}
    return ((x & 1u) | ((x & 2u) << 15)) * 0x3C00u;
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

template <int DH, int WARPS>
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
    const int MT = (B + 15) / 16;
    const int KR = WARPS / MT;

    float* e_s = (float*)sm;                                  // [DH + 1]
    uint32_t* q_s = (uint32_t*)(e_s + DH + 1 + 3);            // [MT*16][DW]
    uint4* qf_s = (uint4*)(q_s + QT * DW);                    // [MT][NKS][32] A fragments
    uint32_t* k_s = (uint32_t*)(qf_s + MT * NKS * 32);        // [L][DW]
    uint32_t* vt_s = k_s + (size_t)L * DW;                    // [DH][LW]
    // merge area (reuses k_s/vt_s after the key loop): [WARPS][16][DH] + m, l
    float* o_s = (float*)k_s;
    float* m_s = o_s + (size_t)WARPS * 16 * DH;
    float* l_s = m_s + WARPS * 16;

    for (int gg = tid; gg <= DH; gg += NTHREADS) e_s[gg] = expf(-__fmul_rn(a.alpha, (float)gg));
    for (int i = tid; i < MT * 16 * DW; i += NTHREADS) {
        const int b = i / DW, w = i % DW;
        q_s[i] = b < B ? a.q[(size_t)((q0 + b) * a.T + t) * WD + h * DW + w] : 0u;
    }
    const uint32_t* kbase = a.k + (size_t)t * a.Ls * WD + h * DW;
    const uint32_t* vbase = a.v + (size_t)t * a.Ls * WD + h * DW;
    for (int i = tid; i < L * DW; i += NTHREADS) {
        const int j = i / DW, w = i % DW;
        k_s[i] = kbase[(size_t)j * WD + w];
    }
    // V^T: bit j%32 of word vt_s[c][j/32] is v[j][c]; a warp transposes 32 keys x 32 channels
    for (int j0 = warp * 32; j0 < L; j0 += WARPS * 32) {
        const int j = j0 + lane;
        uint32_t vw[DW];
#pragma unroll
        for (int w = 0; w < DW; ++w) vw[w] = j < L ? vbase[(size_t)j * WD + w] : 0u;
#pragma unroll
        for (int w = 0; w < DW; ++w)
            vt_s[(size_t)(w * 32 + lane) * LW + (j0 >> 5)] = warp_transpose32(vw[w]);
    }
    __syncthreads();

    // Q as fp16 A fragments, once per CTA (rows mt*16 + g and + 8; channels 16 ks + 2c,
    // +1 and + 8, + 9); kept in shared memory rather than 4*NKS registers per thread.
    for (int i = tid; i < MT * NKS * 32; i += NTHREADS) {
        const int ln = i & 31, ks = (i >> 5) % NKS, mt_ = i / (NKS * 32);
        const int gg = ln >> 2, ch = 16 * ks + 2 * (ln & 3);
        const uint32_t* r0 = q_s + (mt_ * 16 + gg) * DW;
        const uint32_t* r1 = q_s + (mt_ * 16 + gg + 8) * DW;
        qf_s[i] = make_uint4(bitpair_f16x2(r0[ch >> 5] >> (ch & 31)),
                             bitpair_f16x2(r1[ch >> 5] >> (ch & 31)),
                             bitpair_f16x2(r0[(ch + 8) >> 5] >> ((ch + 8) & 31)),
                             bitpair_f16x2(r1[(ch + 8) >> 5] >> ((ch + 8) & 31)));
    }
    __syncthreads();

    const int mt = warp % MT, kr = warp / MT;
    const bool active = kr < KR;
    // key range of this warp, in blocks of 32 keys
    const int nblk = (L + 31) / 32;
    const int kb0 = active ? kr * nblk / KR : 0, kb1 = active ? (kr + 1) * nblk / KR : 0;
    const uint4* qf = qf_s + mt * NKS * 32 + lane;
    float o[NNT][4];
#pragma unroll
    for (int n = 0; n < NNT; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.0f;
    int mrow[2] = {-1, -1};      // running maximum score of rows g and g + 8 (-1: none yet)
    float lrow[2] = {0.f, 0.f};  // this thread's part of the running normaliser

    for (int kb = kb0; kb < kb1; ++kb) {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int key0 = kb * 32 + half * 16;
            // scores of 16 keys: n tile 0 = keys key0..key0+7, n tile 1 = key0+8..key0+15
            float s[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.0f;
#pragma unroll
            for (int ks = 0; ks < NKS; ++ks) {
                const uint4 qv = qf[ks * 32];
                const uint32_t qa[4] = {qv.x, qv.y, qv.z, qv.w};
                const int ch = 16 * ks + 2 * c;
#pragma unroll
                for (int nt = 0; nt < 2; ++nt) {
                    const int key = key0 + nt * 8 + g;
                    const uint32_t* kr_ = k_s + (size_t)min(key, L - 1) * DW;
                    const uint32_t b0 = key < L ? bitpair_f16x2(kr_[ch >> 5] >> (ch & 31)) : 0u;
                    const uint32_t b1 =
                        key < L ? bitpair_f16x2(kr_[(ch + 8) >> 5] >> ((ch + 8) & 31)) : 0u;
                    mma16816(s[nt], qa, b0, b1);
                }
            }
            // keys past L get no weight
            int sc[2][4];
            bool kv[2][2];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                kv[nt][0] = key0 + nt * 8 + 2 * c < L;
                kv[nt][1] = key0 + nt * 8 + 2 * c + 1 < L;
#pragma unroll
                for (int e = 0; e < 4; ++e) sc[nt][e] = (int)s[nt][e];
            }
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
                if (bm > mrow[r]) {
                    if (mrow[r] >= 0) {
                        const float f = e_s[bm - mrow[r]];
                        lrow[r] *= f;
#pragma unroll
                        for (int n = 0; n < NNT; ++n) {
                            o[n][2 * r] *= f;
                            o[n][2 * r + 1] *= f;
                        }
                    }
                    mrow[r] = bm;
                }
            }
            // P = exp(alpha (s - max)) -> fp16 A fragment of the P V product
            float p[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int r = e >> 1;
                    const bool valid = kv[nt][e & 1];
                    p[nt][e] = valid ? e_s[mrow[r] - sc[nt][e]] : 0.0f;
                    lrow[r] += p[nt][e];
                }
            // P = P_hi + P_lo, both fp16: the two products give P V to ~2^-22 relative
            uint32_t ph[4], pl[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float x0 = p[q >> 1][2 * (q & 1)], x1 = p[q >> 1][2 * (q & 1) + 1];
                const __half2 hi = __floats2half2_rn(x0, x1);
                const float2 hf = __half22float2(hi);
                ph[q] = *reinterpret_cast<const uint32_t*>(&hi);
                pl[q] = pack_f16x2(x0 - hf.x, x1 - hf.y);
            }
            // O += P V: B fragment of n tile nt = keys (2c, 2c+1 | 2c+8, 2c+9) at channel 8 nt + g
            const int sh = half * 16 + 2 * c;
#pragma unroll
            for (int n = 0; n < NNT; ++n) {
                const uint32_t vw = vt_s[(size_t)(8 * n + g) * LW + kb];
                const uint32_t b0 = bitpair_f16x2(vw >> sh), b1 = bitpair_f16x2(vw >> (sh + 8));
                mma16816(o[n], ph, b0, b1);
                mma16816(o[n], pl, b0, b1);
            }
        }
    }
    // normaliser of each row summed over the 4 lanes of its group
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
        lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
    }
    __syncthreads();  // k_s / vt_s are reused as the merge area
    if (active) {
        float* ow = o_s + (size_t)warp * 16 * DH;
#pragma unroll
        for (int n = 0; n < NNT; ++n) {
            const int ch = 8 * n + 2 * c;
            ow[g * DH + ch] = o[n][0];
            ow[g * DH + ch + 1] = o[n][1];
            ow[(g + 8) * DH + ch] = o[n][2];
            ow[(g + 8) * DH + ch + 1] = o[n][3];
        }
        if (c == 0) {
            m_s[warp * 16 + g] = (float)mrow[0];
            m_s[warp * 16 + g + 8] = (float)mrow[1];
            l_s[warp * 16 + g] = lrow[0];
            l_s[warp * 16 + g + 8] = lrow[1];
        }
    }
    __syncthreads();
    // merge the key ranges of each query row and write the currents
    const int D = a.H * DH;
    for (int i = tid; i < B * DH; i += NTHREADS) {
        const int b = i / DH, ch = i % DH;
        const int tile = b / 16, row = b % 16;
        int mstar = -1;
        for (int k2 = 0; k2 < KR; ++k2) mstar = max(mstar, (int)m_s[(k2 * MT + tile) * 16 + row]);
        float num = 0.0f, den = 0.0f;
        for (int k2 = 0; k2 < KR; ++k2) {
            const int w = k2 * MT + tile;
            const int mw = (int)m_s[w * 16 + row];
            if (mw < 0) continue;  // this range held no key
            const float f = e_s[mstar - mw];
            num += o_s[((size_t)w * 16 + row) * DH + ch] * f;
            den += l_s[w * 16 + row] * f;
        }
        a.out[(size_t)((q0 + b) * a.T + t) * D + h * DH + ch] = __fdiv_rn(num, den);
    }
}

size_t attention_mma_smem_bytes(int B, int L, int dh, int warps) {
    const int DW = dh / 32, LW = (L + 31) / 32, MT = (B + 15) / 16;
    const size_t head = 4 * (size_t)(dh + 4) + 4 * (size_t)attn2::QT * DW +
                        16 * (size_t)MT * (dh / 16) * 32;
    const size_t kv = 4 * (size_t)L * DW + 4 * (size_t)dh * LW;
    const size_t merge = 4 * (size_t)warps * 16 * dh + 8 * (size_t)warps * 16;
    return head + std::max(kv, merge) + 64;
}

template <int DH, int WARPS>
static nmdlm_status launch_attention_mma_t(const AttnArgs& a, cudaStream_t stream) {
    const size_t smem = attention_mma_smem_bytes(std::min(a.B, attn2::QT), a.L, DH, WARPS);
    if (smem > 220 * 1024) return launch_attention(nullptr, a, stream);
    static size_t configured = 0;
    if (smem > configured) {
        if (cuda_status(cudaFuncSetAttribute(k_attention_mma<DH, WARPS>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem)) != NMDLM_OK)
            return NMDLM_ERR_CUDA;
        configured = smem;
    }
    dim3 grid(a.H, a.T, (a.B + attn2::QT - 1) / attn2::QT);
    const cudaError_t le = launch_pdl(k_attention_mma<DH, WARPS>, dim3(grid), dim3(WARPS * 32),
                                      smem, stream, 1, a);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

// Tensor-core attention when the head width and block size allow, else CUDA cores.
nmdlm_status launch_attention_best(const AttnArgs& a, cudaStream_t stream) {
    if (a.B < 1 || a.L < 1) return launch_attention(nullptr, a, stream);
    static int sweep = getenv("NMDLM_ATTN_WARPS") ? atoi(getenv("NMDLM_ATTN_WARPS")) : 0;
    switch (a.dh) {
        case 32: return launch_attention_mma_t<32, 16>(a, stream);
        case 64: return launch_attention_mma_t<64, 16>(a, stream);
        case 96: return launch_attention_mma_t<96, 16>(a, stream);
        case 128:
            if (sweep == 8) return launch_attention_mma_t<128, 8>(a, stream);
            if (sweep == 16) return launch_attention_mma_t<128, 16>(a, stream);
            return launch_attention_mma_t<128, 12>(a, stream);
        default: return launch_attention(nullptr, a, stream);
    }
}

}  // namespace nmdlm
