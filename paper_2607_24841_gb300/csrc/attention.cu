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
#include "internal.h"

namespace nmdlm {

namespace attn {
constexpr int NTHREADS = 512;
constexpr int KCH = 256;  // keys per mixture chunk
}  // namespace attn

// grid (H, T); one CTA owns every query of the block for one (timestep, head).
__global__ void __launch_bounds__(attn::NTHREADS) k_attention(AttnArgs a) {
    using namespace attn;
    extern __shared__ __align__(16) uint8_t sm[];
    const int h = blockIdx.x, t = blockIdx.y;
    const int B = a.B, L = a.L, dh = a.dh, DW = dh >> 5;
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
        q_s[i] = a.q[(size_t)(b * a.T + t) * WD + h * DW + w];
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
        for (int w = 0; w < 8; ++w) {
            if (w < DW) {
                for (int bit = 0; bit < 32; ++bit) {
                    const uint32_t word = __ballot_sync(0xffffffffu, (vw[w] >> bit) & 1u);
                    if (lane == 0) vt_s[(size_t)(w * 32 + bit) * LW + (j0 >> 5)] = word;
                }
            }
        }
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
                    a.out[(size_t)(qb * a.T + t) * D + h * dh + c] = __fdiv_rn(acc[i], z_s[qb]);
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
    if (a.B > 64 || a.B < 1 || a.L < 1) return NMDLM_ERR_UNSUPPORTED;
    const size_t smem = attention_smem_bytes(a.B, a.L, a.dh);
    if (smem > 220 * 1024) return NMDLM_ERR_UNSUPPORTED;
    static size_t configured = 0;
    if (smem > configured) {
        if (cuda_status(cudaFuncSetAttribute(
                k_attention, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != NMDLM_OK)
            return NMDLM_ERR_CUDA;
        configured = smem;
    }
    dim3 grid(a.H, a.T);
    k_attention<<<grid, attn::NTHREADS, smem, stream>>>(a);
    count_launch();
    return cuda_status(cudaGetLastError());
}

}  // namespace nmdlm
