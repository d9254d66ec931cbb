// spikes.cu -- spike packing, active-channel compaction and IF encoding.
//
// Packing produces the three forms the other kernels read (row bits for attention,
// column masks + active mask for the spiking linears).  Compaction lists the active
// channels in ascending order (Sec. IV-A, assumption (ii)).  The IF kernel is the
// neuron of Sec. II-B, Eq. (3)-(4), read charge-then-fire, fed either by a dense
// current tensor or by the token + position embedding of the block (Sec. III-A).
#include "internal.h"

namespace nmdlm {

// grid.x = groups of 32 channels; block (32, 8).  Lane = channel, ty = row slot.
template <int MAXW>
__global__ void k_pack(const uint8_t* spikes, int BT, int D, uint32_t* row_bits,
                       uint32_t* col_masks, uint32_t* active_mask, int* err) {
    pdl_wait();
    const int lane = threadIdx.x, ty = threadIdx.y, BY = blockDim.y;
    const int d = blockIdx.x * 32 + lane;
    const bool valid = d < D;
    const int DW = words_of(D), BTW = words_of(BT);
    __shared__ uint32_t cm_s[32][MAXW];
    __shared__ int any_s[32];
    for (int i = ty * 32 + lane; i < 32 * MAXW; i += 32 * BY) cm_s[i / MAXW][i % MAXW] = 0;
    if (ty == 0) any_s[lane] = 0;
    __syncthreads();
    uint32_t cmw[MAXW];
#pragma unroll
    for (int w = 0; w < MAXW; ++w) cmw[w] = 0;
    bool any = false, bad = false;
    for (int bt = ty; bt < BT; bt += BY) {
        const uint8_t v = valid ? spikes[(size_t)bt * D + d] : 0;
        if (v > 1) bad = true;
        const bool sp = v != 0;
        const uint32_t word = __ballot_sync(0xffffffffu, sp);
        if (lane == 0) row_bits[(size_t)bt * DW + blockIdx.x] = word;
        if (sp) {
#pragma unroll
            for (int w = 0; w < MAXW; ++w)
                if (w == (bt >> 5)) cmw[w] |= 1u << (bt & 31);
            any = true;
        }
    }
    if (bad) raise_error(err, ERRBIT_VALUE);
#pragma unroll
    for (int w = 0; w < MAXW; ++w)
        if (cmw[w]) atomicOr(&cm_s[lane][w], cmw[w]);
    if (any) any_s[lane] = 1;
    __syncthreads();
    if (ty == 0) {
        if (valid && col_masks)
            for (int w = 0; w < BTW; ++w) col_masks[(size_t)d * BTW + w] = cm_s[lane][w];
        const uint32_t mw = __ballot_sync(0xffffffffu, valid && any_s[lane]);
        if (lane == 0 && active_mask) active_mask[blockIdx.x] = mw;
    }
}

// One CTA: ascending list of the set bits of `mask` (D bits) and their count.
__global__ void k_compact(const uint32_t* mask, int D, int32_t* idx, int32_t* n_active) {
    pdl_wait();
    const int DW = words_of(D);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ int warp_tot[32];
    __shared__ int carry;
    if (tid == 0) carry = 0;
    __syncthreads();
    for (int base = 0; base < DW; base += blockDim.x) {
        const int w = base + tid;
        uint32_t m = w < DW ? mask[w] : 0u;
        if (w == DW - 1 && (D & 31)) m &= (1u << (D & 31)) - 1u;
        const int cnt = __popc(m);
        int x = cnt;
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
            if (lane < nw) warp_tot[lane] = y;
        }
        __syncthreads();
        int pos = carry + x - cnt + (warp > 0 ? warp_tot[warp - 1] : 0);
        while (m) {
            const int bit = __ffs(m) - 1;
            m &= m - 1;
            if (idx) idx[pos] = w * 32 + bit;
            ++pos;
        }
        __syncthreads();
        if (tid == blockDim.x - 1) carry = pos;
        __syncthreads();
    }
    if (tid == 0 && n_active) *n_active = carry;
}

// IF encode.  grid.x = groups of 32 neurons; block (32, BY): lane = neuron n,
// ty = token slot (b = ty, ty + BY, ...).  Each thread runs the T steps of its
// (token, neuron) pairs sequentially.
template <int MAXW>
__global__ void k_if(IfArgs a) {
    pdl_wait();
    const int lane = threadIdx.x, ty = threadIdx.y, BY = blockDim.y;
    const int n = blockIdx.x * 32 + lane;
    const bool valid = n < a.N;
    const int T = a.T, NW = words_of(a.N), BTW = words_of(a.B * a.T);
    __shared__ uint32_t cm_s[32][MAXW];
    __shared__ int any_s[32];
    for (int i = ty * 32 + lane; i < 32 * MAXW; i += 32 * BY) cm_s[i / MAXW][i % MAXW] = 0;
    if (ty == 0) any_s[lane] = 0;
    __syncthreads();
    bool any = false;
    for (int b = ty; b < a.B; b += BY) {
        uint32_t tb = 0;  // bit t: spike of (b, t) for this neuron
        float emb = 0.0f;
        if (a.src_kind == 2) {
            int tok = a.tokens[b];
            if (tok < 0 || tok > a.vocab) {
                if (lane == 0) raise_error(a.err, ERRBIT_VALUE);
                tok = a.vocab;
            }
            if (valid)
                emb = __fadd_rn(a.tok_emb[(size_t)tok * a.N + n],
                                a.pos_emb[(size_t)(a.pos0 + b) * a.N + n]);
        }
        float vf = 0.0f;
        int vi = 0;
        if (a.v_state && valid) {
            if (a.src_kind == 1) vi = ((const int*)a.v_state)[(size_t)b * a.N + n];
            else vf = ((const float*)a.v_state)[(size_t)b * a.N + n];
        }
        // steps in groups of 4 whose currents are loaded before the recurrence runs
        // over them (one memory latency per group, not per step)
        for (int t0 = 0; t0 < T; t0 += 4) {
            int ci[4];
            float cf[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const size_t off = (size_t)(b * T + t0 + u) * a.N + n;
                const bool ld = valid && t0 + u < T;
                ci[u] = (a.src_kind == 1 && ld) ? a.cur_i[off] : 0;
                cf[u] = a.src_kind == 2 ? emb : ((a.src_kind == 0 && ld) ? a.cur_f[off] : 0.0f);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int t = t0 + u;
                if (t >= T) break;
                const int bt = b * T + t;
                const size_t off = (size_t)bt * a.N + n;
                bool sp = false;
                if (a.src_kind == 1) {
                    const int h = vi + ci[u];
                    sp = valid && h >= a.theta_i;
                    vi = sp ? h - a.theta_i : h;
                } else {
                    const float I = cf[u];
                    if (a.cur_out && valid) a.cur_out[off] = I;
                    const float h = __fadd_rn(vf, I);
                    sp = valid && h >= a.theta_f;
                    vf = sp ? __fsub_rn(h, a.theta_f) : h;
                }
                const uint32_t word = __ballot_sync(0xffffffffu, sp);
                if (lane == 0) a.bits[(size_t)bt * NW + blockIdx.x] = word;
                tb |= (sp ? 1u : 0u) << t;
            }
        }
        if (tb) {  // the token's T column-mask bits start at bit b * T
            const int start = b * T, w0 = start >> 5, sh = start & 31;
            atomicOr(&cm_s[lane][w0], tb << sh);
            if (sh + T > 32) atomicOr(&cm_s[lane][w0 + 1], tb >> (32 - sh));
            any = true;
        }
        if (a.v_state && valid) {
            if (a.src_kind == 1) ((int*)a.v_state)[(size_t)b * a.N + n] = vi;
            else ((float*)a.v_state)[(size_t)b * a.N + n] = vf;
        }
    }
    if (any) any_s[lane] = 1;
    __syncthreads();
    if (ty == 0) {
        if (valid && a.cm)
            for (int w = 0; w < BTW; ++w) a.cm[(size_t)n * BTW + w] = cm_s[lane][w];
        const uint32_t mw = __ballot_sync(0xffffffffu, valid && any_s[lane]);
        if (lane == 0 && a.mask) a.mask[blockIdx.x] = mw;
    }
}

nmdlm_status launch_pack(nmdlm_ctx* ctx, const uint8_t* spikes, int BT, int D,
                         uint32_t* row_bits, uint32_t* col_masks, uint32_t* active_mask,
                         int32_t* active_idx, int32_t* n_active, cudaStream_t stream) {
    dim3 block(32, 8);
    const cudaError_t le = launch_pdl(k_pack<8>, dim3(words_of(D)), dim3(block), 0, stream, 1,
                                      spikes, BT, D, row_bits, col_masks, active_mask, ctx->err);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    if (cuda_status(cudaGetLastError()) != NMDLM_OK) return NMDLM_ERR_CUDA;
    if (active_idx || n_active) {
        if (!active_mask) return NMDLM_ERR_INVALID_ARG;
        return launch_compact(ctx, active_mask, D, active_idx, n_active, stream);
    }
    return NMDLM_OK;
}

nmdlm_status launch_compact(nmdlm_ctx*, const uint32_t* mask, int D, int32_t* idx,
                            int32_t* n_active, cudaStream_t stream) {
    const cudaError_t le = launch_pdl(k_compact, dim3(1), dim3(1024), 0, stream, 1, mask, D, idx,
                                      n_active);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

nmdlm_status launch_if(nmdlm_ctx*, const IfArgs& a, cudaStream_t stream) {
    // one token per warp row up to 32 tokens, so that every token's loads are in flight
    const int BY = a.B < 32 ? a.B : 32;
    dim3 block(32, BY > 0 ? BY : 1);
    const cudaError_t le = launch_pdl(k_if<8>, dim3(words_of(a.N)), dim3(block), 0, stream, 1, a);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

}  // namespace nmdlm
