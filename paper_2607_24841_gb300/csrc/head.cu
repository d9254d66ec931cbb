// head.cu -- confidence of each masked position and greedy unmasking.
//
// Sec. III-A: at each denoising step B/S still-masked positions are unmasked; the
// paper defers the selection rule to block diffusion.  Reading: confidence = largest
// softmax probability of the position's logits (computed in fp64, the same precision
// as the reference definition, so that near-ties rank identically), token = argmax
// (lowest id on ties); the B/S most confident masked positions are fixed, ties going
// to the lowest position.  Unmasked tokens never change.
#include <cmath>

#include "internal.h"

namespace nmdlm {

// One CTA per position: argmax of the fp32 logits, then Z = sum exp(l - max) in fp64.
__global__ void k_head_stats(const float* logits, int V, double* conf, int* tok) {
    const int b = blockIdx.x, tid = threadIdx.x;
    const float* l = logits + (size_t)b * V;
    float best = -INFINITY;
    int arg = 0x7fffffff;
    for (int v = tid; v < V; v += blockDim.x) {
        const float x = l[v];
        if (x > best || (x == best && v < arg)) {
            best = x;
            arg = v;
        }
    }
    __shared__ float sb[32];
    __shared__ int sa[32];
    __shared__ double sz[32];
    const int lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    for (int o = 16; o > 0; o >>= 1) {
        const float x = __shfl_xor_sync(0xffffffffu, best, o);
        const int y = __shfl_xor_sync(0xffffffffu, arg, o);
        if (x > best || (x == best && y < arg)) {
            best = x;
            arg = y;
        }
    }
    if (lane == 0) {
        sb[warp] = best;
        sa[warp] = arg;
    }
    __syncthreads();
    if (tid == 0) {
        for (int w = 1; w < nw; ++w)
            if (sb[w] > sb[0] || (sb[w] == sb[0] && sa[w] < sa[0])) {
                sb[0] = sb[w];
                sa[0] = sa[w];
            }
    }
    __syncthreads();
    const double mx = (double)sb[0];
    double z = 0.0;
    for (int v = tid; v < V; v += blockDim.x) z += exp((double)l[v] - mx);
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if (lane == 0) sz[warp] = z;
    __syncthreads();
    if (tid == 0) {
        double zt = 0.0;
        for (int w = 0; w < nw; ++w) zt += sz[w];
        conf[b] = 1.0 / zt;
        tok[b] = sa[0];
    }
}

// One CTA: k rounds of "most confident masked position" (ties -> lowest position).
__global__ void k_unmask(const double* conf, const int* tok, int B, int k, int* tokens,
                         int* mask, int* unmasked_out) {
    __shared__ int taken[1024];
    __shared__ double bc[32];
    __shared__ int bp[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    for (int b = tid; b < B; b += blockDim.x) taken[b] = 0;
    __syncthreads();
    for (int r = 0; r < k; ++r) {
        double best = -1.0;
        int pos = 0x7fffffff;
        for (int b = tid; b < B; b += blockDim.x) {
            if (mask[b] && !taken[b]) {
                const double c = conf[b];
                if (c > best || (c == best && b < pos)) {
                    best = c;
                    pos = b;
                }
            }
        }
        for (int o = 16; o > 0; o >>= 1) {
            const double c = __shfl_xor_sync(0xffffffffu, best, o);
            const int p = __shfl_xor_sync(0xffffffffu, pos, o);
            if (c > best || (c == best && p < pos)) {
                best = c;
                pos = p;
            }
        }
        if (lane == 0) {
            bc[warp] = best;
            bp[warp] = pos;
        }
        __syncthreads();
        if (tid == 0) {
            double c0 = bc[0];
            int p0 = bp[0];
            for (int w = 1; w < nw; ++w)
                if (bc[w] > c0 || (bc[w] == c0 && bp[w] < p0)) {
                    c0 = bc[w];
                    p0 = bp[w];
                }
            if (p0 != 0x7fffffff) {
                taken[p0] = 1;
                tokens[p0] = tok[p0];
                if (unmasked_out) unmasked_out[r] = p0;
            } else if (unmasked_out) {
                unmasked_out[r] = -1;
            }
        }
        __syncthreads();
    }
    for (int b = tid; b < B; b += blockDim.x)
        if (taken[b]) mask[b] = 0;
}

__global__ void k_fill_i32(int* p, int n, int v) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) p[i] = v;
}

nmdlm_status launch_head_unmask(nmdlm_ctx*, const float* logits, int B, int V, int k,
                                int32_t* tokens, int32_t* mask, int32_t* unmasked_out,
                                WsCursor& ws, cudaStream_t stream) {
    if (B > 1024) return NMDLM_ERR_UNSUPPORTED;
    double* conf = ws.take<double>(B);
    int* tok = ws.take<int>(B);
    if (!conf || !tok) return NMDLM_ERR_WORKSPACE;
    k_head_stats<<<B, 512, 0, stream>>>(logits, V, conf, tok);
    count_launch();
    if (cuda_status(cudaGetLastError()) != NMDLM_OK) return NMDLM_ERR_CUDA;
    k_unmask<<<1, 256, 0, stream>>>(conf, tok, B, k, tokens, mask, unmasked_out);
    count_launch();
    return cuda_status(cudaGetLastError());
}

nmdlm_status launch_fill_i32(int* p, int n, int v, cudaStream_t stream) {
    k_fill_i32<<<(n + 255) / 256, 256, 0, stream>>>(p, n, v);
    count_launch();
    return cuda_status(cudaGetLastError());
}

// Fault-injection check: wait on a barrier that nothing ever completes.  The bounded
// wait runs out, records a timeout and the kernel returns.
__global__ void k_wait_test(int* err, unsigned long long ns) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) mbar_init(&bar, 1);
    __syncthreads();
    if (threadIdx.x == 0) {
        if (!mbar_wait_bounded(&bar, 0, ns)) raise_error(err, ERRBIT_TIMEOUT);
    }
}

nmdlm_status launch_wait_test(nmdlm_ctx* ctx, unsigned long long ns, cudaStream_t stream) {
    k_wait_test<<<1, 32, 0, stream>>>(ctx->err, ns);
    count_launch();
    return cuda_status(cudaGetLastError());
}

}  // namespace nmdlm
