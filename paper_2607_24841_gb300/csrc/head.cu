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

// Statistics of one position's logits, split over HS CTAs per position so the fp64
// exponentials (slow on this GPU) use every SM.  CTA (b, s) takes the slice
// [s V / HS, (s+1) V / HS): its argmax (lowest id on ties) and z_s = sum exp(l - m_s)
// in fp64 around its own maximum m_s.  The last CTA of position b to finish (arrival
// counter, reset by that CTA) combines: M = max m_s, Z = sum z_s exp(m_s - M),
// confidence = 1 / Z, token = argmax over the slices (lowest slice on ties, hence
// lowest id).
constexpr int HEAD_SPLITS = 8;

__device__ __forceinline__ void argmax_merge(float& best, int& arg, float x, int y) {
    if (x > best || (x == best && y < arg)) {
        best = x;
        arg = y;
    }
}

__global__ void k_head_stats(const float* logits, int V, double* conf, int* tok, float* part_m,
                             int* part_a, double* part_z, unsigned int* counters) {
    pdl_wait();
    const int b = blockIdx.x, sl = blockIdx.y, tid = threadIdx.x;
    const int v0 = (int)((long long)sl * V / HEAD_SPLITS);
    const int v1 = (int)((long long)(sl + 1) * V / HEAD_SPLITS);
    const float* l = logits + (size_t)b * V;
    float best = -INFINITY;
    int arg = 0x7fffffff;
    for (int v = v0 + tid; v < v1; v += blockDim.x) argmax_merge(best, arg, l[v], v);
    __shared__ float sb[32];
    __shared__ int sa[32];
    __shared__ double sz[32];
    __shared__ int last;
    const int lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    for (int o = 16; o > 0; o >>= 1)
        argmax_merge(best, arg, __shfl_xor_sync(0xffffffffu, best, o),
                     __shfl_xor_sync(0xffffffffu, arg, o));
    if (lane == 0) {
        sb[warp] = best;
        sa[warp] = arg;
    }
    __syncthreads();
    if (tid == 0)
        for (int w = 1; w < nw; ++w) argmax_merge(sb[0], sa[0], sb[w], sa[w]);
    __syncthreads();
    const double mx = (double)sb[0];
    double z = 0.0;
    for (int v = v0 + tid; v < v1; v += blockDim.x) z += exp((double)l[v] - mx);
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if (lane == 0) sz[warp] = z;
    __syncthreads();
    if (tid == 0) {
        double zt = 0.0;
        for (int w = 0; w < nw; ++w) zt += sz[w];
        part_m[b * HEAD_SPLITS + sl] = sb[0];
        part_a[b * HEAD_SPLITS + sl] = sa[0];
        part_z[b * HEAD_SPLITS + sl] = zt;
        __threadfence();
        last = atomicAdd(&counters[b], 1u) == HEAD_SPLITS - 1;
    }
    __syncthreads();
    if (last && tid == 0) {
        __threadfence();
        const volatile float* pm = part_m + b * HEAD_SPLITS;
        const volatile int* pa = part_a + b * HEAD_SPLITS;
        const volatile double* pz = part_z + b * HEAD_SPLITS;
        float m = pm[0];
        int a = pa[0];
        for (int s = 1; s < HEAD_SPLITS; ++s) argmax_merge(m, a, pm[s], pa[s]);
        double zt = 0.0;
        for (int s = 0; s < HEAD_SPLITS; ++s)
            if (pz[s] > 0.0) zt += pz[s] * exp((double)pm[s] - (double)m);
        conf[b] = 1.0 / zt;
        tok[b] = a;
        counters[b] = 0u;
    }
}

// One CTA: k rounds of "most confident masked position" (ties -> lowest position).
__global__ void k_unmask(const double* conf, const int* tok, int B, int k, int* tokens,
                         int* mask, int* unmasked_out) {
    pdl_wait();
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
    pdl_wait();
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) p[i] = v;
}

nmdlm_status launch_head_unmask(nmdlm_ctx* ctx, const float* logits, int B, int V, int k,
                                int32_t* tokens, int32_t* mask, int32_t* unmasked_out,
                                WsCursor& ws, cudaStream_t stream) {
    if (B > 1024) return NMDLM_ERR_UNSUPPORTED;
    double* conf = ws.take<double>(B);
    int* tok = ws.take<int>(B);
    double* part_z = ws.take<double>((size_t)B * HEAD_SPLITS);
    float* part_m = ws.take<float>((size_t)B * HEAD_SPLITS);
    int* part_a = ws.take<int>((size_t)B * HEAD_SPLITS);
    if (!conf || !tok || !part_z || !part_m || !part_a) return NMDLM_ERR_WORKSPACE;
    if (!ctx->counters || ctx->n_counters < (size_t)B) return NMDLM_ERR_WORKSPACE;
    const cudaError_t le = launch_pdl(k_head_stats, dim3(B, HEAD_SPLITS), dim3(256), 0, stream,
                                      1, logits, V, conf, tok, part_m, part_a, part_z,
                                      ctx->counters);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    if (cuda_status(cudaGetLastError()) != NMDLM_OK) return NMDLM_ERR_CUDA;
    const cudaError_t le2 = launch_pdl(k_unmask, dim3(1), dim3(256), 0, stream, 1, conf, tok, B,
                                       k, tokens, mask, unmasked_out);
    count_launch();
    if (le2 != cudaSuccess) return cuda_status(le2);
    return cuda_status(cudaGetLastError());
}

nmdlm_status launch_fill_i32(int* p, int n, int v, cudaStream_t stream) {
    const cudaError_t le = launch_pdl(k_fill_i32, dim3((n + 255) / 256), dim3(256), 0, stream, 1,
                                      p, n, v);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

// Fault-injection check: wait on a barrier that nothing ever completes.  The bounded
// wait runs out, records a timeout and the kernel returns.
__global__ void k_wait_test(int* err, unsigned long long ns) {
    pdl_wait();
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) mbar_init(&bar, 1);
    __syncthreads();
    if (threadIdx.x == 0) {
        if (!mbar_wait_bounded(&bar, 0, ns)) raise_error(err, ERRBIT_TIMEOUT);
    }
}

nmdlm_status launch_wait_test(nmdlm_ctx* ctx, unsigned long long ns, cudaStream_t stream) {
    const cudaError_t le = launch_pdl(k_wait_test, dim3(1), dim3(32), 0, stream, 1, ctx->err, ns);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

}  // namespace nmdlm
