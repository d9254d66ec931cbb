// ternary.cu -- bitwise ternary coding (Sec. II-C, Conversion) on the GPU.
//
// Eq. (7): each activation vector a (one row of D values) is quantised with the
// adaptive step V_th(a) = mean|a| / K, ahat = round(a / V_th).  Eq. (8): ahat is
// written over T timesteps as ternary spikes, ahat_i = sum_t 2^{t-1} s_{i,t}.  The
// library runs the linear on ternary spikes as two binary planes (the +1 spikes and
// the -1 spikes) through the spiking linear, I_t = W^T s+_t - W^T s-_t, and combines
// the planes' integer sums with the 2^{t-1} weights: y = sum_t 2^{t-1} I_t, which
// by Eq. (8) equals W^T ahat exactly.
//
// Precision, shared with the CPU restatement so that both take every quantisation
// decision identically: |a| summed in fp64 (per row, in a block reduction), V_th =
// (mean / K) rounded once to fp32, one IEEE fp32 division a / V_th, round() with
// halves away from zero, |ahat| clamped to 2^T - 1; a row whose V_th is not positive
// (all zeros, or NaN) quantises to 0, and so does a NaN value.
#include "internal.h"

namespace nmdlm {

// One block per row n; 256 threads stride over the row's D values.
__global__ void __launch_bounds__(256) k_ternary_encode(const float* a, int D, float K, int T,
                                                        uint8_t* plus, uint8_t* minus,
                                                        int32_t* ahat, float* vth) {
    pdl_wait();
    const int n = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float* row = a + (size_t)n * D;
    double sum = 0.0;
    for (int i = tid; i < D; i += blockDim.x) sum += fabs((double)__ldg(row + i));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    __shared__ double part[8];
    __shared__ float v_s;
    if (lane == 0) part[warp] = sum;
    __syncthreads();
    if (tid == 0) {
        double tot = 0.0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += part[w];
        const double mean = tot / (double)D;
        v_s = (float)(mean / (double)K);
        if (vth) vth[n] = v_s;
    }
    __syncthreads();
    const float v = v_s;
    const int cap = (1 << T) - 1;
    for (int i = tid; i < D; i += blockDim.x) {
        int q = 0;
        if (v > 0.0f) {
            const float x = __fdiv_rn(__ldg(row + i), v);
            if (x == x) {
                const float r = roundf(x);  // halves away from zero
                q = r >= (float)cap ? cap : (r <= -(float)cap ? -cap : (int)r);
            }
        }
        if (ahat) ahat[(size_t)n * D + i] = q;
        const int mag = q < 0 ? -q : q;
        // plane t of row n is spike row n*T + t of the two binary blocks
        for (int t = 0; t < T; ++t) {
            const uint8_t b = (uint8_t)((mag >> t) & 1);
            const size_t at = ((size_t)n * T + t) * D + i;
            plus[at] = q > 0 ? b : (uint8_t)0;
            minus[at] = q < 0 ? b : (uint8_t)0;
        }
    }
}

// y[n][o] = sum_t 2^t (acc+[n*T + t][o] - acc-[n*T + t][o]); one thread per (n, o),
// consecutive threads on consecutive o.
__global__ void __launch_bounds__(256) k_ternary_combine(const int32_t* accp, const int32_t* accm,
                                                         int N, int T, int d_out, int32_t* y) {
    pdl_wait();
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)N * d_out) return;
    const int n = (int)(idx / d_out), o = (int)(idx % d_out);
    long long s = 0;
    for (int t = 0; t < T; ++t) {
        const size_t at = ((size_t)n * T + t) * d_out + o;
        s += (long long)(__ldg(accp + at) - __ldg(accm + at)) * (1ll << t);
    }
    y[idx] = (int32_t)s;
}

nmdlm_status launch_ternary_encode(const float* a, int N, int D, float K, int T, uint8_t* plus,
                                   uint8_t* minus, int32_t* ahat, float* vth,
                                   cudaStream_t stream) {
    const cudaError_t le = launch_pdl(k_ternary_encode, dim3(N), dim3(256), 0, stream, 1, a, D,
                                      K, T, plus, minus, ahat, vth);
    count_launch();
    return cuda_status(le);
}

nmdlm_status launch_ternary_combine(const int32_t* accp, const int32_t* accm, int N, int T,
                                    int d_out, int32_t* y, cudaStream_t stream) {
    const long long total = (long long)N * d_out;
    const cudaError_t le = launch_pdl(k_ternary_combine, dim3((unsigned)((total + 255) / 256)),
                                      dim3(256), 0, stream, 1, accp, accm, N, T, d_out, y);
    count_launch();
    return cuda_status(le);
}

}  // namespace nmdlm
