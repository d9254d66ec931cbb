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
// decision identically: the sum of |a| over the row is exact (an integer number of
// 2^-149 units held in 32-bit limbs, so no order of summation can change it) and is
// rounded once to fp64 (nearest, ties to even); mean = sum / D and V_th = (mean / K)
// in fp64, rounded once to fp32; one IEEE fp32 division a / V_th, round() with halves
// away from zero, |ahat| clamped to 2^T - 1; a row whose V_th is not positive (all
// zeros, or NaN) quantises to 0, and so does a NaN value.
#include "internal.h"

namespace nmdlm {

// |x| of a finite fp32 value is m * 2^sh * 2^-149 with m < 2^24 and 0 <= sh <= 253:
// add it to the limbs (limb k holds bits [32k, 32k + 32) of the running integer, with
// room above bit 32 so that carries wait until the end).  NaN / Inf only set flags.
constexpr int kAbsLimbs = 10;
__device__ __forceinline__ void abs_limbs_add(uint64_t (&l)[kAbsLimbs], int& nan, int& inf,
                                              float x) {
    const uint32_t b = __float_as_uint(x) & 0x7fffffffu;
    const uint32_t ex = b >> 23, man = b & 0x7fffffu;
    if (ex == 255u) {
        nan |= man != 0u;
        inf |= man == 0u;
        return;
    }
    const uint64_t m = ex ? (uint64_t)(man | 0x800000u) : (uint64_t)man;
    const int sh = ex ? (int)ex - 1 : 0;
    const int j = sh >> 5;
    const uint64_t part = m << (sh & 31);  // < 2^55
    const uint64_t lo = part & 0xffffffffull, hi = part >> 32;
#pragma unroll
    for (int k = 0; k < kAbsLimbs; ++k) {
        l[k] += k == j ? lo : 0ull;
        l[k] += k == j + 1 ? hi : 0ull;
    }
}

// The limbs' integer (carries propagated) times 2^-149, rounded to the nearest double
// (ties to even): a 96-bit window from the top non-zero limb holds the 53 kept bits and
// the rounding bits; lower limbs only decide a tie.
__device__ double abs_limbs_to_double(uint64_t (&l)[kAbsLimbs]) {
#pragma unroll
    for (int k = 0; k + 1 < kAbsLimbs; ++k) {
        l[k + 1] += l[k] >> 32;
        l[k] &= 0xffffffffull;
    }
    int J = kAbsLimbs - 1;
    while (J >= 0 && l[J] == 0ull) --J;
    if (J < 0) return 0.0;
    unsigned __int128 w = (unsigned __int128)l[J] << 64;
    if (J >= 1) w |= (unsigned __int128)l[J - 1] << 32;
    if (J >= 2) w |= (unsigned __int128)l[J - 2];
    bool below = false;
    for (int k = 0; k < J - 2; ++k) below |= l[k] != 0ull;
    const int top = 64 + 63 - __clzll((long long)l[J]);  // l[J] < 2^32: top in [64, 95]
    const int drop = top - 52;                              // >= 12 bits below the kept 53
    unsigned long long mant = (unsigned long long)(w >> drop);
    const unsigned __int128 rest = w & ((((unsigned __int128)1) << drop) - 1);
    const unsigned __int128 half = ((unsigned __int128)1) << (drop - 1);
    if (rest > half || (rest == half && (below || (mant & 1ull)))) mant += 1ull;
    return ldexp((double)mant, 32 * (J - 2) + drop - 149);
}

// One block per row n; 256 threads stride over the row's D values.  Plane t of row n is
// spike row n * rs + t of the plus and of the minus block (rs = T: two blocks of N*T
// rows; rs = 2T with minus = plus + T rows: one block of the interleaved planes).
__global__ void __launch_bounds__(256) k_ternary_encode(const float* a, int D, float K, int T,
                                                        int rs, uint8_t* plus, uint8_t* minus,
                                                        int32_t* ahat, float* vth) {
    pdl_wait();
    const int n = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float* row = a + (size_t)n * D;
    uint64_t l[kAbsLimbs];
#pragma unroll
    for (int k = 0; k < kAbsLimbs; ++k) l[k] = 0ull;
    int nan = 0, inf = 0;
    for (int i = tid; i < D; i += blockDim.x) abs_limbs_add(l, nan, inf, __ldg(row + i));
    // integer sums of the limbs over the block (exact in any order: D < 2^31 terms of
    // less than 2^32 each per limb)
#pragma unroll
    for (int k = 0; k < kAbsLimbs; ++k)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) l[k] += __shfl_xor_sync(0xffffffffu, l[k], o);
    nan = __any_sync(0xffffffffu, nan);
    inf = __any_sync(0xffffffffu, inf);
    __shared__ uint64_t part[8][kAbsLimbs];
    __shared__ int flags[8];
    __shared__ float v_s;
    if (lane == 0) {
#pragma unroll
        for (int k = 0; k < kAbsLimbs; ++k) part[warp][k] = l[k];
        flags[warp] = (nan ? 1 : 0) | (inf ? 2 : 0);
    }
    __syncthreads();
    if (tid == 0) {
        uint64_t tot[kAbsLimbs];
        int f = 0;
#pragma unroll
        for (int k = 0; k < kAbsLimbs; ++k) tot[k] = 0ull;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
#pragma unroll
            for (int k = 0; k < kAbsLimbs; ++k) tot[k] += part[w][k];
            f |= flags[w];
        }
        const double sum = (f & 1) ? (double)NAN : ((f & 2) ? (double)INFINITY : abs_limbs_to_double(tot));
        const double mean = sum / (double)D;
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
        for (int t = 0; t < T; ++t) {
            const uint8_t b = (uint8_t)((mag >> t) & 1);
            const size_t at = ((size_t)n * rs + t) * D + i;
            plus[at] = q > 0 ? b : (uint8_t)0;
            minus[at] = q < 0 ? b : (uint8_t)0;
        }
    }
}

// y[n][o] = sum_t 2^t (acc+[n*T + t][o] - acc-[n*T + t][o]); one thread per (n, o),
// consecutive threads on consecutive o.
__global__ void __launch_bounds__(256) k_ternary_combine(const int32_t* accp, const int32_t* accm,
                                                         int N, int T, int rs, int d_out,
                                                         int32_t* y) {
    pdl_wait();
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)N * d_out) return;
    const int n = (int)(idx / d_out), o = (int)(idx % d_out);
    long long s = 0;
    for (int t = 0; t < T; ++t) {
        const size_t at = ((size_t)n * rs + t) * d_out + o;
        s += (long long)(__ldg(accp + at) - __ldg(accm + at)) * (1ll << t);
    }
    y[idx] = (int32_t)s;
}

// Modified IF of Sec. II-C (Eq. (9)-(10), the library's reading): the bit-weighted
// input y is integrated at once, then steps t = T..1 emit +1 when v >= 2^{t-1} theta,
// -1 when v <= -2^{t-1} theta, else 0, subtracting 2^{t-1} theta s_t from v.  One thread
// per (n, o), consecutive threads on consecutive o; spikes [N][T][d_out] (plane t-1),
// the residual v after step 1 in v_out.
__global__ void __launch_bounds__(256) k_ternary_if(const int32_t* y, int N, int d_out, int T,
                                                    int theta, int8_t* s_out, int32_t* v_out) {
    pdl_wait();
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)N * d_out) return;
    const int n = (int)(idx / d_out), o = (int)(idx % d_out);
    long long v = __ldg(y + idx);
    for (int t = T; t >= 1; --t) {
        const long long thr = (long long)theta << (t - 1);
        const int s = v >= thr ? 1 : (v <= -thr ? -1 : 0);
        v -= thr * s;
        s_out[((size_t)n * T + (t - 1)) * d_out + o] = (int8_t)s;
    }
    if (v_out) v_out[idx] = (int32_t)v;
}

nmdlm_status launch_ternary_if(const int32_t* y, int N, int d_out, int T, int theta,
                               int8_t* s_out, int32_t* v_out, cudaStream_t stream) {
    const long long total = (long long)N * d_out;
    const cudaError_t le = launch_pdl(k_ternary_if, dim3((unsigned)((total + 255) / 256)),
                                      dim3(256), 0, stream, 1, y, N, d_out, T, theta, s_out,
                                      v_out);
    count_launch();
    return cuda_status(le);
}

nmdlm_status launch_ternary_encode(const float* a, int N, int D, float K, int T, int rs,
                                   uint8_t* plus, uint8_t* minus, int32_t* ahat, float* vth,
                                   cudaStream_t stream) {
    const cudaError_t le = launch_pdl(k_ternary_encode, dim3(N), dim3(256), 0, stream, 1, a, D,
                                      K, T, rs, plus, minus, ahat, vth);
    count_launch();
    return cuda_status(le);
}

nmdlm_status launch_ternary_combine(const int32_t* accp, const int32_t* accm, int N, int T,
                                    int rs, int d_out, int32_t* y, cudaStream_t stream) {
    const long long total = (long long)N * d_out;
    const cudaError_t le = launch_pdl(k_ternary_combine, dim3((unsigned)((total + 255) / 256)),
                                      dim3(256), 0, stream, 1, accp, accm, N, T, rs, d_out, y);
    count_launch();
    return cuda_status(le);
}

}  // namespace nmdlm
