// attention_tc.cu -- spike attention with scores and mixture on the 5th-generation tensor
// cores (kind::f8f6f4).
//
// One CTA per (head h, timestep t, tile of up to 32 queries), d_head = 128 (the reading
// of the paper's binary-binary attention, Fig. 1, is the one of attention.cu):
//   score[n][j] = popcount(q_n AND k_j)
//   p[n][j]     = exp(alpha * (score[n][j] - c_n)) / Z_n,  Z_n = sum_j exp(...)
//   out[n][d]   = sum_j p[n][j] * v_j[d]
// Softmax is invariant to the shift c_n; this kernel takes c_n = popcount(q_n), the
// largest score query n can reach, so every exponent is <= 0 and no running maximum or
// rescaling is needed: keys are visited once, in tiles of 128, and the partial sums of
// every tile add into one accumulator.
//
// Spikes enter the tensor cores as e4m3 bytes of 2^-5 (0x10) or 0, so every product of
// two spikes, 2^-10, and every sum of them is exact in fp32; within each 32-channel word
// the bytes follow a fixed permutation of the channels that costs two instructions per
// four bytes (bits_to_e4m3x32).
//
// Scores: S^T = K Q^T per tile, M = 128 keys, N = 32 queries, K = 128 channels in 4
// steps of 32; both operands K-major in shared memory (Q once, K per tile).
//
// Weights: a table holds, for each of the d_head + 1 values x = c_n - score, the weight
// w(x) = 2^8 exp(-alpha x) as four e4m3 pieces e_0..e_3 with w(x) ~ sum_i e_i 2^-4i
// (greedy, round to nearest: each piece carries the next four significant bits, so the
// sum is within 2^-16 of w(x) relatively while w(x) >= 2^-6, and within 2^-22 absolutely
// below).  A score becomes the byte offset of its table entry with one fp32 add and a
// mask: score 2^-10 + 2^11 + (d_head - c_n) 2^-10 has 4 (score + d_head - c_n) in its
// low mantissa bits.
//
// Mixture: O = P V per tile, M = 128 (piece i of query n in row 4 n + i), N = 144 (the
// head's 128 channels, then a channel of ones and 15 zeros), K = 128 keys in 4 steps of
// 32, fp32 accumulation in tensor memory.  Both operands are MN-major e4m3 core matrices
// in shared memory: for a key, its 32 rows of P (8 queries x 4 pieces) are one thread's
// table entries, and its channels are its V bits spread to bytes, so neither needs a
// transpose.  The column of ones makes Z_n come out of the same MMAs, from the same
// pieces: out = sum_i 2^-4i O[4n + i][d] / sum_i 2^-4i O[4n + i][128], numerator and
// denominator over the same weights, an exact softmax of weights within 2^-16 of the
// true ones (2^-12 for the smallest).
//
// Roles: 16 worker warps (warp w: keys 32 (w % 4) .. + 31 of a tile, channel quarter and
// queries 8 (w / 4) .. + 7) stage the K and V words of four tiles ahead (16 bytes per
// key and thread, cp.async counted on an mbarrier), expand the next tile's K and V, read
// this tile's scores from tensor memory and write P; one thread issues the MMAs, the
// scores of tile j + 1 before the mixture of tile j.  NST stages of every operand.  Every
// wait is bounded.
#include <algorithm>

#include "internal.h"

namespace nmdlm {
// Debug timestamps, compiled in with -DNMDLM_ATTN_TRACE: of CTA (0, 0, 0), thread `th`
// (clock64), and per CTA (globaltimer), when a.dbg is set.
#ifdef NMDLM_ATTN_TRACE
#define NMDLM_ASTAMP(a, th, slot)                                                    \
    do {                                                                             \
        if ((a).dbg && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0 &&       \
            threadIdx.x == (th) && (slot) < 4096)                                    \
            (a).dbg[(slot)] = clock64();                                             \
    } while (0)
#define NMDLM_ACSTAMP(a, ev) NMDLM_CSTAMP(a, 1024, ev)
#else
#define NMDLM_ASTAMP(a, th, slot) do {} while (0)
#define NMDLM_ACSTAMP(a, ev) do {} while (0)
#endif
namespace attn3 {
constexpr int DH = 128;                       // head width
constexpr int NQ = 32;                        // queries per CTA
constexpr int KT = 128;                       // keys per tile
constexpr int NPC = 4;                        // e4m3 pieces per weight
constexpr int MO = NQ * NPC;                  // mixture M: 128 rows (query, piece)
constexpr int NO = DH + 16;                   // mixture N: channels, then ones + zeros
constexpr int NST = 4;                        // operand stages
constexpr int NWK = 16;                       // worker warps
constexpr int QQ = 8;                         // queries per worker thread
constexpr int WARP_MMA = NWK;                 // 16
constexpr int NTHREADS = (NWK + 1) * 32;      // 544
constexpr int WSCALE_LOG2 = 8;                // weights scaled by 2^8 (largest 256 <= 448)
constexpr int NLUT = 512;                     // table entries: 0..DH weights, the rest 0
constexpr int MNLBO = 128;                    // MN-major: bytes between K-adjacent cores
constexpr int MNSBO = (KT / 8) * 128;         // ... between 16-row groups along M / N
constexpr int P_BYTES = MO * KT;              // P of a tile: 16 KB
constexpr int V_BYTES = NO * KT;              // V of a tile with the ones: 18 KB
constexpr int SK_BYTES = KT * DH;             // K of a tile, K-major: 16 KB
constexpr int QB_BYTES = NQ * DH;             // Q, K-major: 4 KB
constexpr int KSBO = (DH / 16) * 128;         // K-major: bytes between 8-row groups
constexpr int TM_S = 256;                     // tensor memory: O at 0, score stages
constexpr int NCOL = 512;
constexpr int OFF_P = 0;
constexpr int OFF_V = OFF_P + NST * P_BYTES;
constexpr int OFF_SK = OFF_V + NST * V_BYTES;
constexpr int OFF_QB = OFF_SK + NST * SK_BYTES;
constexpr int OFF_Q = OFF_QB + QB_BYTES;      // [NQ] query words
constexpr int OFF_LUT = OFF_Q + NQ * 16;      // [NLUT] pieces
constexpr int NKV = 4;                        // tiles of K / V words in flight
constexpr int KV_BYTES = 2 * KT * 16;         // a tile's K words, then its V words
constexpr int OFF_KV = OFF_LUT + NLUT * 4;
constexpr int OFF_BAR = OFF_KV + NKV * KV_BYTES;  // 4 per stage + NKV + 1, TMEM, abort
constexpr int SMEM_BYTES = OFF_BAR + 8 * (4 * NST + NKV + 1) + 16 + 1024;
static_assert(NO <= TM_S && TM_S + NST * NQ <= NCOL, "tensor memory budget");
static_assert(SMEM_BYTES <= 225 * 1024, "shared memory budget");

// 32 spike bits -> 32 e4m3 bytes of 2^-5 (0x10) / 0 in a fixed channel order: byte j of
// word i (byte 4i + j of the 32) is bit 8j + i, so each word is one shift and one mask.
// K and Q take the same order (a dot product does not see it); for V it is the order of
// the mixture's columns, which the epilogue undoes (column 4i + j = channel 8j + i).
__device__ __forceinline__ void bits_to_e4m3x32(uint32_t x, uint32_t (&w)[8]) {
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = (i <= 4 ? x << (4 - i) : x >> (i - 4)) & 0x10101010u;
}
// the mixture column of channel c of a 32-channel word
__host__ __device__ constexpr int col_of_channel(int c) { return 4 * (c % 8) + c / 8; }

// e4m3 (1 sign bit, 4 exponent bits of bias 7, 3 mantissa bits, subnormals below 2^-6,
// largest finite 448) nearest to v, ties to even, for |v| <= 256; `back` = its value.
// All in fp32 with power-of-two scalings, so `back` and v - back are exact.
__device__ __forceinline__ uint32_t e4m3_rn(float v, float& back) {
    const uint32_t sign = v < 0.0f ? 0x80u : 0u;
    const float av = fabsf(v);
    int e = (int)((__float_as_uint(av) >> 23) & 0xFFu) - 127;  // floor(log2 av), av normal
    if (e < -6) e = -6;                                          // subnormal quantum 2^-9
    const float up = __uint_as_float((uint32_t)(127 + 3 - e) << 23);    // 2^(3 - e)
    const float qn = __uint_as_float((uint32_t)(127 - 3 + e) << 23);    // 2^(e - 3)
    float m = rintf(av * up);                                    // 0 .. 16
    back = sign ? -m * qn : m * qn;
    if (m >= 16.0f) { m = 8.0f; e += 1; }                        // into the next binade
    if (m < 8.0f) return sign | (uint32_t)m;                     // subnormal, or zero
    return sign | ((uint32_t)(e + 7) << 3) | ((uint32_t)m - 8u);
}

// kind::f8f6f4 instruction descriptor, e4m3 A and B, fp32 accumulate.
__device__ __forceinline__ uint32_t idesc_e4m3(int M, int N, bool a_mn, bool b_mn) {
    return (1u << 4) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
           ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// D[tmem] (+)= A[smem] * B[smem], kind::f8f6f4.
__device__ __forceinline__ void mma_e4m3_ss(uint32_t td, uint64_t ad, uint64_t bd, uint32_t id,
                                            uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(td),
        "l"(ad), "l"(bd), "r"(id), "r"(acc)
        : "memory");
}
}  // namespace attn3

__global__ void __launch_bounds__(attn3::NTHREADS, 1) k_attention_tc(const __grid_constant__ AttnArgs a) {
    using namespace attn3;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const int L = a.L;
    uint4* q_s = (uint4*)(smem + OFF_Q);
    uint32_t* lut = (uint32_t*)(smem + OFF_LUT);
    uint64_t* bar = (uint64_t*)(smem + OFF_BAR);
    uint64_t* p_full = bar;             // [NST] P (and V) of the tile written (NWK)
    uint64_t* st_free = bar + NST;      // [NST] the tile's mixture completed
    uint64_t* k_full = bar + 2 * NST;   // [NST] K of the tile expanded (NWK)
    uint64_t* s_full = bar + 3 * NST;   // [NST] the tile's scores in tensor memory
    uint64_t* kv_full = bar + 4 * NST;  // [NKV] a tile's K and V words landed (2 KT)
    uint64_t* done = bar + 4 * NST + NKV;  // every MMA completed
    uint32_t* tmem_holder = (uint32_t*)(done + 1);
    volatile int* abort_flag = (volatile int*)(done + 1) + 1;

    const int h = blockIdx.x, t = blockIdx.y, q0 = blockIdx.z * NQ;
    const int nq = min(NQ, a.B - q0);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int WD = words_of(a.H * DH);
    const int ntile = (L + KT - 1) / KT;
    NMDLM_ACSTAMP(a, 0);

    // ---- setup that reads nothing another kernel writes
    for (int x = tid; x < NLUT; x += NTHREADS) {
        // table entry x: the weight of score - c = x - DH as four e4m3 pieces
        uint32_t bytes = 0u;
        if (x <= DH) {
            float r = expf(-__fmul_rn(a.alpha, (float)(DH - x))) * (float)(1 << WSCALE_LOG2);
#pragma unroll
            for (int i = 0; i < NPC; ++i) {
                const float sc = __uint_as_float((uint32_t)(127 + 4 * i) << 23);   // 2^4i
                const float isc = __uint_as_float((uint32_t)(127 - 4 * i) << 23);  // 2^-4i
                float back;
                bytes |= e4m3_rn(r * sc, back) << (8 * i);
                r -= back * isc;
            }
        }
        lut[x] = bytes;
    }
    // the ones channel (128) and 15 zero channels of V, every stage, every key
    for (int j = tid; j < NST * KT; j += NTHREADS) {
        const int s = j / KT, key = j % KT;
        *reinterpret_cast<uint4*>(smem + OFF_V + s * V_BYTES + (key >> 3) * MNLBO + (key & 7) * 16 +
                                  (DH / 16) * MNSBO) = make_uint4(0x10u, 0u, 0u, 0u);
    }
    fence_proxy_async_smem();
    if (tid == 0) {
        *abort_flag = 0;
        for (int s = 0; s < NST; ++s) {
            mbar_init(&p_full[s], NWK);
            mbar_init(&st_free[s], 1);
            mbar_init(&k_full[s], NWK);
            mbar_init(&s_full[s], 1);
        }
        for (int r = 0; r < NKV; ++r) mbar_init(&kv_full[r], 2 * KT);
        mbar_init(done, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == WARP_MMA) {
        tmem_alloc(tmem_holder, NCOL);
        tmem_relinquish();
    }
    pdl_wait();
    NMDLM_ASTAMP(a, 0, 40);
    NMDLM_ACSTAMP(a, 1);
    // ---- this tile's queries, and the Q operand: query n's 128 channels as e4m3 bytes,
    // K-major core matrices (8 queries x 16 bytes): group n / 8 at KSBO, chunk j at 128
    if (tid < NQ) {
        uint4 qv = make_uint4(0u, 0u, 0u, 0u);
        if (tid < nq) qv = *reinterpret_cast<const uint4*>(a.q + (size_t)((q0 + tid) * a.T + t) * WD + h * 4);
        q_s[tid] = qv;
        uint8_t* qb = smem + OFF_QB + (tid >> 3) * KSBO + (tid & 7) * 16;
        const uint32_t qw[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            uint32_t e[8];
            bits_to_e4m3x32(qw[w], e);
            *reinterpret_cast<uint4*>(qb + (2 * w) * 128) = make_uint4(e[0], e[1], e[2], e[3]);
            *reinterpret_cast<uint4*>(qb + (2 * w + 1) * 128) = make_uint4(e[4], e[5], e[6], e[7]);
        }
        fence_proxy_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    NMDLM_ASTAMP(a, 0, 41);
    NMDLM_ACSTAMP(a, 2);

    if (warp < NWK) {
        // ------------------------------------------------------------------ workers
        const int lq = warp & 3, qg = warp >> 2;
        const int k = lq * 32 + lane;          // key row of the tile
        const uint32_t tl = tmem + ((uint32_t)(lq * 32) << 16);  // this warp's lanes
        // K (warps of query group 0) and V (group 1) words of key k of tile j into ring
        // slot j % NKV, 16 bytes a thread (zeros past L), counted on kv_full.  Slot j % NKV
        // last held tile j - NKV, which every warp expanded before tile j - NKV's scores
        // (k_full), and the load is issued only after this thread saw those scores.
        const uint32_t* kvg = (qg == 0 ? a.k : a.v) + (size_t)t * a.Ls * WD + h * 4;
        auto load_kv = [&](int j) {
            if (qg < 2 && j < ntile) {
                const int key = j * KT + k;
                cp_async16(smem + OFF_KV + (j % NKV) * KV_BYTES + qg * (KT * 16) + k * 16,
                           kvg + (size_t)(key < L ? key : 0) * WD, key < L ? 16u : 0u);
                cp_async_mbar_arrive(&kv_full[j % NKV]);
            }
        };
        // table offset base per query: 2^11 + (DH - c_n) 2^-10; keys past L add 2^-2
        // (entry + 256, a zero entry)
        float base[QQ];
#pragma unroll
        for (int i = 0; i < QQ; ++i) {
            const uint4 qv = q_s[qg * QQ + i];
            const int cq = __popc(qv.x) + __popc(qv.y) + __popc(qv.z) + __popc(qv.w);
            base[i] = 2048.0f + (float)(DH - cq) * (1.0f / 1024.0f);
        }
        const uint8_t* lutb = reinterpret_cast<const uint8_t*>(lut);
        // K and V of tile j into stage j % NST: K K-major (key group k / 8 at KSBO, 16-channel
        // chunk at 128), V MN-major (key group at MNLBO, 16-channel group at MNSBO).  The
        // stage's previous readers are tile j - NST's MMAs (st_free); its score MMA also
        // completed before this thread read that tile's scores.  Warp w expands keys
        // 8 w .. 8 w + 7, lane = key (lane % 8) x 32-channel word (lane / 8): the warp's
        // word loads cover 128 contiguous bytes of the ring, and each 8 lanes' 16-byte
        // stores one 128-byte row of core matrices.
        const int ek = warp * 8 + (lane & 7), ew = lane >> 3;
        auto expand = [&](int j) -> bool {
            const int s = j % NST, u = j / NST;
            bool ok = mbar_wait_bounded(&kv_full[j % NKV], (j / NKV) & 1, a.wait_ns);
            if (u > 0 && ok) ok = mbar_wait_bounded(&st_free[s], (u - 1) & 1, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok)) return false;  // bounded: a stalled role ends it
            NMDLM_ASTAMP(a, 0, 800 + j);
            const uint8_t* slot = smem + OFF_KV + (j % NKV) * KV_BYTES + ek * 16 + ew * 4;
            const uint32_t kw = *reinterpret_cast<const uint32_t*>(slot);
            const uint32_t vw = *reinterpret_cast<const uint32_t*>(slot + KT * 16);
            uint32_t e[8];
            bits_to_e4m3x32(kw, e);
            uint8_t* kd = smem + OFF_SK + s * SK_BYTES + (ek >> 3) * KSBO + (2 * ew) * 128 + (ek & 7) * 16;
            *reinterpret_cast<uint4*>(kd) = make_uint4(e[0], e[1], e[2], e[3]);
            *reinterpret_cast<uint4*>(kd + 128) = make_uint4(e[4], e[5], e[6], e[7]);
            bits_to_e4m3x32(vw, e);
            uint8_t* vd = smem + OFF_V + s * V_BYTES + (ek >> 3) * MNLBO + (ek & 7) * 16 + (2 * ew) * MNSBO;
            *reinterpret_cast<uint4*>(vd) = make_uint4(e[0], e[1], e[2], e[3]);
            *reinterpret_cast<uint4*>(vd + MNSBO) = make_uint4(e[4], e[5], e[6], e[7]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&k_full[s]);
            NMDLM_ASTAMP(a, 0, 900 + j);
            return true;
        };
        // the words of tiles 0 .. NKV - 1 in flight
#pragma unroll
        for (int j = 0; j < NKV; ++j) load_kv(j);
        bool run = ntile > 0 ? expand(0) : true;
        for (int kt = 0; kt < ntile && run; ++kt) {
            const int s = kt % NST, u = kt / NST;
            if (kt + 1 < ntile && !expand(kt + 1)) { run = false; break; }
            // this tile's scores: lane = key, columns = the group's 8 queries
            const bool okS = mbar_wait_bounded(&s_full[s], u & 1, a.wait_ns);
            if (!__all_sync(0xffffffffu, okS)) { run = false; break; }
            load_kv(kt + NKV);
            NMDLM_ASTAMP(a, 0, 400 + kt);
            tc_fence_after();
            uint32_t sv[8];
            tmem_ld8(tl + (uint32_t)(TM_S + s * NQ + qg * QQ), sv);
            // mantissa bits 2..10 = entry score + DH - c_n (+ 256 past L); whatever the
            // accumulator holds, the offset stays inside the table
            constexpr uint32_t OMASK = (NLUT - 1) * 4;
            uint32_t pc[QQ];
            if ((kt + 1) * KT <= L) {
#pragma unroll
                for (int i = 0; i < QQ; ++i)
                    pc[i] = *reinterpret_cast<const uint32_t*>(
                        lutb + (__float_as_uint(__fadd_rn(__uint_as_float(sv[i]), base[i])) & OMASK));
            } else {
                const float past = kt * KT + k < L ? 0.0f : 0.25f;
#pragma unroll
                for (int i = 0; i < QQ; ++i)
                    pc[i] = *reinterpret_cast<const uint32_t*>(
                        lutb + (__float_as_uint(__fadd_rn(__uint_as_float(sv[i]), base[i] + past)) & OMASK));
            }
            // P rows 4 n + i of queries 8 qg .. + 7 = 32 consecutive rows for key k: two
            // 16-byte pieces, 16-row group at MNSBO, key group k / 8 at MNLBO.  The stage
            // was freed before tile kt's V went in (expand).
            uint8_t* P = smem + OFF_P + s * P_BYTES + (k >> 3) * MNLBO + (k & 7) * 16 + (2 * qg) * MNSBO;
            *reinterpret_cast<uint4*>(P) = make_uint4(pc[0], pc[1], pc[2], pc[3]);
            *reinterpret_cast<uint4*>(P + MNSBO) = make_uint4(pc[4], pc[5], pc[6], pc[7]);
            fence_proxy_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_full[s]);
            NMDLM_ASTAMP(a, 0, 200 + kt);
        }
        if (!run && lane == 0) { *abort_flag = 1; raise_error(a.err, ERRBIT_TIMEOUT); }
    } else {
        // -------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc_s = idesc_e4m3(KT, NQ, false, false);
            const uint32_t idesc_o = idesc_e4m3(MO, NO, true, true);
            const uint64_t kd0 = smem_desc(smem_u32(smem + OFF_SK), 128, KSBO);
            const uint64_t qd0 = smem_desc(smem_u32(smem + OFF_QB), 128, KSBO);
            const uint64_t pd0 = smem_desc(smem_u32(smem + OFF_P), MNLBO, MNSBO);
            const uint64_t vd0 = smem_desc(smem_u32(smem + OFF_V), MNLBO, MNSBO);
            constexpr uint64_t CSTEP = 2 * 128 / 16;    // 32 channels = two 16-byte chunks
            constexpr uint64_t KSTEP = 4 * MNLBO / 16;  // 32 keys = four core matrices
            // scores of tile kt: S^T = K Q^T into the stage's score columns
            auto issue_s = [&](int kt) -> bool {
                const int s = kt % NST, u = kt / NST;
                if (*abort_flag || !mbar_wait_bounded(&k_full[s], u & 1, a.wait_ns)) return false;
                tc_fence_after();
                const uint64_t kd = kd0 + (uint64_t)(s * (SK_BYTES >> 4));
#pragma unroll
                for (int j = 0; j < DH / 32; ++j)
                    mma_e4m3_ss(tmem + (uint32_t)(TM_S + s * NQ), kd + j * CSTEP, qd0 + j * CSTEP,
                                idesc_s, j > 0 ? 1u : 0u);
                mma_commit(&s_full[s]);
                return true;
            };
            bool ok = ntile > 0 ? issue_s(0) : true;
            for (int kt = 0; kt < ntile && ok; ++kt) {
                const int s = kt % NST, u = kt / NST;
                NMDLM_ASTAMP(a, WARP_MMA * 32, 300 + 2 * kt);
                // the next tile's scores go ahead of this tile's mixture
                if (kt + 1 < ntile && !issue_s(kt + 1)) { ok = false; break; }
                NMDLM_ASTAMP(a, WARP_MMA * 32, 600 + kt);
                ok = !*abort_flag && mbar_wait_bounded(&p_full[s], u & 1, a.wait_ns);
                if (!ok) break;
                NMDLM_ASTAMP(a, WARP_MMA * 32, 700 + kt);
                tc_fence_after();
                const uint64_t pd = pd0 + (uint64_t)(s * (P_BYTES >> 4));
                const uint64_t vd = vd0 + (uint64_t)(s * (V_BYTES >> 4));
#pragma unroll
                for (int kk = 0; kk < KT / 32; ++kk)
                    mma_e4m3_ss(tmem, pd + kk * KSTEP, vd + kk * KSTEP, idesc_o, (kt > 0 || kk > 0) ? 1u : 0u);
                mma_commit(&st_free[s]);
                NMDLM_ASTAMP(a, WARP_MMA * 32, 301 + 2 * kt);
            }
            if (!ok) {
                *abort_flag = 1;
                raise_error(a.err, ERRBIT_TIMEOUT);
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
    const bool aborted = __syncthreads_or(!ok);
    tc_fence_after();
    NMDLM_ASTAMP(a, 0, 42);
    if (!aborted && warp < NWK) {
        // ---------- epilogue: out[n][d] = sum_i 2^-4i O[4n + i][d] / (same at column DH)
        // (V and the ones column carry the same 2^-5, which cancels)
        // warp w: rows 32 (w % 4) .. + 31 (lane = 4 n' + i), channels 32 (w / 4) .. + 31;
        // the pieces of a query are 4 adjacent lanes, summed smallest first (Horner)
        const int lq = warp & 3, cg = warp >> 2, i = lane & 3;
        const int n = lq * 8 + (lane >> 2);
        uint32_t o[32], oz[8];
        tmem_ld32(tmem + ((uint32_t)(lq * 32) << 16) + (uint32_t)(cg * 32), o);
        tmem_ld8(tmem + ((uint32_t)(lq * 32) << 16) + (uint32_t)DH, oz);
        auto horner = [&](float x) {
            float y = __shfl_down_sync(0xffffffffu, x, 1);
            x = i == 2 ? __fmaf_rn(y, 0.0625f, x) : x;
            y = __shfl_down_sync(0xffffffffu, x, 1);
            x = i == 1 ? __fmaf_rn(y, 0.0625f, x) : x;
            y = __shfl_down_sync(0xffffffffu, x, 1);
            return i == 0 ? __fmaf_rn(y, 0.0625f, x) : x;
        };
        const float z = horner(__uint_as_float(oz[0]));
        float num[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) num[j] = horner(__uint_as_float(o[j]));
        if (i == 0 && n < nq) {
            // one reciprocal per query: each output within 1.5 ulp of the quotient
            const float rz = __frcp_rn(z);
            float4* dst = reinterpret_cast<float4*>(a.out + (size_t)((q0 + n) * a.T + t) * (a.H * DH) + h * DH + cg * 32);
#pragma unroll
            for (int j = 0; j < 8; ++j)
                dst[j] = make_float4(__fmul_rn(num[col_of_channel(4 * j)], rz),
                                     __fmul_rn(num[col_of_channel(4 * j + 1)], rz),
                                     __fmul_rn(num[col_of_channel(4 * j + 2)], rz),
                                     __fmul_rn(num[col_of_channel(4 * j + 3)], rz));
        }
    }
    if (aborted && tid == 0) raise_error(a.err, ERRBIT_TIMEOUT);
    tc_fence_before();
    __syncthreads();
    NMDLM_ASTAMP(a, 0, 43);
    NMDLM_ACSTAMP(a, 3);
    if (warp == WARP_MMA) tmem_dealloc(tmem, NCOL);
}

// UNSUPPORTED unless d_head is 128 and alpha is small enough that the weight of the
// lowest score, 2^8 exp(-128 alpha), is at least 2^-10: the pieces of a weight below the
// normal range still carry it to 2^-22 absolutely, so every weight keeps a relative
// error of at most 2^-12 (2^-16 for weights of 2^-6 and more).  Shared memory does not
// depend on the number of keys (their words stream through a ring of NKV tiles).
nmdlm_status launch_attention_tc(const AttnArgs& a, cudaStream_t stream) {
    using namespace attn3;
    if (a.dh != DH || a.L < 1 || a.B < 1) return NMDLM_ERR_UNSUPPORTED;
    if (!(a.alpha >= 0.0f) || (double)a.alpha * DH > (WSCALE_LOG2 + 10) * 0.6931471805599453)
        return NMDLM_ERR_UNSUPPORTED;
    if (ensure_dyn_smem((const void*)k_attention_tc, SMEM_BYTES) != NMDLM_OK) return NMDLM_ERR_CUDA;
    const dim3 grid(a.H, a.T, (a.B + NQ - 1) / NQ);
    const cudaError_t le = launch_pdl(k_attention_tc, grid, dim3(NTHREADS), (size_t)SMEM_BYTES, stream, 1, a);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

}  // namespace nmdlm
