// linear.cu -- QBSM spiking linear layers with the IF epilogue fused in.
//
// acc[bt][o] = sum over active input channels d of x[bt][d] * W^T[d][o]  (Sec. IV-A):
// a row of W^T is fetched only when its input channel spiked in some row of the
// block (assumption (ii)).  Two kernel families compute the same exact int32 sums:
//   k_linear_simt  CUDA-core accumulation (small blocks, any shape);
//   k_linear_tc    gather-then-MMA on the 5th-generation tensor cores: the active
//                  rows of W^T are gathered into shared memory as the K dimension,
//                  converted int8 -> fp16 (exact), multiplied by the 0/1 spike operand
//                  with tcgen05.mma kind::f16 into fp32 TMEM accumulators.  Products
//                  are exact and every partial sum is an integer below 2^24
//                  (|acc| <= 127 * d_in), so the fp32 result equals the int32 sum.
// Both end in the same IF epilogue (Sec. II-B, Eq. (3)-(4)), so spikes leave the
// kernel packed and never round-trip through memory as integers.
#include <algorithm>
#include <cstdio>

#include <cudaTypedefs.h>

#include <type_traits>

#include "internal.h"

namespace nmdlm {

// ------------------------------------------------------------------ SIMT ----
// grid.x: groups of 32 output channels; block (32, BY).  Thread (lane, ty) owns
// channel lo0 + lane for tokens ty, ty + BY, ...
template <int MAXT, int MAXW>
__global__ void k_linear_simt(LinArgs a) {
    pdl_wait();
    const int g = blockIdx.x;
    const int si = seg_of_tile(a, g);
    const LinSeg& s = a.seg[si];
    const int lane = threadIdx.x, ty = threadIdx.y, BY = blockDim.y;
    const int lo = (g - s.tile_begin) * 32 + lane;
    const bool valid = lo < s.n_out;
    __shared__ uint32_t cm_s[32][MAXW];
    __shared__ int any_s[32];
    for (int i = threadIdx.y * 32 + lane; i < 32 * MAXW; i += 32 * BY) cm_s[i / MAXW][i % MAXW] = 0;
    if (ty == 0) any_s[lane] = 0;
    __syncthreads();

    uint32_t cmw[MAXW];
#pragma unroll
    for (int w = 0; w < MAXW; ++w) cmw[w] = 0;
    bool any = false;
    const int DW = words_of(a.d_in);
    const int T = a.T, BTW = a.BTW;
    for (int b = ty; b < a.B; b += BY) {
        int acc[MAXT];
#pragma unroll
        for (int t = 0; t < MAXT; ++t) acc[t] = 0;
        const int bt0 = b * T, w0 = bt0 >> 5, sh = bt0 & 31;
        for (int w = 0; w < DW; ++w) {
            uint32_t m;
            if (a.dense) {
                const int rem = a.d_in - w * 32;
                m = rem >= 32 ? 0xffffffffu : ((1u << rem) - 1u);
            } else {
                m = a.in_mask[w];
            }
            while (m) {
                const int d = w * 32 + __ffs(m) - 1;
                m &= m - 1;
                const int wv = valid ? (int)s.wT[(size_t)d * s.ld_w + lo] : 0;
                const uint32_t* c = a.in_cm + (size_t)d * BTW;
                uint64_t win = c[w0];
                if (w0 + 1 < BTW) win |= (uint64_t)c[w0 + 1] << 32;
                const uint32_t bits = (uint32_t)(win >> sh);
#pragma unroll
                for (int t = 0; t < MAXT; ++t)
                    if (t < T) acc[t] += ((bits >> t) & 1u) ? wv : 0;
            }
        }
        epi_token<MAXT, MAXW>(a, s, lo, valid, b, [&](int t) { return acc[t]; }, cmw, any);
    }
#pragma unroll
    for (int w = 0; w < MAXW; ++w)
        if (w < BTW && cmw[w]) atomicOr(&cm_s[lane][w], cmw[w]);
    if (any) any_s[lane] = 1;
    __syncthreads();
    if (ty == 0) {
        if (valid && s.cm)
            for (int w = 0; w < BTW; ++w) s.cm[(size_t)lo * BTW + w] = cm_s[lane][w];
        const uint32_t mw = __ballot_sync(0xffffffffu, valid && any_s[lane]);
        if (lane == 0 && s.mask) s.mask[lo >> 5] = mw;
    }
}

// ------------------------------------------------------- block scan (256) ----
// Exclusive prefix sum over the words of the active mask (or all channels when
// dense) into prefix[0..DW]; prefix[DW] is the number of active rows.
// The launch arguments come by value: through a reference the kernel's parameter block
// is read with generic loads of ~1 k cycles each, three of them in a row here.
__device__ void active_prefix(bool dense, int d_in, const uint32_t* in_mask, uint32_t* mask_s,
                              int* prefix, int DW) {
    const int tid = threadIdx.x;
    const int per = (DW + blockDim.x - 1) / blockDim.x;
    const int beg = tid * per, end = min(beg + per, DW);
    int local = 0;
    for (int w = beg; w < end; ++w) {
        uint32_t m;
        if (dense) {
            const int rem = d_in - w * 32;
            m = rem >= 32 ? 0xffffffffu : ((1u << rem) - 1u);
        } else {
            m = in_mask[w];
        }
        mask_s[w] = m;
        local += __popc(m);
    }
    // inclusive scan of `local` across the block
    __shared__ int warp_tot[32];
    const int lane = tid & 31, warp = tid >> 5;
    int x = local;
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
        if (lane < nw) warp_tot[lane] = y;  // inclusive warp totals
    }
    __syncthreads();
    int run = x - local + (warp > 0 ? warp_tot[warp - 1] : 0);  // exclusive prefix
    for (int w = beg; w < end; ++w) {
        prefix[w] = run;
        run += __popc(mask_s[w]);
    }
    if (tid == blockDim.x - 1) prefix[DW] = run;  // last thread holds the total
    __syncthreads();
}

// Row of W^T (input channel) holding compacted position p, or -1 past the end.
__device__ __forceinline__ int active_row(const uint32_t* mask_s, const int* prefix, int DW,
                                          int p) {
    if (p >= prefix[DW]) return -1;
    int lo = 0, hi = DW;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (prefix[mid] <= p) lo = mid; else hi = mid;
    }
    return lo * 32 + (int)__fns(mask_s[lo], 0, p - prefix[lo] + 1);
}

// ---------------------------------------------------------------- tcgen05 ----
// Gather-then-MMA, warp-specialised.  A CTA owns TILE output channels (one or two
// 128-lane TMEM accumulators), every row bt of the block (MMA N = BT padded to NP) and
// one split of the active rows of W^T, taken 64 rows (one chunk) at a time:
//   2 producer warps (alternating chunks) load each 128-channel half of the chunk's
//       active rows with TMA -- a 2-D tile when the rows are consecutive, else
//       tile::gather4 (4 rows per instruction) -- with the 128-byte swizzle, plus the
//       rows' column-mask words, into a ring of NRAW stages;
//   16 converter warps in 2 groups (alternating chunks) turn int8 into fp16 (exact)
//       and spike bits into a 0/1 fp16 operand, both MN-major;
//   1 MMA warp issues tcgen05.mma (M 128, N NP, K 16) per half and K step into fp32
//       TMEM and commits to the operand stage's "free" barrier.
// Every hand-off is an mbarrier with a bounded wait.  Splits of one tile form a
// thread-block cluster and add their partial tiles through distributed shared memory;
// every partial sum is an exact integer below 2^24, so the order does not matter.
namespace tcl {
constexpr int M = 128;         // TMEM lanes per accumulator (output channels per half)
constexpr int KC = 64;         // rows of W^T per chunk
constexpr int NOP = 2;         // fp16 operand stages (one per converter group)
constexpr int NCONV = 16;      // converter warps (also the epilogue warps)
constexpr int NGRP = 2;        // converter groups
constexpr int GWARPS = NCONV / NGRP;
constexpr int NPROD = 2;       // producer warps
constexpr int WARP_PROD = NCONV;
constexpr int WARP_MMA = NCONV + NPROD;
constexpr int NTHREADS = (NCONV + NPROD + 1) * 32;
constexpr int GTHREADS = GWARPS * 32;
constexpr int SBO = (KC / 8) * 128;    // bytes between 8-wide MN core-matrix groups
constexpr int LBO = 128;               // bytes between K-adjacent core matrices
constexpr int MAXROWS = 12288;         // active rows one CTA may own (u16 row list)
constexpr int PFD = 8;                 // chunks prefetched into L2 ahead of the loads

template <int NP, int TILE>
struct Smem {
    static constexpr int HALVES = TILE / M;
    static constexpr int NRAW = TILE == 256 ? 4 : 8;
    static constexpr int RAW_BYTES = KC * TILE;          // int8 weights of one chunk
    static constexpr int A_BYTES = M * KC * 2;            // fp16 operand of one half
    static constexpr int B_BYTES = NP * KC * 2;
    static constexpr int OFF_RAW = 0;
    static constexpr int OFF_A = OFF_RAW + NRAW * RAW_BYTES;
    static constexpr int OFF_B = OFF_A + NOP * HALVES * A_BYTES;
    static constexpr int OFF_CM = OFF_B + NOP * B_BYTES;
    static constexpr int OFF_LUT = OFF_CM + NRAW * KC * 8 * 4;
    static constexpr int OFF_BAR = OFF_LUT + 256 * 16;
    static constexpr int NBAR = 2 * NRAW + 2 * NOP + 3;
    static constexpr int OFF_MISC = OFF_BAR + 8 * NBAR;
    static constexpr int OFF_CMACC = OFF_MISC + 16;           // [TILE][8] u32
    static constexpr int OFF_ANY = OFF_CMACC + TILE * 8 * 4;  // [TILE] int
    static constexpr int OFF_MASK = OFF_ANY + TILE * 4;
    static constexpr int ACC = NP * TILE * 4;  // int32 sums after the main loop, reuse raw/A/B
    static_assert(ACC <= OFF_CM, "accumulator staging must fit in the operand buffers");
    static_assert(RAW_BYTES % 1024 == 0 && OFF_A % 1024 == 0, "swizzle atoms");
    static constexpr int NCOL_NEED = HALVES * NP;
    static constexpr int NCOL = NCOL_NEED <= 32 ? 32 : (NCOL_NEED <= 64 ? 64 : (NCOL_NEED <= 128 ? 128 : (NCOL_NEED <= 256 ? 256 : 512)));
    static size_t bytes(int DW, int rows) {
        return OFF_MASK + 4 * (size_t)(2 * DW + 1) + 2 * (size_t)rows + 1024;
    }
};

// 2-D TMA gather of four rows (x = innermost coordinate), completion on `bar`.
__device__ __forceinline__ void tma_gather4(void* dst, const CUtensorMap* map, int x, int r0,
                                            int r1, int r2, int r3, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cta.global.tile::gather4.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(smem_u32(dst)),
        "l"(map), "r"(x), "r"(r0), "r"(r1), "r"(r2), "r"(r3), "r"(smem_u32(bar))
        : "memory");
}
}  // namespace tcl

template <int NP, int TILE>
__global__ void __launch_bounds__(tcl::NTHREADS, 1) k_linear_tc(const __grid_constant__ LinArgs a) {
    pdl_wait();
    using namespace tcl;
    using SM = Smem<NP, TILE>;
    constexpr int HALVES = SM::HALVES, NRAW = SM::NRAW;
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte aligned start (swizzle atoms), derived by pointer arithmetic so the
    // compiler keeps every access below in the shared state space.
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint32_t* cm_s = (uint32_t*)(smem + SM::OFF_CM);
    const uint4* lut = (const uint4*)(smem + SM::OFF_LUT);
    uint64_t* raw_full = (uint64_t*)(smem + SM::OFF_BAR);
    uint64_t* raw_empty = raw_full + NRAW;
    uint64_t* op_full = raw_empty + NRAW;
    uint64_t* op_empty = op_full + NOP;
    uint64_t* done_bar = op_empty + NOP;
    uint64_t* red_bar = done_bar + 1;  // split-K sums arriving from the peers
    uint64_t* res_bar = done_bar + 2;  // prefetched residual currents
    uint32_t* tmem_holder = (uint32_t*)(smem + SM::OFF_MISC);
    volatile int* abort_flag = (volatile int*)(smem + SM::OFF_MISC + 4);
    uint32_t* cm_acc = (uint32_t*)(smem + SM::OFF_CMACC);
    int* any_acc = (int*)(smem + SM::OFF_ANY);
    const int DW = words_of(a.d_in);
    uint32_t* mask_s = (uint32_t*)(smem + SM::OFF_MASK);
    int* prefix = (int*)(mask_s + DW);
    uint16_t* rowlist = (uint16_t*)(prefix + DW + 1);  // this CTA's active rows, in order

    const int tile = blockIdx.x, split = blockIdx.y;
    const int si = seg_of_tile(a, tile);
    const LinSeg& s = a.seg[si];
    const CUtensorMap* tmap = si == 0 ? &a.tmap[0] : (si == 1 ? &a.tmap[1] : &a.tmap[2]);
    const CUtensorMap* gmap = si == 0 ? &a.gmap[0] : (si == 1 ? &a.gmap[1] : &a.gmap[2]);
    const int lo0 = (tile - s.tile_begin) * TILE;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int BTW = a.BTW;

    NMDLM_TSTAMP(a, 7);
    active_prefix(a.dense != 0, a.d_in, a.in_mask, mask_s, prefix, DW);
    const int n_active = prefix[DW];
    const int nch = (n_active + KC - 1) / KC;
    const int c0 = (int)((long long)split * nch / a.nsplit);
    const int c1 = (int)((long long)(split + 1) * nch / a.nsplit);
    const int nj = c1 - c0;

    // This CTA's compacted rows [c0*KC, c1*KC) of W^T in ascending order; 0xFFFF past
    // the last active row.
    const int r0 = c0 * KC, nrows = nj * KC;
    for (int i = tid; i < nrows; i += NTHREADS) rowlist[i] = 0xFFFFu;
    __syncthreads();
    if (a.dense || n_active == a.d_in) {  // every row active: rows in order
        for (int i = tid; i < nrows; i += NTHREADS)
            if (r0 + i < a.d_in) rowlist[i] = (uint16_t)(r0 + i);
    } else {
        for (int w = tid; w < DW; w += NTHREADS) {
            uint32_t m = mask_s[w];
            int pos = prefix[w];
            if (pos >= r0 + nrows || prefix[w + 1] <= r0) continue;
            while (m) {
                const int bit = __ffs(m) - 1;
                m &= m - 1;
                if (pos >= r0 && pos < r0 + nrows) rowlist[pos - r0] = (uint16_t)(w * 32 + bit);
                ++pos;
            }
        }
    }
    for (int i = tid; i < 256; i += NTHREADS)
        ((uint4*)lut)[i] = make_uint4(bits2_to_f16x2(i), bits2_to_f16x2(i >> 2),
                                      bits2_to_f16x2(i >> 4), bits2_to_f16x2(i >> 6));
    for (int i = tid; i < TILE * 8; i += NTHREADS) cm_acc[i] = 0;
    for (int i = tid; i < TILE; i += NTHREADS) any_acc[i] = 0;
    if (tid == 0) {
        *abort_flag = 0;
        for (int i = 0; i < NRAW; ++i) {
            mbar_init(&raw_full[i], 1 + 32);  // producer's expect_tx + 32 cp.async arrivals
            mbar_init(&raw_empty[i], GWARPS);
        }
        for (int i = 0; i < NOP; ++i) {
            mbar_init(&op_full[i], GWARPS);
            mbar_init(&op_empty[i], 1);
        }
        mbar_init(done_bar, 1);
        mbar_init(red_bar, 1);
        mbar_init(res_bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == WARP_MMA) {
        tmem_alloc(tmem_holder, SM::NCOL);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    NMDLM_TSTAMP(a, 0);

    if (warp >= WARP_PROD && warp < WARP_PROD + NPROD) {
        // ---------------------------------------------------------- producers
        const int p = warp - WARP_PROD;
        // L2 prefetch PFD chunks ahead of the loads: the ring alone keeps too few bytes
        // in flight to cover the memory latency at full bandwidth.
        const int8_t* const wT = s.wT;
        const size_t ldw = (size_t)s.ld_w;
        auto prefetch_chunk = [&](int jj) {
            const uint16_t* ix = rowlist + jj * KC;
            const int row0 = ix[0];
            if (row0 != 0xFFFF && ix[KC - 1] == row0 + KC - 1) {
                if (lane < HALVES) tma_prefetch_2d(tmap, lo0 + lane * M, row0);
            } else {
                for (int k = lane; k < KC; k += 32) {
                    const int d = ix[k];
                    if (d != 0xFFFF) bulk_prefetch_l2(wT + (size_t)d * ldw + lo0, HALVES * M);
                }
            }
        };
        for (int j = p; j < min(nj, PFD); j += NPROD) prefetch_chunk(j);
        for (int j = p; j < nj; j += NPROD) {
            if (j + PFD < nj) prefetch_chunk(j + PFD);
            const int st = j % NRAW, u = j / NRAW;
            if (u > 0) {
                const bool ok = mbar_wait_bounded(&raw_empty[st], (u - 1) & 1, a.wait_ns);
                if (!__all_sync(0xffffffffu, ok) || *abort_flag) {
                    if (lane == 0) { *abort_flag = 1; raise_error(a.err, ERRBIT_TIMEOUT); }
                    break;
                }
            }
            const uint16_t* ix = rowlist + j * KC;
            const int row0 = ix[0];
            const bool contiguous = row0 != 0xFFFF && ix[KC - 1] == row0 + KC - 1;
            uint8_t* raw = smem + SM::OFF_RAW + st * SM::RAW_BYTES;
            uint32_t* cmr = cm_s + st * KC * 8;
            const uint32_t cm_bytes = KC * BTW * 4;
            const bool cm_bulk = contiguous && ((((size_t)row0 * BTW * 4) & 15) == 0) &&
                                 ((((uintptr_t)a.in_cm) & 15) == 0);
            if (lane == 0)
                mbar_arrive_expect_tx(&raw_full[st], (uint32_t)SM::RAW_BYTES +
                                                         (cm_bulk ? cm_bytes : 0u));
            __syncwarp();
            if (contiguous) {
                if (lane < HALVES)
                    tma_load_2d(raw + lane * (KC * M), tmap, lo0 + lane * M, row0, &raw_full[st]);
            } else if (lane < HALVES * (KC / 4)) {
                const int h = lane / (KC / 4), g = lane % (KC / 4);
                int rr[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int d = ix[4 * g + q];
                    rr[q] = d == 0xFFFF ? a.d_in : d;  // out of range: zero fill
                }
                tma_gather4(raw + h * (KC * M) + g * 4 * M, gmap, lo0 + h * M, rr[0], rr[1],
                            rr[2], rr[3], &raw_full[st]);
            }
            if (cm_bulk) {
                if (lane == 0) bulk_load(cmr, a.in_cm + (size_t)row0 * BTW, cm_bytes, &raw_full[st]);
            } else {
                for (int k = lane >> 3; k < KC; k += 4) {
                    const int w = lane & 7;
                    if (w < BTW) {
                        const int d = ix[k];
                        const bool v = d != 0xFFFF;
                        cp_async4(cmr + k * BTW + w, v ? a.in_cm + (size_t)d * BTW + w : a.in_cm,
                                  v ? 4u : 0u);
                    }
                }
            }
            cp_async_mbar_arrive(&raw_full[st]);
        }
        cp_async_wait<0>();
    } else if (warp == WARP_MMA) {
        // ---------------------------------------------------------- MMA issuer
        const uint32_t idesc = idesc_f16_mn(M, NP);
        const uint32_t lbo = a.desc_swap ? SBO : LBO, sbo = a.desc_swap ? LBO : SBO;
        uint64_t ad0[NOP][HALVES], bd0[NOP];
#pragma unroll
        for (int o = 0; o < NOP; ++o) {
#pragma unroll
            for (int h = 0; h < HALVES; ++h)
                ad0[o][h] = smem_desc(smem_u32(smem + SM::OFF_A + (o * HALVES + h) * SM::A_BYTES),
                                      lbo, sbo);
            bd0[o] = smem_desc(smem_u32(smem + SM::OFF_B + o * SM::B_BYTES), lbo, sbo);
        }
        constexpr uint64_t KSTEP = 2 * LBO / 16;  // start-address units per 16-row K step
        for (int j = 0; j < nj; ++j) {
            const int op = j % NOP, v = j / NOP;
            bool ok = true;
            if (lane == 0) ok = mbar_wait_bounded(&op_full[op], v & 1, a.wait_ns);
            if (!__shfl_sync(0xffffffffu, ok, 0) || *abort_flag) {
                if (lane == 0) { *abort_flag = 1; raise_error(a.err, ERRBIT_TIMEOUT); }
                break;
            }
            if (lane == 0) {
                tc_fence_after();
                const uint64_t bd = op == 0 ? bd0[0] : bd0[NOP - 1];
#pragma unroll
                for (int h = 0; h < HALVES; ++h) {
                    const uint64_t ad = op == 0 ? ad0[0][h] : ad0[NOP - 1][h];
                    const uint32_t dt = tmem + (uint32_t)(h * NP);
#pragma unroll
                    for (int kk = 0; kk < KC / 16; ++kk)
                        mma_f16(dt, ad + kk * KSTEP, bd + kk * KSTEP, idesc,
                                (j > 0 || kk > 0) ? 1u : 0u);
                }
                mma_commit(&op_empty[op]);
            }
            __syncwarp();
        }
        if (lane == 0) mma_commit(done_bar);  // fires once every issued MMA completed
    } else if (warp < NCONV) {
        // ---------------------------------------------------------- converters
        const int grp = warp / GWARPS;
        const int gtid = tid - grp * GTHREADS;  // 0 .. GTHREADS-1
        for (int j = grp; j < nj; j += NGRP) {
            const int st = j % NRAW, u = j / NRAW, op = j % NOP, v = j / NOP;
            bool ok = mbar_wait_bounded(&raw_full[st], u & 1, a.wait_ns);
            if (ok && v > 0) ok = mbar_wait_bounded(&op_empty[op], (v - 1) & 1, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok) || *abort_flag) {
                if (lane == 0) { *abort_flag = 1; raise_error(a.err, ERRBIT_TIMEOUT); }
                break;
            }
            const uint8_t* raw = smem + SM::OFF_RAW + st * SM::RAW_BYTES;
            uint8_t* A = smem + SM::OFF_A + op * HALVES * SM::A_BYTES;
            uint8_t* Bm = smem + SM::OFF_B + op * SM::B_BYTES;
            const uint32_t* cmr = cm_s + st * KC * 8;
            // raw layout: [half][row k][128 B], 16-byte pieces XOR-swizzled by (k & 7)
            constexpr int NAI = HALVES * KC * 8;               // 16-byte weight pieces
            constexpr int NA = NAI / GTHREADS;
            constexpr int NBI = (NP / 8) * KC;                 // 16-byte spike pieces
            constexpr int NB = (NBI + GTHREADS - 1) / GTHREADS;
            uint4 r[NA];
            uint32_t cw[NB];
#pragma unroll
            for (int i = 0; i < NA; ++i) {
                const int e = gtid + i * GTHREADS;
                const int k = e % KC, q = (e / KC) & 7, h = e / (KC * 8);
                r[i] = *reinterpret_cast<const uint4*>(raw + h * (KC * M) + k * 128 +
                                                       ((q ^ (k & 7)) << 4));
            }
#pragma unroll
            for (int i = 0; i < NB; ++i) {
                const int e = gtid + i * GTHREADS;
                const int k = e % KC, ng = e / KC;
                cw[i] = (e < NBI && (ng >> 2) < BTW) ? cmr[k * BTW + (ng >> 2)] : 0u;
            }
            uint4 bv[NB];
#pragma unroll
            for (int i = 0; i < NB; ++i) {
                const int e = gtid + i * GTHREADS;
                const int ng = e / KC;
                bv[i] = lut[(cw[i] >> (8 * (ng & 3))) & 0xFFu];
            }
#pragma unroll
            for (int i = 0; i < NA; ++i) {
                const int e = gtid + i * GTHREADS;
                const int k = e % KC, q = (e / KC) & 7, h = e / (KC * 8);
                uint4 f0, f1;
                i8x4_to_f16x4(r[i].x, f0.x, f0.y);
                i8x4_to_f16x4(r[i].y, f0.z, f0.w);
                i8x4_to_f16x4(r[i].z, f1.x, f1.y);
                i8x4_to_f16x4(r[i].w, f1.z, f1.w);
                uint8_t* dst = A + h * SM::A_BYTES + (2 * q) * SBO + (k >> 3) * LBO + (k & 7) * 16;
                *reinterpret_cast<uint4*>(dst) = f0;
                *reinterpret_cast<uint4*>(dst + SBO) = f1;
            }
#pragma unroll
            for (int i = 0; i < NB; ++i) {
                const int e = gtid + i * GTHREADS;
                if (e < NBI) {
                    const int k = e % KC, ng = e / KC;
                    *reinterpret_cast<uint4*>(Bm + ng * SBO + (k >> 3) * LBO + (k & 7) * 16) = bv[i];
                }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&op_full[op]);
                mbar_arrive(&raw_empty[st]);
            }
        }
    }
    NMDLM_TSTAMP(a, 1);
    __syncthreads();
    bool ok = !*abort_flag;
    if (nj > 0) {
        const bool done = mbar_wait_bounded(done_bar, 0, ok ? a.wait_ns : 1000000000ull);
        if (!done) ok = false;
    }
    const bool aborted = __syncthreads_or(!ok);
    if (aborted && tid == 0) raise_error(a.err, ERRBIT_TIMEOUT);
    NMDLM_TSTAMP(a, 2);

    // This CTA's slice of the tile after the split-K reduction: 32-channel groups
    // [g0, g1) (the whole tile without splits).
    constexpr int NGROUPS = TILE / 32;
    const int ns = a.nsplit;
    const int rank = split;  // cluster dims (1, nsplit, 1) over grid (tiles, nsplit, 1)
    const int g0 = rank * NGROUPS / ns, g1 = (rank + 1) * NGROUPS / ns, ngr = g1 - g0;
    constexpr int GROUP_BYTES = NP * 32 * 4;  // one channel group of int32 sums
    int32_t* accs = (int32_t*)smem;           // [NGROUPS][NP][32], reuses the operand rings

    // Residual currents of the slice, prefetched into the operand region past the sums
    // while the sums are staged and reduced.
    const int res_c0 = lo0 + g0 * 32;
    const int res_c1 = min(lo0 + g1 * 32, s.n_out);
    const uint32_t res_row_bytes = res_c1 > res_c0 ? (uint32_t)(res_c1 - res_c0) * 4u : 0u;
    float* res_s = (float*)(smem + SM::ACC);
    const bool res_pref = !aborted && s.res && a.kind == EPI_KIND_F32 && res_row_bytes > 0 &&
                          (((uintptr_t)s.res) & 15) == 0 &&
                          SM::ACC + (size_t)a.BT * ngr * 128 <= (size_t)SM::OFF_CM;
    if (res_pref && warp == WARP_PROD) {
        if (lane == 0) mbar_arrive_expect_tx(res_bar, (uint32_t)a.BT * res_row_bytes);
        __syncwarp();
        for (int bt = lane; bt < a.BT; bt += 32)
            bulk_load(res_s + (size_t)bt * ngr * 32, s.res + (size_t)bt * s.n_out + res_c0,
                      res_row_bytes, res_bar);
    }

    // TMEM -> shared, exact fp32 -> int32: warp w reads TMEM lanes 32 (w % 4) + lane of
    // half (w / 4) % HALVES and one share of the columns.
    if (!aborted && warp < NCONV) {
        constexpr int COMBOS = 4 * HALVES, CSPLIT = NCONV / COMBOS, NCOLS = NP / CSPLIT;
        static_assert(NCOLS % 8 == 0, "column share");
        const int combo = warp % COMBOS, cs = warp / COMBOS;
        const int q = combo & 3, h = combo >> 2;
        const int cg = h * 4 + q;
        int32_t* dst = accs + (size_t)cg * NP * 32 + lane;
        for (int cb = cs * NCOLS; cb < (cs + 1) * NCOLS; cb += 8) {
            uint32_t v[8];
            if (nj > 0) {
                tmem_ld8(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(h * NP + cb), v);
            } else {
#pragma unroll
                for (int i = 0; i < 8; ++i) v[i] = 0;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) dst[(cb + i) * 32] = __float2int_rn(__uint_as_float(v[i]));
        }
    }
    fence_proxy_async_smem();  // the sums are read by the bulk reduction (async proxy)
    tc_fence_before();
    __syncthreads();
    if (warp == WARP_MMA) tmem_dealloc(tmem, SM::NCOL);
    NMDLM_TSTAMP(a, 3);

    // Split-K: every CTA of the cluster adds its partial sums of each peer's slice into
    // that peer's shared memory with one bulk reduction per peer.
    if (ns > 1) {
        if (tid == 0) mbar_arrive_expect_tx(red_bar, (uint32_t)((ns - 1) * ngr * GROUP_BYTES));
        cluster_arrive();
        cluster_wait();  // every partial staged, every reduction barrier armed
        NMDLM_TSTAMP(a, 12);
        if (tid == 0) {
            for (int k = 1; k < ns; ++k) {
                const int qr = (rank + k) % ns;
                const int q0 = qr * NGROUPS / ns, q1 = (qr + 1) * NGROUPS / ns;
                if (q1 > q0) {
                    const uint32_t off = (uint32_t)(q0 * GROUP_BYTES);
                    bulk_reduce_add_u32_peer(mapa_shared(smem_u32(smem) + off, (uint32_t)qr),
                                             smem + off, (uint32_t)((q1 - q0) * GROUP_BYTES),
                                             mapa_shared(smem_u32(red_bar), (uint32_t)qr));
                }
            }
        }
        const bool got = mbar_wait_bounded(red_bar, 0, a.wait_ns);
        NMDLM_TSTAMP(a, 13);
        if (!got) raise_error(a.err, ERRBIT_TIMEOUT);
        ok = __syncthreads_and(got) && !aborted;
        cluster_arrive();  // nothing is added into this CTA any more; waited for at exit
    } else {
        ok = !aborted;
    }
    NMDLM_TSTAMP(a, 4);

    // Epilogue over the converter warps: (channel group, token group) pairs.
    bool res_ok = true;
    if (res_pref) res_ok = mbar_wait_bounded(res_bar, 0, a.wait_ns);
    if (!res_ok && tid == 0) raise_error(a.err, ERRBIT_TIMEOUT);
    NMDLM_TSTAMP_W(a, 0, 8);
    NMDLM_TSTAMP_W(a, 15, 10);
    if (ok && res_ok && warp < NCONV && ngr > 0) {
        // The segment's fields in registers: `s` lives in the kernel's parameter block
        // and is indexed at run time, so every read through it would be a generic load
        // that the compiler must repeat after each global store.
        const int n_out = s.n_out, T = a.T, kind = a.kind, theta_i = a.theta_i;
        const float theta_f = a.theta_f;
        const float* const g_scale = s.scale;
        const float* const g_res = s.res;
        const uint32_t* const g_gate = s.gate;
        float* const g_cur = s.cur;
        int32_t* const g_acc = s.acc_out;
        uint32_t* const g_bits = s.bits;
        const long long sb = s.sb, sst = s.st;
        const int nw = words_of(n_out);
        const int tgroups = NCONV / ngr > 0 ? NCONV / ngr : 1;
        for (int pair = warp; pair < ngr * tgroups; pair += NCONV) {
            const int cgl = pair % ngr, tg = pair / ngr;
            const int cg = g0 + cgl;
            const int m = cg * 32 + lane;
            const int lo = lo0 + m;
            const bool valid = lo < n_out;
            const bool lead = lane == 0 && (lo >> 5) < nw;
            const int b0 = tg * a.B / tgroups, b1 = (tg + 1) * a.B / tgroups;
            const int32_t* acol = accs + (size_t)cg * NP * 32 + lane;
            const float* rcol = res_s + cgl * 32 + lane;
            const int rstride = ngr * 32;
            const float sc = (valid && g_scale) ? __ldg(g_scale + lo) : 0.0f;
            bool any = false;
            if (kind == EPI_KIND_LOGITS) {
                for (int b = b0; b < b1; ++b) {
                    int sum = 0;
                    for (int t = 0; t < T; ++t) sum += acol[(b * T + t) * 32];
                    if (valid)
                        g_cur[(size_t)b * n_out + lo] = __fdiv_rn(__fmul_rn((float)sum, sc), (float)T);
                }
                continue;
            }
            for (int b = b0; b < b1; b += 4) {
                const int nt = min(4, b1 - b);
                int vi[4] = {0, 0, 0, 0};
                float vf[4] = {0.f, 0.f, 0.f, 0.f};
                uint32_t tb[4] = {0u, 0u, 0u, 0u};  // bit t: spike of token b + i at step t
                for (int t = 0; t < T; ++t) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        if (i >= nt) break;
                        const int bt = (b + i) * T + t;
                        const int acc = acol[bt * 32];
                        bool sp;
                        if (kind == EPI_KIND_INT) {
                            const int hh = vi[i] + acc;
                            sp = valid && hh >= theta_i;
                            vi[i] = sp ? hh - theta_i : hh;
                            if (valid && g_cur) g_cur[(size_t)bt * n_out + lo] = __fmul_rn((float)acc, sc);
                        } else {
                            float I = __fmul_rn((float)acc, sc);
                            if (g_res) {
                                const float r = res_pref ? rcol[bt * rstride]
                                                         : (valid ? __ldg(g_res + (size_t)bt * n_out + lo) : 0.0f);
                                I = __fadd_rn(I, valid ? r : 0.0f);
                            }
                            if (g_gate && valid) {
                                const uint32_t gw = __ldg(g_gate + (size_t)bt * nw + (lo >> 5));
                                if (!((gw >> (lo & 31)) & 1u)) I = 0.0f;
                            }
                            if (valid && g_cur) g_cur[(size_t)bt * n_out + lo] = I;
                            const float hh = __fadd_rn(vf[i], I);
                            sp = valid && hh >= theta_f;
                            vf[i] = sp ? __fsub_rn(hh, theta_f) : hh;
                        }
                        if (valid && g_acc) g_acc[(size_t)bt * n_out + lo] = acc;
                        const uint32_t word = __ballot_sync(0xffffffffu, sp);
                        // lane 0 holds the group's first channel: a group wholly past n_out
                        // writes nothing
                        if (lead) g_bits[(long long)(b + i) * sb + (long long)t * sst + (lo >> 5)] = word;
                        tb[i] |= (sp ? 1u : 0u) << t;
                    }
                }
                // column-mask bits (b + i) * T + t, t < T <= 32: at most two words per token
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    if (i >= nt || !tb[i]) continue;
                    const int start = (b + i) * T, w0 = start >> 5, sh = start & 31;
                    atomicOr(&cm_acc[m * 8 + w0], tb[i] << sh);
                    if (sh + T > 32) atomicOr(&cm_acc[m * 8 + w0 + 1], tb[i] >> (32 - sh));
                    any = true;
                }
            }
            if (any) any_acc[m] = 1;
        }
    }
    NMDLM_TSTAMP_W(a, 0, 9);
    NMDLM_TSTAMP_W(a, 15, 11);
    NMDLM_TSTAMP_W(a, 16, 14);
    NMDLM_TSTAMP_W(a, 18, 15);
    __syncthreads();
    if (ok && res_ok && warp < NCONV && a.kind != EPI_KIND_LOGITS) {
        uint32_t* const g_cm = s.cm;
        uint32_t* const g_mask = s.mask;
        const int n_out = s.n_out;
        for (int cg = g0 + warp; cg < g1; cg += NCONV) {
            const int m = cg * 32 + lane;
            const int lo = lo0 + m;
            const bool valid = lo < n_out;
            if (valid && g_cm)
                for (int w = 0; w < BTW; ++w) g_cm[(size_t)lo * BTW + w] = cm_acc[m * 8 + w];
            const uint32_t mw = __ballot_sync(0xffffffffu, valid && any_acc[m]);
            if (lane == 0 && g_mask && lo < n_out) g_mask[lo >> 5] = mw;
        }
    }
    NMDLM_TSTAMP(a, 5);
    // Peers may still be reading this CTA's partial sums for their own slices.
    if (ns > 1) cluster_wait();
    NMDLM_TSTAMP(a, 6);
}

// ------------------------------------------------------- tcgen05, TMEM A ----
// The same sums for blocks of at most 128 rows, with the operands swapped so that the
// weights pass through shared memory once:
//   A = the 0/1 spike tile, M = 128 rows bt (padded), held in tensor memory: the
//       converter warps transpose the chunk's column-mask words (32 x 32 bit blocks)
//       and store fp16 pairs with tcgen05.st -- no shared-memory operand;
//   B = W^T rows as fp16, K = 64 rows per chunk, N = 256 output channels, MN-major in
//       shared memory, read once per K step by a single N = 256 MMA;
//   D = fp32 [bt][channel] in tensor memory.
// Producers, split-K clusters and the epilogue follow k_linear_tc; the partial sums are
// staged channel-major ([channel][bt], padded) so the epilogue keeps lane = channel.
namespace tcs {
constexpr int M = 128;         // TMEM lanes = block rows (padded)
constexpr int NOP = 3;         // fp16 weight stages / TMEM spike stages
constexpr int NCONV = 16, NGRP = 2, GWARPS = NCONV / NGRP, NPROD = 2;
constexpr int WARP_PROD = NCONV, WARP_MMA = NCONV + NPROD;
constexpr int NTHREADS = (NCONV + NPROD + 1) * 32;
constexpr int GTHREADS = GWARPS * 32;
constexpr int LBO = 128;               // bytes between K-adjacent core matrices
constexpr int ACC_STRIDE = M + 1;      // words per channel row of the sums
constexpr int GROUP_BYTES = 32 * ACC_STRIDE * 4;  // one 32-channel group of sums
constexpr int NCOL = 512;
// Exact encodings: weights enter the MMA as fp16 1152 + w (the int8 byte xor 0x80 is
// the low byte of 0x64xx), spikes as fp16 2^-16 (0x0100, subnormal) or 0.  Every
// product is exact, and sum_rows (1152 + w) <= 1279 * rows < 2^24 for rows <= MAX_ROWS,
// so the fp32 accumulator holds 2^-16 * (1152 * count + sum w) exactly; the staging
// step scales by 2^16 and subtracts 1152 * count per row.
constexpr int W_BIAS = 1152;
constexpr int MAX_ROWS = 13056;        // active rows one split may own (2^24 / 1279)
constexpr int PREFETCH_CHUNKS = 8;     // weight chunks prefetched into L2 before the wait
// Chunk shape: TILE output channels (MMA N) x KC rows of W^T, 16 KB of int8 either way.
template <int TILE>
struct Cfg {
    // rows per chunk: 16 KB of int8 for TILE 128 / 256, 12 KB for TILE 192
    static constexpr int KC = TILE == 192 ? 64 : 16384 / TILE;
    // int8 stages: a stage is held from its copy's issue until the converters have read
    // it, so the ring bounds the bytes in flight per SM.  The 192 tile's paired launch
    // runs on fewer SMs than the split launches and has the shared memory for 6.
    static constexpr int NRAW = TILE == 192 ? 6 : 4;
    // TMA boxes of a chunk: 128-channel boxes with the 128-byte swizzle for TILE 128 /
    // 256; for TILE 192, whose paired halves are 96 channels wide, one unswizzled
    // 96-channel box per half (rows 96 bytes apart, so rows 4 apart share banks; the
    // converters' lane mapping keeps their reads conflict-free).  Boxes of 16 channels
    // streamed ~13 % slower: the tensor engine moves 16-byte rows at a fraction of its
    // rate for 96- or 128-byte rows.
    static constexpr int BOXW = TILE == 192 ? 96 : 128;
    static constexpr int NBOX = TILE / BOXW;
    static constexpr bool SWZ = BOXW == 128;
    static constexpr int HALF = TILE / 2;               // paired: channels of each half
    static constexpr int SBO = (KC / 8) * 128;          // bytes between 8-channel groups of B
    static constexpr int RAW_BYTES = KC * TILE;         // 16 KB
    static constexpr int B_BYTES = KC * TILE * 2;       // 32 KB
    static constexpr int CM_WORDS = KC * 4;             // column-mask words of a chunk (BT <= 128)
    static constexpr int ACOLS = KC / 2;                // TMEM columns of one spike stage
    static constexpr int OFF_RAW = 0;
    static constexpr int OFF_B = OFF_RAW + NRAW * RAW_BYTES;
    static constexpr int OFF_CM = OFF_B + NOP * B_BYTES;
    static constexpr int OFF_BAR = OFF_CM + NRAW * CM_WORDS * 4;
    static constexpr int NBAR = 2 * NRAW + 2 * NOP + 3;
    static constexpr int OFF_MISC = OFF_BAR + 8 * NBAR;
    static constexpr int OFF_CMACC = OFF_MISC + 16;            // [TILE][4] u32
    static constexpr int OFF_ANY = OFF_CMACC + TILE * 4 * 4;   // [TILE] int
    static constexpr int OFF_CNT = OFF_ANY + TILE * 4;         // [M] int: spikes per row
    static constexpr int OFF_SCL = OFF_CNT + M * 4;            // [TILE] fp32 channel scales
    static constexpr int OFF_MASK = OFF_SCL + TILE * 4;
    static constexpr int ACC_BYTES = (TILE / 32) * GROUP_BYTES;
    static_assert(ACC_BYTES <= OFF_BAR, "sums must fit below the barriers");
    static_assert(OFF_B % 1024 == 0 && RAW_BYTES % 1024 == 0, "swizzle atoms");
    static_assert(GROUP_BYTES % 16 == 0, "bulk reduction granularity");
    static_assert(TILE + NOP * ACOLS <= NCOL, "tensor memory budget");
    static constexpr int TM_D = 0;        // D: columns [0, TILE)
    static constexpr int TM_A = TILE;     // spike stages: ACOLS columns each
    static constexpr size_t bytes(int DW, int rows) {
        return (size_t)OFF_MASK + 4 * (size_t)(2 * DW + 1) + 2 * (size_t)rows + 1024;
    }
};
}  // namespace tcs

// IF epilogue of one warp: lane = output channel lo, tokens [b0, b1), T steps each.
// acol[bt] is the exact sum of row bt.  Specialised at compile time on the current's
// kind and sources, so the loop body is straight-line code: the run-time flags are
// warp-uniform, but each branch on them costs a branch resolution per element.
struct EpiWarp {
    const int32_t* acol;     // sums of this lane's channel, indexed by bt
    const float* rcol;       // residual of this lane's channel in shared memory (RES_SMEM)
    int rstride;             // words between consecutive bt in rcol
    const float* g_res;      // residual in global memory (RES_GLOBAL)
    const uint32_t* g_gate;  // gate row bits
    float* g_cur;            // current out
    uint32_t* g_bits;        // row-bit destination
    long long sb, sst;       // word strides of token b and step t in g_bits
    int n_out, nw, lo, T;
    float sc, theta_f;
    int theta_i;
    bool valid, lead;
    bool lead_word;          // this warp's channel group has a row-bit word (lo / 32 < nw)
    unsigned long long* dbg; // debug: per-token timestamps of one warp, or null
};
enum { EPI_RES_NONE = 0, EPI_RES_SMEM = 1, EPI_RES_GLOBAL = 2 };


// Rows are taken in order in windows of 32 (the rows of one column-mask word).  A lane
// (one channel) collects its spikes over the window as the bits of one word, which is
// the channel's column-mask word; at the window's end one 32 x 32 bit transpose across
// the warp turns the 32 channels' words into the 32 rows' row-bit words, and lane j
// stores the word of the window's row j.
template <int TT>
__device__ __forceinline__ void epi_flush(const EpiWarp& e, uint32_t bits, uint32_t gbits_w,
                                          int wbase, int r0, int r1, uint32_t* cmrow,
                                          uint32_t* gdst, long long gsb, long long gsst,
                                          bool& any) {
    const int lane = threadIdx.x & 31;
    const int T = TT ? TT : e.T;
    const uint32_t word = warp_transpose32(bits);
    const uint32_t gword = gdst ? warp_transpose32(gbits_w) : 0u;
    const int row = wbase + lane;
    if (e.lead_word && row >= r0 && row < r1) {
        const int b = row / T, t = row - b * T;
        e.g_bits[(long long)b * e.sb + (long long)t * e.sst + (e.lo >> 5)] = word;
        if (gdst) gdst[(long long)b * gsb + (long long)t * gsst + (e.lo >> 5)] = gword;
    }
    if (bits) {
        atomicOr(&cmrow[wbase >> 5], bits);
        any = true;
    }
}

// IF epilogue of one warp: lane = output channel e.lo, the rows of tokens [b0, b1) in
// order, T steps per token with the membrane reset at each token (TT: T known at compile
// time, 32 % TT == 0, else 0).  acol[bt] is the exact sum of row bt.  Specialised at
// compile time on the current's kind and sources.  Returns whether the channel fired.
template <int TT, bool F32, int RESM, bool GATE, bool CUR>
__device__ __forceinline__ bool epi_rows(const EpiWarp& e, int b0, int b1, uint32_t* cmrow) {
    const int T = TT ? TT : e.T;
    const int r0 = b0 * T, r1 = b1 * T;
    bool any = false;
    uint32_t bits = 0u;
    int wbase = r0 & ~31;
    float* cur = CUR ? e.g_cur + (size_t)r0 * e.n_out + e.lo : nullptr;
    if (e.dbg && (threadIdx.x & 31) == 0) e.dbg[40] = clock64();
    for (int b = b0; b < b1; ++b) {
        if (e.dbg && (threadIdx.x & 31) == 0 && b - b0 < 8) e.dbg[41 + b - b0] = clock64();
        int vi = 0;
        float vf = 0.0f;
#pragma unroll(TT ? TT : 1)
        for (int t = 0; t < T; ++t) {
            const int bt = b * T + t;
            if (!TT && bt - wbase == 32) {
                epi_flush<TT>(e, bits, 0u, wbase, r0, r1, cmrow, nullptr, 0, 0, any);
                bits = 0u;
                wbase += 32;
            }
            const int acc = e.acol[bt];
            bool sp;
            if constexpr (!F32) {
                const int hh = vi + acc;
                sp = e.valid && hh >= e.theta_i;
                vi = sp ? hh - e.theta_i : hh;
            } else {
                float I = __fmul_rn((float)acc, e.sc);
                if constexpr (RESM == EPI_RES_SMEM) I = __fadd_rn(I, e.valid ? e.rcol[bt * e.rstride] : 0.0f);
                if constexpr (RESM == EPI_RES_GLOBAL)
                    I = __fadd_rn(I, e.valid ? __ldg(e.g_res + (size_t)bt * e.n_out + e.lo) : 0.0f);
                if constexpr (GATE) {
                    const uint32_t gw = e.valid ? __ldg(e.g_gate + (size_t)bt * e.nw + (e.lo >> 5)) : 0u;
                    I = ((gw >> (e.lo & 31)) & 1u) ? I : 0.0f;
                }
                if constexpr (CUR) {
                    if (e.valid) *cur = I;
                    cur += e.n_out;
                }
                const float hh = __fadd_rn(vf, I);
                sp = e.valid && hh >= e.theta_f;
                vf = sp ? __fsub_rn(hh, e.theta_f) : hh;
            }
            bits |= sp ? (1u << (bt - wbase)) : 0u;
        }
        if (TT && ((b + 1) * T & 31) == 0) {
            epi_flush<TT>(e, bits, 0u, wbase, r0, r1, cmrow, nullptr, 0, 0, any);
            bits = 0u;
            wbase += 32;
        }
    }
    if (r1 > wbase) epi_flush<TT>(e, bits, 0u, wbase, r0, r1, cmrow, nullptr, 0, 0, any);
    return any;
}

// Gated MLP epilogue of one warp (lane = channel lo), tokens [b0, b1): per step the
// gate's IF runs on fp32(acc_gate) * gate_scale, and the up projection's IF on the current
// fp32(acc_up) * scale passed only where the gate fired at that step (reading: the down
// projection's input current is gate spike * I_up).  Gate spikes go to gdst when given;
// the up spikes follow e.g_bits / column masks as in epi_rows.
template <int TT, bool CUR>
__device__ __forceinline__ bool epi_gated_rows(const EpiWarp& e, const int32_t* gcol, float gsc,
                                               uint32_t* gdst, long long gsb, long long gsst,
                                               int b0, int b1, uint32_t* cmrow) {
    const int T = TT ? TT : e.T;
    const int r0 = b0 * T, r1 = b1 * T;
    bool any = false;
    uint32_t bits = 0u, gb = 0u;
    int wbase = r0 & ~31;
    float* cur = CUR ? e.g_cur + (size_t)r0 * e.n_out + e.lo : nullptr;
    if (e.dbg && (threadIdx.x & 31) == 0) e.dbg[50] = clock64();
    for (int b = b0; b < b1; ++b) {
        if (e.dbg && (threadIdx.x & 31) == 0 && b - b0 < 8) e.dbg[51 + b - b0] = clock64();
        float vg = 0.0f, vu = 0.0f;
#pragma unroll(TT ? TT : 1)
        for (int t = 0; t < T; ++t) {
            const int bt = b * T + t;
            if (!TT && bt - wbase == 32) {
                epi_flush<TT>(e, bits, gb, wbase, r0, r1, cmrow, gdst, gsb, gsst, any);
                bits = gb = 0u;
                wbase += 32;
            }
            const float ig = __fmul_rn((float)gcol[bt], gsc);
            const float hg = __fadd_rn(vg, ig);
            const bool sg = e.valid && hg >= e.theta_f;
            vg = sg ? __fsub_rn(hg, e.theta_f) : hg;
            const float iu = sg ? __fmul_rn((float)e.acol[bt], e.sc) : 0.0f;
            if constexpr (CUR) {
                if (e.valid) *cur = iu;
                cur += e.n_out;
            }
            const float hu = __fadd_rn(vu, iu);
            const bool sp = e.valid && hu >= e.theta_f;
            vu = sp ? __fsub_rn(hu, e.theta_f) : hu;
            const uint32_t m = 1u << (bt - wbase);
            gb |= sg ? m : 0u;
            bits |= sp ? m : 0u;
        }
        if (TT && ((b + 1) * T & 31) == 0) {
            epi_flush<TT>(e, bits, gb, wbase, r0, r1, cmrow, gdst, gsb, gsst, any);
            bits = gb = 0u;
            wbase += 32;
        }
    }
    if (r1 > wbase) epi_flush<TT>(e, bits, gb, wbase, r0, r1, cmrow, gdst, gsb, gsst, any);
    return any;
}

__device__ __forceinline__ bool epi_gated_run(const EpiWarp& e, const int32_t* gcol, float gsc,
                                              uint32_t* gdst, long long gsb, long long gsst,
                                              int b0, int b1, uint32_t* cmrow) {
    if (e.T == 4)
        return e.g_cur ? epi_gated_rows<4, true>(e, gcol, gsc, gdst, gsb, gsst, b0, b1, cmrow)
                       : epi_gated_rows<4, false>(e, gcol, gsc, gdst, gsb, gsst, b0, b1, cmrow);
    return e.g_cur ? epi_gated_rows<0, true>(e, gcol, gsc, gdst, gsb, gsst, b0, b1, cmrow)
                   : epi_gated_rows<0, false>(e, gcol, gsc, gdst, gsb, gsst, b0, b1, cmrow);
}

template <int TT>
__device__ __forceinline__ bool epi_dispatch_t(const EpiWarp& e, bool f32, int resm, int b0, int b1,
                                               uint32_t* cmrow) {
    if (!f32) return epi_rows<TT, false, EPI_RES_NONE, false, false>(e, b0, b1, cmrow);
    const bool gate = e.g_gate != nullptr, cur = e.g_cur != nullptr;
#define NMDLM_EPI_CASE(R)                                                                   \
    if (resm == R) {                                                                        \
        if (gate) return cur ? epi_rows<TT, true, R, true, true>(e, b0, b1, cmrow)          \
                             : epi_rows<TT, true, R, true, false>(e, b0, b1, cmrow);        \
        return cur ? epi_rows<TT, true, R, false, true>(e, b0, b1, cmrow)                   \
                   : epi_rows<TT, true, R, false, false>(e, b0, b1, cmrow);                 \
    }
    NMDLM_EPI_CASE(EPI_RES_NONE)
    NMDLM_EPI_CASE(EPI_RES_SMEM)
    NMDLM_EPI_CASE(EPI_RES_GLOBAL)
#undef NMDLM_EPI_CASE
    return false;
}

__device__ __forceinline__ bool epi_dispatch(const EpiWarp& e, bool f32, int resm, int b0, int b1,
                                             uint32_t* cmrow) {
    return e.T == 4 ? epi_dispatch_t<4>(e, f32, resm, b0, b1, cmrow)
                    : epi_dispatch_t<0>(e, f32, resm, b0, b1, cmrow);
}

template <int TILE>
__global__ void __launch_bounds__(tcs::NTHREADS, 1) k_linear_ts(const __grid_constant__ LinArgs a) {
    using namespace tcs;
    using C = Cfg<TILE>;
    constexpr int KC = C::KC, SBO = C::SBO, RAW_BYTES = C::RAW_BYTES, NRAW = C::NRAW;
    constexpr int BOXW = C::BOXW, NBOX = C::NBOX, HALF = C::HALF;
    constexpr bool SWZ = C::SWZ;
    constexpr int B_BYTES = C::B_BYTES, CM_WORDS = C::CM_WORDS, ACC_BYTES = C::ACC_BYTES;
    constexpr int OFF_RAW = C::OFF_RAW, OFF_B = C::OFF_B, OFF_CM = C::OFF_CM;
    constexpr int OFF_BAR = C::OFF_BAR, OFF_MISC = C::OFF_MISC, OFF_CMACC = C::OFF_CMACC;
    constexpr int OFF_ANY = C::OFF_ANY, OFF_MASK = C::OFF_MASK, TM_D = C::TM_D, TM_A = C::TM_A;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint32_t* cm_s = (uint32_t*)(smem + OFF_CM);
    uint64_t* raw_full = (uint64_t*)(smem + OFF_BAR);
    uint64_t* raw_empty = raw_full + NRAW;
    uint64_t* op_full = raw_empty + NRAW;
    uint64_t* op_empty = op_full + NOP;
    uint64_t* done_bar = op_empty + NOP;
    uint64_t* red_bar = done_bar + 1;
    uint64_t* res_bar = done_bar + 2;
    uint32_t* tmem_holder = (uint32_t*)(smem + OFF_MISC);
    volatile int* abort_flag = (volatile int*)(smem + OFF_MISC + 4);
    uint32_t* cm_acc = (uint32_t*)(smem + OFF_CMACC);
    int* any_acc = (int*)(smem + OFF_ANY);
    int* cnt_s = (int*)(smem + C::OFF_CNT);
    const int DW = words_of(a.d_in);
    uint32_t* mask_s = (uint32_t*)(smem + OFF_MASK);
    int* prefix = (int*)(mask_s + DW);
    uint16_t* rowlist = (uint16_t*)(prefix + DW + 1);

    NMDLM_CSTAMP(a, 256, 0);
    const int tile = blockIdx.x, split = blockIdx.y;
    // Paired (gated MLP, TILE 256 or 192): half 0 of every chunk holds HALF channels of
    // the gate weights and half 1 the same HALF channels of the up weights; seg[1] (up)
    // owns the outputs.  Otherwise the tile's segment supplies every box.
    const bool paired = (TILE == 256 || TILE == 192) && a.paired;
    const int si = paired ? 1 : seg_of_tile(a, tile);
    // The tile's segment, copied once into shared memory: read through a run-time
    // index, the parameter block is reached by generic loads of ~1 k cycles each.
    __shared__ LinSeg seg_s;
    if (threadIdx.x == 0) {
        seg_s = si == 0 ? a.seg[0] : (si == 1 ? a.seg[1] : a.seg[2]);
    }
    __syncthreads();
    const LinSeg& s = seg_s;
    const CUtensorMap* tmap = si == 0 ? &a.tmap[0] : (si == 1 ? &a.tmap[1] : &a.tmap[2]);
    const CUtensorMap* gmap = si == 0 ? &a.gmap[0] : (si == 1 ? &a.gmap[1] : &a.gmap[2]);
    const int lo0 = paired ? tile * HALF : (tile - s.tile_begin) * TILE;
    // tensor map and first channel of box b of a chunk (paired: boxes [0, NBOX / 2) are
    // the gate half, the rest the up half)
    auto box_half = [&](int b) { return paired ? b / (NBOX / 2) : 0; };
    auto half_map = [&](int b) { return paired ? &a.tmap[box_half(b)] : tmap; };
    auto half_gmap = [&](int b) { return paired ? &a.gmap[box_half(b)] : gmap; };
    auto half_x = [&](int b) { return lo0 + (paired ? b % (NBOX / 2) : b) * BOXW; };
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int BTW = a.BTW;  // <= 4

    // Setup that touches nothing another kernel writes, done before waiting for the
    // previous kernel: shared-memory state, barriers, tensor memory, and an L2
    // prefetch of this split's first weight chunks in dense row order (the common
    // case at these block sizes; a sparse block merely wastes the prefetch).
    for (int i = tid; i < TILE * 4; i += NTHREADS) cm_acc[i] = 0;
    for (int i = tid; i < TILE; i += NTHREADS) any_acc[i] = 0;
    for (int i = tid; i < M; i += NTHREADS) cnt_s[i] = 0;
    {
        // the tile's output-channel scales (paired: the up half, then the gate half), read
        // before the dependency wait: weights, not results
        float* scl = (float*)(smem + C::OFF_SCL);
        const float* up_sc = paired ? a.seg[1].scale : s.scale;
        const float* gate_sc = paired ? a.seg[0].scale : nullptr;
        for (int i = tid; i < TILE; i += NTHREADS) {
            const bool gate_half = paired && i >= HALF;
            const int ch = lo0 + (gate_half ? i - HALF : i);
            const float* src = gate_half ? gate_sc : up_sc;
            scl[i] = (src && ch < s.n_out) ? __ldg(src + ch) : 0.0f;
        }
    }
    if (tid == 0) {
        *abort_flag = 0;
        for (int i = 0; i < NRAW; ++i) {
            mbar_init(&raw_full[i], 1 + 32);  // producer's expect_tx + 32 cp.async arrivals
            mbar_init(&raw_empty[i], GWARPS);
        }
        for (int i = 0; i < NOP; ++i) {
            mbar_init(&op_full[i], GWARPS);
            mbar_init(&op_empty[i], 1);
        }
        mbar_init(done_bar, 1);
        // cluster mode: split-K exchange (red_bar) and residual prefetch (res_bar)
        mbar_init(red_bar, 1);
        mbar_init(res_bar, 32);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == WARP_MMA) {
        tmem_alloc(tmem_holder, NCOL);
        tmem_relinquish();
    }
    if (warp == WARP_PROD) {
        const int nch_d = (a.d_in + KC - 1) / KC;
        const int c0d = split * nch_d / a.nsplit, c1d = (split + 1) * nch_d / a.nsplit;
        for (int jj = 0; jj < min(PREFETCH_CHUNKS, c1d - c0d); ++jj)
            if (lane < NBOX) tma_prefetch_2d(half_map(lane), half_x(lane), (c0d + jj) * KC);
    }
    pdl_wait();
    NMDLM_TSTAMP(a, 7);
    NMDLM_CSTAMP(a, 256, 1);
    // AUTO: when most rows are active, stream every row in order -- contiguous chunks
    // load as whole TMA tiles, and an inactive row only multiplies zero spikes.  A
    // sparser block gathers its active rows only (row skipping, Sec. IV-A).  One warp
    // counts the active rows; the prefix sums and the row list are built only to gather.
    __shared__ int nact_s;
    if (warp == 0) {
        int c = 0;
        if (a.dense) {
            c = a.d_in;
        } else {
            for (int w = lane; w < DW; w += 32) c += __popc(__ldg(a.in_mask + w));
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
        }
        if (lane == 0) nact_s = c;
    }
    __syncthreads();
    NMDLM_TSTAMP(a, 20);
    const int n_counted = nact_s;
    const bool all_rows = a.dense || (a.auto_dense && n_counted * 4 >= a.d_in) ||
                          n_counted == a.d_in;
    const int n_active = all_rows ? a.d_in : n_counted;
    const int nch = (n_active + KC - 1) / KC;
    const int c0 = split * nch / a.nsplit, c1 = (split + 1) * nch / a.nsplit;
    const int nj = c1 - c0;
    const int r0 = c0 * KC, nrows = nj * KC;
    if (!all_rows) {
        // this split's compacted rows [r0, r0 + nrows) in ascending order, 0xFFFF past the
        // last active row
        active_prefix(false, a.d_in, a.in_mask, mask_s, prefix, DW);
        for (int i = tid; i < nrows; i += NTHREADS) rowlist[i] = 0xFFFFu;
        __syncthreads();
        for (int w = tid; w < DW; w += NTHREADS) {
            uint32_t m = mask_s[w];
            int pos = prefix[w];
            if (pos >= r0 + nrows || prefix[w + 1] <= r0) continue;
            while (m) {
                const int bit = __ffs(m) - 1;
                m &= m - 1;
                if (pos >= r0 && pos < r0 + nrows) rowlist[pos - r0] = (uint16_t)(w * 32 + bit);
                ++pos;
            }
        }
    }
    NMDLM_TSTAMP(a, 21);
    // input channel (row of W^T) k of chunk j, 0xFFFF past the end
    auto row_of = [&](int j, int k) -> int {
        if (all_rows) {
            const int r = (c0 + j) * KC + k;
            return r < a.d_in ? r : 0xFFFF;
        }
        return rowlist[j * KC + k];
    };
    NMDLM_TSTAMP(a, 22);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    NMDLM_TSTAMP(a, 0);

    if (warp >= WARP_PROD && warp < WARP_PROD + NPROD) {
        // ---------------------------------------------------------- producers
        const int p = warp - WARP_PROD;
        const int8_t* const gw0 = paired ? a.seg[0].wT : s.wT;  // constant-index reads
        const int8_t* const gw1 = paired ? a.seg[1].wT : s.wT;
        const int gld0 = paired ? a.seg[0].ld_w : s.ld_w;
        const int gld1 = paired ? a.seg[1].ld_w : s.ld_w;
        const int gn0 = paired ? a.seg[0].n_out : s.n_out;
        const int gn1 = paired ? a.seg[1].n_out : s.n_out;
        // the weights pass through L2 once per launch: first to be evicted, so that
        // what is reused (code, activations, partial sums, the K/V caches) stays
        const uint64_t wpol = l2_policy_evict_first();
        for (int j = p; j < nj; j += NPROD) {
            const int st = j % NRAW, u = j / NRAW;
            if (u > 0) {
                const bool ok = mbar_wait_bounded(&raw_empty[st], (u - 1) & 1, a.wait_ns);
                if (!__all_sync(0xffffffffu, ok) || *abort_flag) {
                    if (lane == 0) { *abort_flag = 1; raise_error(a.err, ERRBIT_TIMEOUT); }
                    break;
                }
            }
            const int row0 = row_of(j, 0);
            const bool contiguous = row0 != 0xFFFF && row_of(j, KC - 1) == row0 + KC - 1;
            uint8_t* raw = smem + OFF_RAW + st * RAW_BYTES;
            uint32_t* cmr = cm_s + st * CM_WORDS;
            const uint32_t cm_bytes = KC * BTW * 4;
            const bool cm_bulk = contiguous && ((((size_t)row0 * BTW * 4) & 15) == 0) &&
                                 ((((uintptr_t)a.in_cm) & 15) == 0);
            // weight bytes the tensor engine delivers (the 16-channel gather below uses
            // cp.async, counted by the lanes' arrivals instead)
            const uint32_t tma_bytes = (contiguous || SWZ) ? (uint32_t)RAW_BYTES : 0u;
            if (lane == 0)
                mbar_arrive_expect_tx(&raw_full[st], tma_bytes + (cm_bulk ? cm_bytes : 0u));
            __syncwarp();
            if (contiguous) {
                if (lane < NBOX)
                    tma_load_2d_hint(raw + lane * (KC * BOXW), half_map(lane), half_x(lane), row0,
                                     &raw_full[st], wpol);
            } else if (SWZ) {
                if (lane < NBOX * (KC / 4)) {
                    const int h = lane / (KC / 4), g = lane % (KC / 4);
                    int rr[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int d = row_of(j, 4 * g + q);
                        rr[q] = d == 0xFFFF ? a.d_in : d;  // out of range: zero fill
                    }
                    tcl::tma_gather4(raw + h * (KC * 128) + g * 4 * 128, half_gmap(h), half_x(h),
                                     rr[0], rr[1], rr[2], rr[3], &raw_full[st]);
                }
            } else {
                // unswizzled boxes: one 16-byte cp.async per (row, piece), zero past the end
                constexpr int PPB = BOXW / 16;
                for (int i = lane; i < NBOX * PPB * KC; i += 32) {
                    const int k = i % KC, pc = i / KC, b = pc / PPB, q = pc % PPB;
                    const int d = row_of(j, k);
                    const int h = box_half(b);
                    const int8_t* w = h ? gw1 : gw0;
                    const size_t ld = h ? (size_t)gld1 : (size_t)gld0;
                    const int x = half_x(b) + q * 16;
                    // n_out is a multiple of 16: a piece is wholly inside or past the end
                    const bool v = d != 0xFFFF && x < (h ? gn1 : gn0);
                    cp_async16(raw + b * (KC * BOXW) + k * BOXW + q * 16,
                               v ? w + (size_t)d * ld + x : w, v ? 16u : 0u);
                }
            }
            if (cm_bulk) {
                if (lane == 0) bulk_load(cmr, a.in_cm + (size_t)row0 * BTW, cm_bytes, &raw_full[st]);
            } else {
                for (int k = lane >> 2; k < KC; k += 8) {
                    const int w = lane & 3;
                    if (w < BTW) {
                        const int d = row_of(j, k);
                        const bool v = d != 0xFFFF;
                        cp_async4(cmr + k * BTW + w, v ? a.in_cm + (size_t)d * BTW + w : a.in_cm,
                                  v ? 4u : 0u);
                    }
                }
            }
            cp_async_mbar_arrive(&raw_full[st]);
        }
        cp_async_wait<0>();
    } else if (warp == WARP_MMA) {
        // ---------------------------------------------------------- MMA issuer
        // One thread runs the loop, with the stage and parity counted rather than
        // divided out and no warp-wide step per chunk.  The tensor pipe queues few MMAs
        // and a barrier query is a round trip to shared memory, so a query between two
        // chunks leaves the pipe idle for that long: chunk j + 1's readiness is asked
        // (without suspending) before chunk j's MMAs and read after them.
        if (lane == 0) {
            const uint32_t idesc = idesc_f16_tmemA_mnB(M, TILE);
            // stage o's descriptor: the start-address field (bytes / 16) advanced by o * B_BYTES
            const uint64_t bd_base = smem_desc(smem_u32(smem + OFF_B), LBO, SBO);
            constexpr uint64_t KSTEP = 2 * LBO / 16;  // descriptor units per 16-row K step
            const uint32_t td = tmem + TM_D;
            int op = 0;
            uint32_t ph = 0;
            bool ready = false;  // chunk j's operands known to be staged
            for (int j = 0; j < nj; ++j) {
                if (!ready && !mbar_try_wait(&op_full[op], ph) &&
                    (*abort_flag || !mbar_wait_bounded(&op_full[op], ph, a.wait_ns))) {
                    *abort_flag = 1;
                    raise_error(a.err, ERRBIT_TIMEOUT);
                    break;
                }
                tc_fence_after();
                const int op1 = op + 1 == NOP ? 0 : op + 1;
                ready = j + 1 < nj && mbar_test_wait(&op_full[op1], op1 == 0 ? ph ^ 1u : ph);
                const uint64_t bd = bd_base + (uint64_t)(op * (B_BYTES >> 4));
                const uint32_t ta = tmem + (uint32_t)(TM_A + op * C::ACOLS);
#pragma unroll
                for (int kk = 0; kk < KC / 16; ++kk)
                    mma_f16_ts(td, ta + kk * 8, bd + kk * KSTEP, idesc, (j > 0 || kk > 0) ? 1u : 0u);
                mma_commit(&op_empty[op]);
                if (++op == NOP) { op = 0; ph ^= 1; }
            }
            mma_commit(done_bar);
        }
        __syncwarp();
    } else if (warp < NCONV) {
        // ---------------------------------------------------------- converters
        const int grp = warp / GWARPS, gw = warp % GWARPS;
        const int gtid = tid - grp * GTHREADS;
        const int q = gw & 3, khalf = gw >> 2;  // TMEM lane quarter (= warp % 4), half of K
        int cnt = 0;                             // spikes of row 32 q + lane in this warp's rows
        // rows in order (dense stream) and the block's row bits given: no transpose needed
        const bool use_rows = a.in_rows != nullptr && (all_rows || n_active == a.d_in);
        const int row_words = words_of(a.d_in);
        // Rows in order: this lane's row-bit words of a chunk (32 rows of K each), loaded
        // one chunk of the group ahead so that their L2 latency is off the chain
        // (spikes -> TMEM, weights -> fp16 stage -> operands staged) that sets the rate.
        auto load_rw = [&](int jj, uint32_t (&dst)[KC / 64]) {
            const int bt = q * 32 + lane;
#pragma unroll
            for (int sl = 0; sl < KC / 64; ++sl) {
                const int w = ((c0 + jj) * KC + khalf * (KC / 2) + sl * 32) >> 5;
                dst[sl] = (use_rows && jj < nj && bt < a.BT && w < row_words)
                              ? __ldg(a.in_rows + (size_t)bt * row_words + w) : 0u;
            }
        };
        uint32_t rw_next[KC / 64];
        load_rw(grp, rw_next);
        for (int j = grp; j < nj; j += NGRP) {
            const int st = j % NRAW, u = j / NRAW, op = j % NOP, v = j / NOP;
            uint32_t rw[KC / 64];
#pragma unroll
            for (int sl = 0; sl < KC / 64; ++sl) rw[sl] = rw_next[sl];
            load_rw(j + NGRP, rw_next);
            bool ok = mbar_wait_bounded(&raw_full[st], u & 1, a.wait_ns);
            if (ok && v > 0) ok = mbar_wait_bounded(&op_empty[op], (v - 1) & 1, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok) || *abort_flag) {
                if (lane == 0) { *abort_flag = 1; raise_error(a.err, ERRBIT_TIMEOUT); }
                break;
            }
            tc_fence_after();
            const uint8_t* raw = smem + OFF_RAW + st * RAW_BYTES;
            uint8_t* Bw = smem + OFF_B + op * B_BYTES;
            const uint32_t* cmr = cm_s + st * CM_WORDS;
            // spikes into the stage's TMEM columns as fp16 pairs of 2^-16 / 0, lane = row
            // bt = 32 q + lane holding its 32 bits over k: read from the row bits when the
            // rows are in order, else transposed from the chunk's column-mask words.
#pragma unroll
            for (int sl = 0; sl < KC / 64; ++sl) {
                const int k0 = khalf * (KC / 2) + sl * 32;
                const uint32_t xb =
                    use_rows ? rw[sl] : warp_transpose32(q < BTW ? cmr[(k0 + lane) * BTW + q] : 0u);
                cnt += __popc(xb);
                uint32_t av[16];
                bits_to_e16_pairs(xb, av);
                tmem_st16(tmem + ((uint32_t)(q * 32) << 16) +
                              (uint32_t)(TM_A + op * C::ACOLS + (k0 >> 1)), av);
            }
            // weights: int8 -> fp16, MN-major core matrices (8 channels x 16 bytes).  The
            // int8 stage is handed back to the producers as soon as its bytes are
            // converted in registers, before the fp16 stores: the stage's round trip
            // (HBM load, conversion, refill) bounds the chunk rate with 4 stages.
            constexpr int NAI = (TILE / 16) * KC;  // 16-byte weight pieces
            constexpr int NA = NAI / GTHREADS;
            // element e -> (row k, 16-channel piece pc).  Swizzled boxes: lanes take
            // consecutive rows of one piece.  Unswizzled 96-byte rows (the 192 tile): rows
            // 4 apart fall on the same banks, so each group of 8 lanes takes 8 consecutive
            // rows over a pair of pieces, the first 4 rows one piece and the last 4 the
            // other (and a second group the swap): its 16-byte reads land on 8 distinct
            // bank quads, and its stores on the two halves of a 128-byte row of core
            // matrices.
            auto piece_of = [&](int e, int& k, int& pc) {
                if constexpr (SWZ) {
                    k = e % KC;
                    pc = e / KC;
                } else {
                    constexpr int R8 = KC / 8, NPP = TILE / 32;
                    static_assert(NAI == 8 * R8 * NPP * 2 && (BOXW / 16) % 2 == 0,
                                  "octets of rows x piece pairs x two orders");
                    const int o = e >> 3, l = e & 7;
                    const int pp = (o / R8) % NPP, v = o / (R8 * NPP);
                    k = (o % R8) * 8 + l;
                    pc = 2 * pp + (((l >> 2) ^ v) & 1);
                }
            };
            uint4 f[2 * NA];
#pragma unroll
            for (int i = 0; i < NA; ++i) {
                const int e = gtid + i * GTHREADS;
                int k, pc;  // row, 16-channel piece
                piece_of(e, k, pc);
                constexpr int PPB = BOXW / 16;  // 16-byte pieces per box row
                const uint4 r = *reinterpret_cast<const uint4*>(
                    SWZ ? raw + (pc >> 3) * (KC * 128) + k * 128 + (((pc & 7) ^ (k & 7)) << 4)
                        : raw + (pc / PPB) * (KC * BOXW) + k * BOXW + (pc % PPB) * 16);
                i8x4_to_f16x4_biased(r.x, f[2 * i].x, f[2 * i].y);
                i8x4_to_f16x4_biased(r.y, f[2 * i].z, f[2 * i].w);
                i8x4_to_f16x4_biased(r.z, f[2 * i + 1].x, f[2 * i + 1].y);
                i8x4_to_f16x4_biased(r.w, f[2 * i + 1].z, f[2 * i + 1].w);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&raw_empty[st]);
#pragma unroll
            for (int i = 0; i < NA; ++i) {
                const int e = gtid + i * GTHREADS;
                int k, pc;
                piece_of(e, k, pc);
                uint8_t* dst = Bw + (2 * pc) * SBO + (k >> 3) * LBO + (k & 7) * 16;
                *reinterpret_cast<uint4*>(dst) = f[2 * i];
                *reinterpret_cast<uint4*>(dst + SBO) = f[2 * i + 1];
            }
            tmem_wait_st();
            fence_proxy_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&op_full[op]);
        }
        if (cnt) atomicAdd(&cnt_s[q * 32 + lane], cnt);
    }
    NMDLM_TSTAMP(a, 1);
    __syncthreads();
    bool ok = !*abort_flag;
    if (nj > 0) {
        const bool done = mbar_wait_bounded(done_bar, 0, ok ? a.wait_ns : 1000000000ull);
        if (!done) ok = false;
    }
    const bool aborted = __syncthreads_or(!ok);
    if (aborted && tid == 0) raise_error(a.err, ERRBIT_TIMEOUT);
    tc_fence_after();
    NMDLM_TSTAMP(a, 2);
    NMDLM_CSTAMP(a, 256, 2);

    const bool sync_slots = a.slot_mode && a.slot_sync;
    // The epilogue kernel that follows a slot launch may be scheduled onto the SMs this
    // launch frees as its CTAs exit (it waits for the whole grid before reading).
    if (a.slot_mode && !sync_slots) pdl_trigger();
    if (a.slot_mode) {
        // Partial sums of this split into its slot of the launch's L2-resident partials,
        // straight from tensor memory: lane = row bt holds 32 channels, and for each
        // channel the warp's 32 lanes store 32 consecutive words of the channel-major
        // slot ([channel][BTP]).  (Bulk adds into one shared accumulator were slower:
        // every element then took ns atomic adds at L2.)  The slots are summed (integer
        // addition is exact and order-free) either below, each split taking one slice of
        // the tile once every split of the tile has stored, or by k_linear_epi.
        const int BTP = a.btp;
        if (!aborted && warp < NCONV) {
            const int q = warp & 3, cs = warp >> 2;
            const int bt = q * 32 + lane;
            int32_t* const slot = a.acc_g + (size_t)split * a.acc_stride;
            const int scol0 = paired ? a.seg[0].col0 : s.col0;  // constant-index reads
            const int scol1 = paired ? a.seg[1].col0 : s.col0;
            if (q * 32 < BTP) {
                const int bias = W_BIAS * cnt_s[bt];
#pragma unroll 1
                for (int cb = cs * 32; cb < TILE; cb += 128) {
                    // column group -> accumulator columns (paired: gate half, up half)
                    const int half = paired ? cb / HALF : 0;
                    const int ch = paired ? cb % HALF : cb;
                    const int col0 = half ? scol1 : scol0;
                    const int nc = min(32, s.n_out - (lo0 + ch));
                    if (nc <= 0) continue;
                    uint32_t v[32];
                    if (nj > 0) {
                        tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(TM_D + cb), v);
                    } else {  // no chunk: the slot still takes this split's zeros
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = 0u;
                    }
                    int32_t* dst = slot + (size_t)(col0 + lo0 + ch) * BTP + bt;
                    if (bt < BTP)
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (i < nc)
                                dst[(size_t)i * BTP] =
                                    __float2int_rn(__fmul_rn(__uint_as_float(v[i]), 65536.0f)) - bias;
                }
            }
        }
        if (!sync_slots) {
            // the output mask words are ORed by k_linear_epi: the tile's split 0 clears them
            if (a.kind != EPI_KIND_LOGITS) {
                const int wpt = paired ? HALF / 32 : TILE / 32;  // mask words per tile
                if (split == 0 && tid < wpt && s.mask && lo0 + tid * 32 < s.n_out)
                    s.mask[(lo0 + tid * 32) >> 5] = 0u;
            }
            tc_fence_before();
            __syncthreads();
            if (warp == WARP_MMA) tmem_dealloc(tmem, NCOL);
            NMDLM_TSTAMP(a, 6);
            NMDLM_CSTAMP(a, 256, 3);
            return;
        }
        // Every split of the tile stores before any sums: one arrival per CTA, released
        // by a fence after its stores; every CTA of the launch is resident at once (one
        // per SM, at most one wave), and the wait is bounded all the same.
        tc_fence_before();
        __threadfence();
        __syncthreads();
        if (warp == WARP_MMA) tmem_dealloc(tmem, NCOL);
        if (tid == 0) {
            unsigned* const tk = a.tickets + 2 * tile;
            atomicAdd(&tk[0], 1u);
            if (!wait_count_bounded(&tk[0], (unsigned)a.nsplit, a.wait_ns)) {
                *abort_flag = 1;
                raise_error(a.err, ERRBIT_TIMEOUT);
            }
            __threadfence();
        }
        __syncthreads();
        NMDLM_TSTAMP(a, 3);
    }

    // 32-channel groups of this CTA's slice after the split-K reduction; paired, a group
    // is a gate group g with its up group 4 + g (rows 32 g and 128 + 32 g of the sums).
    const int NGROUPS = paired ? HALF / 32 : TILE / 32;
    const int ns = a.nsplit;
    const int rank = split;
    const int g0 = rank * NGROUPS / ns, g1 = (rank + 1) * NGROUPS / ns, ngr = g1 - g0;
    const int parts = paired ? 2 : 1;  // contiguous row blocks per slice
    int32_t* accs = (int32_t*)smem;  // [TILE][ACC_STRIDE]: channel-major, padded

    const int res_c0 = lo0 + g0 * 32;
    const int res_c1 = min(lo0 + g1 * 32, s.n_out);
    const uint32_t res_row_bytes = res_c1 > res_c0 ? (uint32_t)(res_c1 - res_c0) * 4u : 0u;
    float* res_s = (float*)(smem + ACC_BYTES);
    const bool res_pref = !aborted && !paired && s.res && a.kind == EPI_KIND_F32 && res_row_bytes > 0 &&
                          (((uintptr_t)s.res) & 15) == 0 &&
                          (size_t)ACC_BYTES + (size_t)a.BT * ngr * 128 <= (size_t)OFF_BAR;
    if (res_pref && warp == WARP_PROD) {
        // 16-byte cp.async pieces over the warp (many small TMA bulk copies issue slowly)
        const int pieces = (int)(res_row_bytes >> 4), total = a.BT * pieces;
        const float* src = s.res + res_c0;
        const size_t ld = (size_t)s.n_out;
        for (int i = lane; i < total; i += 32) {
            const int bt = i / pieces, pc = i - bt * pieces;
            cp_async16(res_s + (size_t)bt * ngr * 32 + pc * 4, src + (size_t)bt * ld + pc * 4, 16u);
        }
        cp_async_mbar_arrive(res_bar);
    }

    if (sync_slots) {
        // This split's slice of the tile, summed over the splits' slots into the sums'
        // shared-memory layout: item = (channel of the slice, 4 rows).  A thread takes IB
        // items at a time with up to 8 of their 16-byte pieces in flight.
        const int BTP = a.btp, nq = BTP >> 2;
        const int n_items = parts * ngr * 32 * nq;
        const bool live = !*abort_flag && !aborted;
        // segment columns read with constant indices (a run-time index into the parameter
        // block is a slow generic load)
        const int col0_h0 = paired ? a.seg[0].col0 : s.col0;
        const int col0_h1 = paired ? a.seg[1].col0 : s.col0;
        auto slice_sum = [&](auto IBc) {
            constexpr int IB = decltype(IBc)::value, SB = 8 / IB;
            for (int base = tid; base < n_items && live; base += IB * NTHREADS) {
                const int4* src[IB];
                int m[IB];
                int4 sum[IB];
#pragma unroll
                for (int u = 0; u < IB; ++u) {
                    const int it = base + u * NTHREADS;
                    const int k = it % nq, cidx = it / nq;
                    const int c = cidx & 31, gl = (cidx >> 5) % ngr, pt = (cidx >> 5) / ngr;
                    const int ch = (g0 + gl) * 32 + c;  // channel within the half / tile
                    m[u] = it < n_items ? (pt * HALF + ch) * ACC_STRIDE + 4 * k : -1;
                    const int col0 = pt ? col0_h1 : col0_h0;
                    src[u] = (it < n_items && lo0 + ch < s.n_out)
                                 ? (const int4*)(a.acc_g + (size_t)(col0 + lo0 + ch) * BTP) + k
                                 : nullptr;
                    sum[u] = make_int4(0, 0, 0, 0);
                }
                for (int sp0 = 0; sp0 < ns; sp0 += SB) {
                    int4 v[IB][SB];
#pragma unroll
                    for (int u = 0; u < IB; ++u)
#pragma unroll
                        for (int q = 0; q < SB; ++q)
                            v[u][q] = (src[u] && sp0 + q < ns)
                                          ? __ldcg(src[u] + (size_t)(sp0 + q) * (a.acc_stride / 4))
                                          : make_int4(0, 0, 0, 0);
#pragma unroll
                    for (int u = 0; u < IB; ++u)
#pragma unroll
                        for (int q = 0; q < SB; ++q) {
                            sum[u].x += v[u][q].x; sum[u].y += v[u][q].y;
                            sum[u].z += v[u][q].z; sum[u].w += v[u][q].w;
                        }
                }
#pragma unroll
                for (int u = 0; u < IB; ++u)
                    if (m[u] >= 0) {
                        int32_t* d = accs + m[u];
                        d[0] = sum[u].x; d[1] = sum[u].y; d[2] = sum[u].z; d[3] = sum[u].w;
                    }
            }
        };
        if (ns <= 2) slice_sum(std::integral_constant<int, 4>());
        else if (ns <= 4) slice_sum(std::integral_constant<int, 2>());
        else slice_sum(std::integral_constant<int, 1>());
        __syncthreads();
        // departure: the last split of the tile to have read the slots zeroes the counters
        if (tid == 0) {
            unsigned* const tk = a.tickets + 2 * tile;
            if (atomicAdd(&tk[1], 1u) == (unsigned)ns - 1) {
                tk[0] = 0u;
                tk[1] = 0u;
            }
        }
        NMDLM_TSTAMP(a, 12);
    }

    // TMEM -> shared, exact fp32 -> int32: warp w reads lanes 32 (w % 4) + lane (rows bt)
    // and 64 of the 256 channel columns.
    if (!sync_slots && !aborted && warp < NCONV) {
        const int q = warp & 3, cs = warp >> 2;
        const int bt = q * 32 + lane;
        const int bias = W_BIAS * cnt_s[bt];
#pragma unroll 1
        for (int cb = cs * 32; cb < TILE; cb += 128) {
            uint32_t v[32];
            if (nj > 0) {
                tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(TM_D + cb), v);
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = 0;
            }
#pragma unroll
            for (int i = 0; i < 32; ++i)
                accs[(cb + i) * ACC_STRIDE + bt] =
                    __float2int_rn(__fmul_rn(__uint_as_float(v[i]), 65536.0f)) - bias;
        }
    }
    if (!sync_slots) {
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (warp == WARP_MMA) tmem_dealloc(tmem, NCOL);
        NMDLM_TSTAMP(a, 3);
    }

    if (ns > 1 && !sync_slots) {
        if (tid == 0)
            mbar_arrive_expect_tx(red_bar, (uint32_t)((ns - 1) * parts * ngr * GROUP_BYTES));
        cluster_arrive();
        cluster_wait();
        if (tid == 0) {
            for (int k = 1; k < ns; ++k) {
                const int qr = (rank + k) % ns;
                const int q0 = qr * NGROUPS / ns, q1 = (qr + 1) * NGROUPS / ns;
                for (int pt = 0; pt < parts && q1 > q0; ++pt) {
                    const uint32_t off = (uint32_t)((q0 + pt * (HALF / 32)) * GROUP_BYTES);
                    bulk_reduce_add_u32_peer(mapa_shared(smem_u32(smem) + off, (uint32_t)qr),
                                             smem + off, (uint32_t)((q1 - q0) * GROUP_BYTES),
                                             mapa_shared(smem_u32(red_bar), (uint32_t)qr));
                }
            }
        }
        const bool got = mbar_wait_bounded(red_bar, 0, a.wait_ns);
        if (!got) raise_error(a.err, ERRBIT_TIMEOUT);
        ok = __syncthreads_and(got) && !aborted;
        cluster_arrive();
    } else {
        ok = !aborted && !*abort_flag;
    }
    NMDLM_TSTAMP(a, 4);

    bool res_ok = true;
    if (res_pref) res_ok = mbar_wait_bounded(res_bar, 0, a.wait_ns);
    if (!res_ok && tid == 0) raise_error(a.err, ERRBIT_TIMEOUT);
    NMDLM_TSTAMP_W(a, 0, 8);
    if (ok && res_ok && warp < NCONV && ngr > 0) {
        // The segment's fields in registers: `s` lives in the kernel's parameter block
        // and is indexed at run time, so every read through it is a generic load.
        EpiWarp e;
        e.dbg = (a.dbg && blockIdx.x == 0 && blockIdx.y == 0 && warp == 0) ? a.dbg : nullptr;
        e.n_out = s.n_out;
        e.T = a.T;
        e.theta_i = a.theta_i;
        e.theta_f = a.theta_f;
        e.g_res = s.res;
        e.g_gate = s.gate;
        e.g_cur = s.cur;
        e.g_bits = s.bits;
        e.sb = s.sb;
        e.sst = s.st;
        e.nw = words_of(e.n_out);
        e.rstride = ngr * 32;
        const float* const scl = (const float*)(smem + C::OFF_SCL);
        int32_t* const g_acc = s.acc_out;
        const int kind = a.kind;
        const int resm = !e.g_res ? EPI_RES_NONE : (res_pref ? EPI_RES_SMEM : EPI_RES_GLOBAL);
        // (channel group, token) units shared evenly by the converter warps: warp w takes
        // units [w U / NCONV, (w + 1) U / NCONV), U = groups x tokens, one call per group
        // its range touches
        const int U = ngr * a.B;
        const int u0 = warp * U / NCONV, u1 = (warp + 1) * U / NCONV;
        for (int cgl = u0 / a.B; cgl < ngr && cgl * a.B < u1; ++cgl) {
            const int b0 = max(u0 - cgl * a.B, 0), b1 = min(u1 - cgl * a.B, a.B);
            if (b0 >= b1) continue;
            const int m = (g0 + cgl) * 32 + lane;  // paired: gate row m, up row HALF + m
            e.lo = lo0 + m;
            e.valid = e.lo < e.n_out;
            e.lead = lane == 0 && (e.lo >> 5) < e.nw;
            e.lead_word = (e.lo >> 5) < e.nw;
            e.sc = e.valid ? scl[m] : 0.0f;
            if (paired) {
                e.acol = accs + (size_t)(HALF + m) * ACC_STRIDE;
                const float gsc = e.valid ? scl[HALF + m] : 0.0f;
                if (epi_gated_run(e, accs + (size_t)m * ACC_STRIDE, gsc, a.seg[0].bits,
                                  a.seg[0].sb, a.seg[0].st, b0, b1, cm_acc + m * 4))
                    any_acc[m] = 1;
                continue;
            }
            e.acol = accs + (size_t)m * ACC_STRIDE;
            e.rcol = res_s + cgl * 32 + lane;
            if (kind == EPI_KIND_LOGITS) {
                for (int b = b0; b < b1; ++b) {
                    int sum = 0;
                    for (int t = 0; t < e.T; ++t) sum += e.acol[b * e.T + t];
                    if (e.valid)
                        e.g_cur[(size_t)b * e.n_out + e.lo] =
                            __fdiv_rn(__fmul_rn((float)sum, e.sc), (float)e.T);
                }
                continue;
            }
            if (kind == EPI_KIND_INT && e.g_cur && e.valid)  // integer kind: current = acc * scale
                for (int bt = b0 * e.T; bt < b1 * e.T; ++bt)
                    e.g_cur[(size_t)bt * e.n_out + e.lo] = __fmul_rn((float)e.acol[bt], e.sc);
            if (g_acc && e.valid)
                for (int bt = b0 * e.T; bt < b1 * e.T; ++bt)
                    g_acc[(size_t)bt * e.n_out + e.lo] = e.acol[bt];
            if (epi_dispatch(e, kind == EPI_KIND_F32, resm, b0, b1, cm_acc + m * 4)) any_acc[m] = 1;
        }
    }
    NMDLM_TSTAMP_W(a, 0, 9);
    __syncthreads();
    if (ok && res_ok && warp < NCONV && a.kind != EPI_KIND_LOGITS) {
        uint32_t* const g_cm = s.cm;
        uint32_t* const g_mask = s.mask;
        const int n_out = s.n_out;
        for (int cg = g0 + warp; cg < g1; cg += NCONV) {
            const int m = cg * 32 + lane;
            const int lo = lo0 + m;
            const bool valid = lo < n_out;
            if (valid && g_cm)
                for (int w = 0; w < BTW; ++w) g_cm[(size_t)lo * BTW + w] = cm_acc[m * 4 + w];
            const uint32_t mw = __ballot_sync(0xffffffffu, valid && any_acc[m]);
            if (lane == 0 && g_mask && lo < n_out) g_mask[lo >> 5] = mw;
        }
    }
    NMDLM_TSTAMP(a, 5);
    if (ns > 1 && !sync_slots) cluster_wait();
    NMDLM_TSTAMP(a, 6);
    NMDLM_CSTAMP(a, 256, 3);
}

// ------------------------------------------------------------ IF epilogue ----
// The IF epilogue of k_linear_ts in slot mode: grid (groups of 32 output channels,
// blocks of 32 rows), block (32, 8): lane = channel, warp = token slot.  T divides 32, so
// a row block holds whole tokens and writes whole column-mask words; the active-channel
// mask words (cleared by k_linear_ts) are ORed over the row blocks.
enum { EPI_M_INT = 0, EPI_M_F32 = 1, EPI_M_LOGITS = 2, EPI_M_PAIRED = 3 };
constexpr int EPI_SB = 16;  // splits whose slots are read at once (one L2 round trip up to 16)

// Sum of the first NS splits' 16-byte pieces at base, base + stride, ...: every load
// issued before any is added (one L2 round trip).
template <int NS>
__device__ __forceinline__ int4 epi_sum_slots(const int4* base, size_t stride) {
    int4 v[NS];
#pragma unroll
    for (int u = 0; u < NS; ++u) v[u] = __ldcg(base + (size_t)u * stride);
    int4 s = make_int4(0, 0, 0, 0);
#pragma unroll
    for (int u = 0; u < NS; ++u) {
        s.x += v[u].x; s.y += v[u].y; s.z += v[u].z; s.w += v[u].w;
    }
    return s;
}
// The splits in groups of at most 12, each group's loads in flight together.
__device__ __forceinline__ int4 epi_sum(const int4* base, size_t stride, int ns) {
    int4 s = make_int4(0, 0, 0, 0);
    for (int sp0 = 0; sp0 < ns; sp0 += 12) {
        const int k = min(12, ns - sp0);
        const int4* b = base + (size_t)sp0 * stride;
        int4 t;
        switch (k) {
            case 1: t = epi_sum_slots<1>(b, stride); break;
            case 2: t = epi_sum_slots<2>(b, stride); break;
            case 3: t = epi_sum_slots<3>(b, stride); break;
            case 4: t = epi_sum_slots<4>(b, stride); break;
            case 5: t = epi_sum_slots<5>(b, stride); break;
            case 6: t = epi_sum_slots<6>(b, stride); break;
            case 7: t = epi_sum_slots<7>(b, stride); break;
            case 8: t = epi_sum_slots<8>(b, stride); break;
            case 9: t = epi_sum_slots<9>(b, stride); break;
            case 10: t = epi_sum_slots<10>(b, stride); break;
            case 11: t = epi_sum_slots<11>(b, stride); break;
            default: t = epi_sum_slots<12>(b, stride); break;
        }
        s.x += t.x; s.y += t.y; s.z += t.z; s.w += t.w;
    }
    return s;
}

// Specialised at compile time on the kind and on every optional stream: a warp-uniform
// branch on a run-time flag costs a branch resolution (~100 cycles here) per step.
// A CTA takes a.epi_rb consecutive 32-row blocks (2 when the grid would not fit the GPU
// in one wave), their sums requested together.
template <int MODE, bool RES, bool GATE, bool CUR, bool ACCO, bool GB>
__global__ void __launch_bounds__(256) k_linear_epi(const __grid_constant__ LinArgs a) {
    NMDLM_CSTAMP(a, 1024, 0);
    pdl_wait();
    NMDLM_TSTAMP(a, 30);
    NMDLM_CSTAMP(a, 1024, 1);
    const int lane = threadIdx.x, ty = threadIdx.y, tid = ty * 32 + lane;
    constexpr bool paired = MODE == EPI_M_PAIRED;
    // this block's segment and channel group; the segment is copied into registers with
    // constant indices (a run-time index into the parameter block costs a generic load
    // of ~1 k cycles per field read)
    int si = paired ? 1 : 0, grp = blockIdx.x;
    if (!paired) {
        const int ng0 = words_of(a.seg[0].n_out), ng1 = words_of(a.seg[1].n_out);
        if (a.nseg > 1 && grp >= ng0) {
            grp -= ng0;
            si = 1;
            if (a.nseg > 2 && grp >= ng1) { grp -= ng1; si = 2; }
        }
    }
    LinSeg s = a.seg[0];
    if (si == 1) s = a.seg[1];
    else if (si == 2) s = a.seg[2];
    const int gcol0 = a.seg[0].col0;
    const float* const gscale = a.seg[0].scale;
    uint32_t* const gbits = a.seg[0].bits;
    const long long gsb = a.seg[0].sb, gsst = a.seg[0].st;
    const int n_out = s.n_out;
    const int lo = grp * 32 + lane;
    const bool valid = lo < n_out;
    const int T = a.T, BTP = a.btp, BTW = words_of(a.BT);
    const int RB = a.epi_rb > 1 ? 2 : 1;
    const int q0 = blockIdx.y * RB;  // first 32-row block of this CTA
    const float sc = (valid && s.scale) ? __ldg(s.scale + lo) : 0.0f;
    const float gsc = (valid && paired && gscale) ? __ldg(gscale + lo) : 0.0f;
    const int nw = words_of(n_out);
    __shared__ int32_t a_s[2][2][32][33];  // [row block][src][channel][row]
    __shared__ uint32_t cm_s[2][32];
    const int nparts = a.nsplit;  // the splits' slots
    // T <= 4: this thread's first token's residuals (per row block) requested with the
    // slot loads below, so their latency overlaps
    float rv0[2][4] = {{0.0f, 0.0f, 0.0f, 0.0f}, {0.0f, 0.0f, 0.0f, 0.0f}};
    if constexpr (RES) {
        const int T0 = a.T;
        for (int rb = 0; rb < RB; ++rb) {
            const int r0 = (q0 + rb) * 32, b = r0 / T0 + threadIdx.y;
            if (T0 <= 4 && valid && s.res && b < min((r0 + 32) / T0, a.B))
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (u < T0) rv0[rb][u] = __ldg(s.res + (size_t)(b * T0 + u) * n_out + lo);
        }
    }
    // the blocks' sums: thread = (channel tid / 8, rows r0 + 4 (tid % 8) .. + 3), every
    // split's 16-byte piece of every row block and source requested before any is added
    {
        const int c = tid >> 3, k = tid & 7;
        const int ncol = min(32, n_out - grp * 32);
        const size_t stride = (size_t)(a.acc_stride / 4);
        int4 sum[2][2];
#pragma unroll
        for (int rb = 0; rb < 2; ++rb)
#pragma unroll
            for (int src = 0; src < 2; ++src) {
                const int r0 = (q0 + rb) * 32;
                const bool in = rb < RB && (src == 0 || paired) && c < ncol && r0 + 4 * k < BTP;
                const int col0 = (src == 0 ? s.col0 : gcol0) + grp * 32 + c;
                sum[rb][src] = make_int4(0, 0, 0, 0);
                if (in)
                    sum[rb][src] = epi_sum((const int4*)(a.acc_g + (size_t)col0 * BTP + r0) + k,
                                           stride, nparts);
            }
#pragma unroll
        for (int rb = 0; rb < 2; ++rb)
#pragma unroll
            for (int src = 0; src < 2; ++src) {
                a_s[rb][src][c][4 * k] = sum[rb][src].x;
                a_s[rb][src][c][4 * k + 1] = sum[rb][src].y;
                a_s[rb][src][c][4 * k + 2] = sum[rb][src].z;
                a_s[rb][src][c][4 * k + 3] = sum[rb][src].w;
            }
    }
    if (ty == 0) {
        cm_s[0][lane] = 0u;
        cm_s[1][lane] = 0u;
    }
    __syncthreads();
    NMDLM_TSTAMP(a, 31);
    float* const cur = s.cur;
    int32_t* const acco = s.acc_out;
    const float* const res = s.res;
    const uint32_t* const gate = s.gate;
    uint32_t* const bits = s.bits;
    const long long sb = s.sb, sst = s.st;
    const bool lead = lane == 0 && grp < nw;
    for (int rb = 0; rb < RB; ++rb) {
        const int r0 = (q0 + rb) * 32;
        const int32_t* const acol = a_s[rb][0][lane];  // output channels (paired: up)
        const int32_t* const gcol = a_s[rb][1][lane];  // paired: gate
        const int b_end = min((r0 + 32) / T, a.B);
        for (int b = r0 / T + ty; b < b_end; b += 8) {
            uint32_t tb = 0;
            int vi = 0;
            float vf = 0.0f, vg = 0.0f;
            int lsum = 0;
            for (int t0 = 0; t0 < T; t0 += 4) {
                // four steps' residuals requested before the recurrence runs over them
                float rv[4];
                const bool pre = T <= 4 && b == r0 / T + ty;  // preloaded above
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    rv[u] = pre ? rv0[rb][u]
                                : ((RES && valid && res && t0 + u < T)
                                       ? __ldg(res + (size_t)(b * T + t0 + u) * n_out + lo) : 0.0f);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int t = t0 + u;
                    if (t >= T) break;
                    const int bt = b * T + t;
                    const int acc = acol[bt - r0];
                    if constexpr (MODE == EPI_M_LOGITS) {
                        lsum += acc;
                        continue;
                    }
                    if (ACCO && valid && acco) acco[(size_t)bt * n_out + lo] = acc;
                    bool sp, gsp = false;
                    if constexpr (MODE == EPI_M_PAIRED) {
                        const float ig = __fmul_rn((float)gcol[bt - r0], gsc);
                        const float hg = __fadd_rn(vg, ig);
                        gsp = valid && hg >= a.theta_f;
                        vg = gsp ? __fsub_rn(hg, a.theta_f) : hg;
                        const float iu = gsp ? __fmul_rn((float)acc, sc) : 0.0f;
                        if (CUR && valid && cur) cur[(size_t)bt * n_out + lo] = iu;
                        const float hu = __fadd_rn(vf, iu);
                        sp = valid && hu >= a.theta_f;
                        vf = sp ? __fsub_rn(hu, a.theta_f) : hu;
                    } else if constexpr (MODE == EPI_M_INT) {
                        const int h = vi + acc;
                        sp = valid && h >= a.theta_i;
                        vi = sp ? h - a.theta_i : h;
                        if (CUR && valid && cur) cur[(size_t)bt * n_out + lo] = __fmul_rn((float)acc, sc);
                    } else {
                        float I = __fmul_rn((float)acc, sc);
                        if (RES) I = __fadd_rn(I, rv[u]);
                        if (GATE) {
                            const uint32_t gw = gate ? (valid ? __ldg(gate + (size_t)bt * nw + (lo >> 5)) : 0u) : ~0u;
                            I = ((gw >> (lo & 31)) & 1u) ? I : 0.0f;
                        }
                        if (CUR && valid && cur) cur[(size_t)bt * n_out + lo] = I;
                        const float h = __fadd_rn(vf, I);
                        sp = valid && h >= a.theta_f;
                        vf = sp ? __fsub_rn(h, a.theta_f) : h;
                    }
                    const uint32_t word = __ballot_sync(0xffffffffu, sp);
                    if (lead) bits[(long long)b * sb + (long long)t * sst + grp] = word;
                    if constexpr (MODE == EPI_M_PAIRED && GB) {
                        const uint32_t gword = __ballot_sync(0xffffffffu, gsp);
                        if (lead) gbits[(long long)b * gsb + (long long)t * gsst + grp] = gword;
                    }
                    tb |= (sp ? 1u : 0u) << t;
                }
            }
            if constexpr (MODE == EPI_M_LOGITS) {
                if (valid && cur) cur[(size_t)b * n_out + lo] = __fdiv_rn(__fmul_rn((float)lsum, sc), (float)T);
                continue;
            }
            if (tb) atomicOr(&cm_s[rb][lane], tb << (b * T - r0));
        }
    }
    NMDLM_TSTAMP(a, 32);
    if constexpr (MODE != EPI_M_LOGITS) {
        __syncthreads();
        if (ty == 0) {
            uint32_t any = 0u;
            for (int rb = 0; rb < RB; ++rb) {
                const uint32_t w = cm_s[rb][lane];
                if (valid && s.cm) s.cm[(size_t)lo * BTW + q0 + rb] = w;
                any |= w;
            }
            const uint32_t act = __ballot_sync(0xffffffffu, valid && any != 0u);
            if (lane == 0 && act && s.mask) atomicOr(&s.mask[grp], act);
        }
    }
    NMDLM_CSTAMP(a, 1024, 3);
}

// ------------------------------------------------------------------ stats ----
__global__ void k_linear_stats(const uint32_t* cm, const uint32_t* mask, int d_in, int BTW,
                               int dense, unsigned long long dout, unsigned long long* stats) {
    pdl_wait();
    unsigned long long rows = 0, nnz = 0;
    for (int d = blockIdx.x * blockDim.x + threadIdx.x; d < d_in; d += gridDim.x * blockDim.x) {
        const bool act = (mask[d >> 5] >> (d & 31)) & 1u;
        rows += (dense || act) ? 1 : 0;
        if (act)
            for (int w = 0; w < BTW; ++w) nnz += __popc(cm[(size_t)d * BTW + w]);
    }
    for (int o = 16; o > 0; o >>= 1) {
        rows += __shfl_down_sync(0xffffffffu, rows, o);
        nnz += __shfl_down_sync(0xffffffffu, nnz, o);
    }
    if ((threadIdx.x & 31) == 0) {
        if (rows) atomicAdd(&stats[0], rows);
        if (nnz) atomicAdd(&stats[1], nnz * dout);
    }
}

nmdlm_status launch_linear_stats(const uint32_t* cm, const uint32_t* mask, int d_in, int BTW,
                                 int dense, unsigned long long dout,
                                 unsigned long long* stats, cudaStream_t stream) {
    const int threads = 256;
    const int blocks = std::min(64, (d_in + threads - 1) / threads);
    const cudaError_t le = launch_pdl(k_linear_stats, dim3(blocks), dim3(threads), 0, stream, 1,
                                      cm, mask, d_in, BTW, dense, dout, stats);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

// ------------------------------------------------------------------ launch ----
template <int MAXT, int MAXW>
static nmdlm_status launch_simt_t(LinArgs& a, cudaStream_t stream) {
    int groups = 0;
    for (int i = 0; i < a.nseg; ++i) {
        a.seg[i].tile_begin = groups;
        groups += words_of(a.seg[i].n_out);
    }
    a.n_tiles = groups;
    int g = 1;
    while (g < 32 && (g * a.T) % 32 != 0) g <<= 1;  // tokens per 32-bit column word
    const int BY = std::max(1, std::min(a.B, std::max(g, 8)));
    dim3 block(32, BY);
    const cudaError_t le = launch_pdl(k_linear_simt<MAXT, MAXW>, dim3(groups), dim3(block), 0,
                                      stream, 1, a);
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

static nmdlm_status launch_simt(LinArgs& a, cudaStream_t stream) {
    if (a.T <= 4 && a.BTW <= 8) return launch_simt_t<4, 8>(a, stream);
    if (a.T <= 8 && a.BTW <= 8) return launch_simt_t<8, 8>(a, stream);
    return launch_simt_t<32, 8>(a, stream);
}

template <int NP, int TILE>
static nmdlm_status launch_tc_t(nmdlm_ctx* ctx, LinArgs& a, WsCursor&, cudaStream_t stream) {
    using SM = tcl::Smem<NP, TILE>;
    if (a.d_in > 65535) return NMDLM_ERR_UNSUPPORTED;  // u16 row indices
    int tiles = 0;
    for (int i = 0; i < a.nseg; ++i) {
        a.seg[i].tile_begin = tiles;
        tiles += (a.seg[i].n_out + TILE - 1) / TILE;
    }
    a.n_tiles = tiles;
    // Shared memory is sized for the worst split (one split holds every row).
    const int max_chunks = std::max(1, (a.d_in + tcl::KC - 1) / tcl::KC);
    const int rows_cap = std::min(tcl::MAXROWS, (max_chunks + 1) * tcl::KC);
    const size_t smem = SM::bytes(words_of(a.d_in), rows_cap);
    if (smem > 225 * 1024) return NMDLM_ERR_UNSUPPORTED;
    if (ensure_dyn_smem((const void*)k_linear_tc<NP, TILE>, smem) != NMDLM_OK)
        return NMDLM_ERR_CUDA;
    // Splits per tile (cluster size, <= 8): the largest whose clusters all fit on the
    // GPU at once (measured by the occupancy API for this size) while each split keeps
    // at least 4 chunks of rows.
    int max_clusters[9];
    if (cluster_capacity((const void*)k_linear_tc<NP, TILE>, tcl::NTHREADS, smem, ctx->sm_count,
                         max_clusters) != NMDLM_OK)
        return NMDLM_ERR_CUDA;
    int nsplit = 1;
    for (int n = 2; n <= 8; ++n)
        if (tiles <= max_clusters[n] && max_chunks / n >= 4) nsplit = n;
    const int rows_max = ((max_chunks + nsplit - 1) / nsplit + 1) * tcl::KC;
    if (rows_max > rows_cap) return NMDLM_ERR_UNSUPPORTED;
    a.nsplit = nsplit;
    a.ws = nullptr;
    a.counters = nullptr;
    for (int i = 0; i < a.nseg; ++i) {
        nmdlm_status st = weight_tensor_map(ctx, a.seg[i].wT, a.d_in, a.seg[i].n_out,
                                            a.seg[i].ld_w, tcl::KC, &a.tmap[i]);
        if (st == NMDLM_OK)
            st = weight_tensor_map(ctx, a.seg[i].wT, a.d_in, a.seg[i].n_out, a.seg[i].ld_w, 1,
                                   &a.gmap[i]);
        if (st != NMDLM_OK) return st;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(tiles, nsplit, 1);
    cfg.blockDim = dim3(tcl::NTHREADS, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 1;
    attr[1].val.clusterDim.y = nsplit;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = nsplit > 1 ? 2 : 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, k_linear_tc<NP, TILE>, a);
    count_launch();
    return cuda_status(e);
}

// Launch geometry of k_linear_ts<TILE>: shared memory, and the clusters of each size
// that fit on the GPU at once (occupancy API), cached per tile width.
template <int TILE>
struct TsPlan {
    size_t smem = 0;
    int max_clusters[9] = {0};
};

template <int TILE>
static nmdlm_status ts_plan(nmdlm_ctx* ctx, const LinArgs& a, TsPlan<TILE>& plan) {
    using C = tcs::Cfg<TILE>;
    const int max_chunks = std::max(1, (a.d_in + C::KC - 1) / C::KC);
    const int rows_cap = std::min(tcl::MAXROWS, (max_chunks + 1) * C::KC);
    plan.smem = C::bytes(words_of(a.d_in), rows_cap);
    if (plan.smem > 225 * 1024) return NMDLM_ERR_UNSUPPORTED;
    if (ensure_dyn_smem((const void*)k_linear_ts<TILE>, plan.smem) != NMDLM_OK)
        return NMDLM_ERR_CUDA;
    int cached[9];
    if (cluster_capacity((const void*)k_linear_ts<TILE>, tcs::NTHREADS, plan.smem, ctx->sm_count,
                         cached) != NMDLM_OK)
        return NMDLM_ERR_CUDA;
    for (int n = 0; n <= 8; ++n) plan.max_clusters[n] = cached[n];
    return NMDLM_OK;
}

// Estimated cycles of one launch.  Main loop: the split with the most weight bytes at
// the per-SM streaming rate (bounded by the HBM share when many CTAs stream); measured
// on GB300 ~14.5 B/cycle per SM with 256-channel tiles and ~12.5 with 128-channel tiles
// (an MMA of N <= 128 costs ~100 cycles, one of N = 256 ~135), ~3.5 KB/cycle for the
// whole GPU from HBM.  Tail, cluster mode: the in-kernel IF epilogue (~8 k cycles) and
// the split-K exchange through distributed shared memory (~14 B/cycle per CTA).  Slot
// mode: each CTA's 128 KB of partial sums to L2 (~4.6 k cycles), the epilogue launch
// (~6 k cycles) and its reading of every slot (~4 KB/cycle for the GPU).
static double ts_cost(int tiles, int tile_w, int ns, int rows, int sm_count, bool slot,
                      double slot_bytes) {
    const int ctas = tiles * ns;
    const int waves = (ctas + sm_count - 1) / sm_count;
    const double per_cta =
        std::min(tile_w == 256 ? 14.5 : (tile_w == 192 ? 14.0 : 12.5), 3500.0 / std::min(ctas, sm_count));
    const double rows_split = (double)((rows + ns - 1) / ns);
    double c = waves * rows_split * tile_w / per_cta;
    if (slot) return c + 3000.0 + 6000.0 + slot_bytes / 8192.0;
    c += 8000.0;
    if (ns > 1) c += (double)(tile_w / 32) * tcs::GROUP_BYTES * (ns - 1) / ns / 14.0;
    return c;
}

// The IF epilogue over the splits' slots (grid: groups of 32 output channels x blocks
// of 32 rows).
static nmdlm_status launch_ts_epi(const LinArgs& a0, int sm_count, cudaStream_t stream) {
    LinArgs a = a0;
    int groups = 0;
    if (a.paired) groups = words_of(a.seg[1].n_out);
    else
        for (int i = 0; i < a.nseg; ++i) groups += words_of(a.seg[i].n_out);
    // two 32-row blocks per CTA when one per CTA would not fit the GPU in one wave
    // (about 5 CTAs of 256 threads per SM)
    const int BTW = words_of(a.BT);
    a.epi_rb = (BTW % 2 == 0 && (size_t)groups * BTW > (size_t)5 * sm_count) ? 2 : 1;
    const dim3 grid(groups, BTW / a.epi_rb), block(32, 8);
    cudaError_t le = cudaErrorInvalidValue;
    bool cur = false, acco = false, res = false, gate = false;
    for (int i = 0; i < a.nseg; ++i) {
        if (a.paired && i == 0) continue;
        cur |= a.seg[i].cur != nullptr;
        acco |= a.seg[i].acc_out != nullptr;
        res |= a.seg[i].res != nullptr;
        gate |= a.seg[i].gate != nullptr;
    }
    // (the flags say which streams any segment has; a segment's null pointer is still
    // checked before each access)
#define NMDLM_EPI_LAUNCH(MODE, R, G, C, A, GB) \
    le = launch_pdl(k_linear_epi<MODE, R, G, C, A, GB>, grid, block, 0, stream, 1, a)
    if (a.paired) {
        const bool gb = a.seg[0].bits != nullptr;
        if (cur) { if (gb) NMDLM_EPI_LAUNCH(EPI_M_PAIRED, false, false, true, false, true);
                   else NMDLM_EPI_LAUNCH(EPI_M_PAIRED, false, false, true, false, false); }
        else { if (gb) NMDLM_EPI_LAUNCH(EPI_M_PAIRED, false, false, false, false, true);
               else NMDLM_EPI_LAUNCH(EPI_M_PAIRED, false, false, false, false, false); }
    } else if (a.kind == EPI_KIND_LOGITS) {
        NMDLM_EPI_LAUNCH(EPI_M_LOGITS, false, false, true, false, false);
    } else if (a.kind == EPI_KIND_INT) {
        if (cur) { if (acco) NMDLM_EPI_LAUNCH(EPI_M_INT, false, false, true, true, false);
                   else NMDLM_EPI_LAUNCH(EPI_M_INT, false, false, true, false, false); }
        else { if (acco) NMDLM_EPI_LAUNCH(EPI_M_INT, false, false, false, true, false);
               else NMDLM_EPI_LAUNCH(EPI_M_INT, false, false, false, false, false); }
    } else {
#define NMDLM_EPI_F32(R, G)                                                                   \
        if (cur) { if (acco) NMDLM_EPI_LAUNCH(EPI_M_F32, R, G, true, true, false);             \
                   else NMDLM_EPI_LAUNCH(EPI_M_F32, R, G, true, false, false); }               \
        else { if (acco) NMDLM_EPI_LAUNCH(EPI_M_F32, R, G, false, true, false);                \
               else NMDLM_EPI_LAUNCH(EPI_M_F32, R, G, false, false, false); }
        if (res) { if (gate) { NMDLM_EPI_F32(true, true) } else { NMDLM_EPI_F32(true, false) } }
        else { if (gate) { NMDLM_EPI_F32(false, true) } else { NMDLM_EPI_F32(false, false) } }
#undef NMDLM_EPI_F32
    }
#undef NMDLM_EPI_LAUNCH
    count_launch();
    if (le != cudaSuccess) return cuda_status(le);
    return cuda_status(cudaGetLastError());
}

template <int TILE>
static nmdlm_status launch_ts_t(nmdlm_ctx* ctx, LinArgs& a, const TsPlan<TILE>& plan, int nsplit,
                                bool slot, cudaStream_t stream) {
    using C = tcs::Cfg<TILE>;
    int tiles = 0;
    if (a.paired) {  // one tile = HALF gate channels + the same HALF up channels
        tiles = (a.seg[1].n_out + C::HALF - 1) / C::HALF;
        a.seg[0].tile_begin = a.seg[1].tile_begin = 0;
    } else {
        for (int i = 0; i < a.nseg; ++i) {
            a.seg[i].tile_begin = tiles;
            tiles += (a.seg[i].n_out + TILE - 1) / TILE;
        }
    }
    int cols = 0;
    for (int i = 0; i < a.nseg; ++i) {
        a.seg[i].col0 = cols;
        cols += a.seg[i].n_out;
    }
    a.btp = (a.BT + 3) & ~3;
    a.acc_stride = (long long)cols * a.btp;
    a.slot_mode = slot ? 1 : 0;
    if (slot && (size_t)nsplit * cols * a.btp * sizeof(int32_t) > ctx->acc_bytes)
        return NMDLM_ERR_UNSUPPORTED;
    // slot split-K: the slots are summed by the epilogue kernel, or, on request (debug key
    // 3 = 3), by the tile's splits themselves after meeting at a counter (every CTA of the
    // launch resident at once).  The in-kernel meeting measured 1.5-3 us slower per launch
    // on the decode shapes: each split's slice sum is bound by L2 latency, the separate
    // kernel spreads the same sums over more threads.
    a.slot_sync = (slot && ctx->split_force == 3) ? 1 : 0;
    a.tickets = ctx->counters ? ctx->counters + kLinTicketBase : nullptr;
    if (a.slot_sync && (!a.tickets || kLinTicketBase + 2 * (size_t)tiles > ctx->n_counters ||
                        (size_t)tiles * nsplit > (size_t)ctx->sm_count))
        return NMDLM_ERR_UNSUPPORTED;
    a.acc_g = ctx->acc;
    a.n_tiles = tiles;
    a.nsplit = nsplit;
    a.ws = nullptr;
    a.counters = nullptr;
    for (int i = 0; i < a.nseg; ++i) {
        nmdlm_status st = weight_tensor_map(ctx, a.seg[i].wT, a.d_in, a.seg[i].n_out,
                                            a.seg[i].ld_w, C::KC, &a.tmap[i], C::BOXW);
        if (st == NMDLM_OK)
            st = weight_tensor_map(ctx, a.seg[i].wT, a.d_in, a.seg[i].n_out, a.seg[i].ld_w, 1,
                                   &a.gmap[i]);
        if (st != NMDLM_OK) return st;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(tiles, nsplit, 1);
    cfg.blockDim = dim3(tcs::NTHREADS, 1, 1);
    cfg.dynamicSmemBytes = plan.smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 1;
    attr[1].val.clusterDim.y = nsplit;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = (!slot && nsplit > 1) ? 2 : 1;
    a.nsplit = nsplit;
    cudaError_t e = cudaLaunchKernelEx(&cfg, k_linear_ts<TILE>, a);
    count_launch();
    if (e != cudaSuccess) return cuda_status(e);
    return (slot && !a.slot_sync) ? launch_ts_epi(a, ctx->sm_count, stream) : NMDLM_OK;
}

// k_linear_ts for blocks of at most 128 rows: picks the tile width (128 or 256
// channels) and the split count with the lowest estimated time (one wave of CTAs at
// most); UNSUPPORTED when no choice keeps a split's active rows within the exact range.
static nmdlm_status launch_ts(nmdlm_ctx* ctx, LinArgs& a, cudaStream_t stream) {
    if (a.d_in > 65535) return NMDLM_ERR_UNSUPPORTED;  // u16 row indices
    if (a.T > 32 || a.BT > 128) return NMDLM_ERR_UNSUPPORTED;
    TsPlan<128> p128;
    TsPlan<192> p192;
    TsPlan<256> p256;
    const bool ok128 = ts_plan<128>(ctx, a, p128) == NMDLM_OK;
    const bool ok192 = a.paired && ts_plan<192>(ctx, a, p192) == NMDLM_OK;
    const bool ok256 = ts_plan<256>(ctx, a, p256) == NMDLM_OK;
    int tiles128 = 0, tiles192 = 0, tiles256 = 0;
    for (int i = 0; i < a.nseg; ++i) {
        tiles128 += (a.seg[i].n_out + 127) / 128;
        tiles256 += (a.seg[i].n_out + 255) / 256;
    }
    if (a.paired) {  // gate + up pairs: the two halves of a 256 (or 192) tile
        if (a.nseg != 2 || a.seg[0].n_out != a.seg[1].n_out) return NMDLM_ERR_INVALID_ARG;
        tiles256 = (a.seg[1].n_out + 127) / 128;
        tiles192 = (a.seg[1].n_out + 95) / 96;
    }
    int cols_total = 0;
    for (int i = 0; i < a.nseg; ++i) cols_total += a.seg[i].n_out;
    const double slot_words = (double)cols_total * ((a.BT + 3) & ~3);
    double best = 1e300;
    int best_tile = 0, best_ns = 1;
    bool best_slot = false;
    // debug key 6: the tile width to use when this launch can use it
    const int pt_req = ctx->plan_tile;
    const bool pt_ok = pt_req == 128 ? (ok128 && !a.paired)
                                     : (pt_req == 192 ? ok192 : (pt_req == 256 && ok256));
    const int plan_tile = pt_ok ? pt_req : 0;
    for (int tw = 128; tw <= 256; tw += 64) {
        if ((tw == 128 && (!ok128 || a.paired)) || (tw == 192 && !ok192) || (tw == 256 && !ok256))
            continue;
        const int tiles = tw == 128 ? tiles128 : (tw == 192 ? tiles192 : tiles256);
        const int kc = tw == 192 ? tcs::Cfg<192>::KC : 16384 / tw;
        const int max_chunks = std::max(1, (a.d_in + kc - 1) / kc);
        const int* mc = tw == 128 ? p128.max_clusters
                                  : (tw == 192 ? p192.max_clusters : p256.max_clusters);
        for (int n = 1; n <= 16; ++n) {
            if (n > 1 && max_chunks / n < 2) continue;
            const int rows_split = ((max_chunks + n - 1) / n + 1) * kc;
            if (rows_split > tcl::MAXROWS || (max_chunks + n - 1) / n * kc > tcs::MAX_ROWS) continue;
            if ((plan_tile && plan_tile != tw) || (ctx->plan_ns && ctx->plan_ns != n)) continue;
            for (int slot = 0; slot < 2; ++slot) {
                if ((ctx->split_force == 1 && slot) || (ctx->split_force >= 2 && !slot && n > 1))
                    continue;
                if (!slot && n > 1 && (n > 8 || tiles > mc[n])) continue;
                if (slot && (n == 1 || 32 % a.T != 0 || tiles * n > ctx->sm_count ||
                             (size_t)n * slot_words * sizeof(int32_t) > ctx->acc_bytes))
                    continue;
                double c = ts_cost(tiles, tw, n, a.d_in, ctx->sm_count, slot != 0,
                                   n * slot_words * sizeof(int32_t));
                if (ctx->split_force && n == 1) c *= 4.0;  // forced modes: prefer splitting
                if (c < best) { best = c; best_tile = tw; best_ns = n; best_slot = slot != 0; }
            }
        }
    }
    if (getenv("NMDLM_PLAN_LOG"))
        fprintf(stderr, "ts plan: d_in %d tiles128 %d tiles256 %d -> tile %d ns %d slot %d\n", a.d_in,
                tiles128, tiles256, best_tile, best_ns, (int)best_slot);
    if (best_tile == 128) return launch_ts_t<128>(ctx, a, p128, best_ns, best_slot, stream);
    if (best_tile == 192) return launch_ts_t<192>(ctx, a, p192, best_ns, best_slot, stream);
    if (best_tile == 256) return launch_ts_t<256>(ctx, a, p256, best_ns, best_slot, stream);
    return NMDLM_ERR_UNSUPPORTED;
}

nmdlm_status launch_linear(nmdlm_ctx* ctx, LinArgs& a, nmdlm_impl impl, WsCursor& ws,
                           cudaStream_t stream) {
    a.err = ctx->err;
    a.wait_ns = ctx->wait_ns;
    a.desc_swap = ctx->desc_swap;
    bool stamp = ctx->dbg_on != 0;
    if (stamp && ctx->dbg_shape) {
        int n_out = 0;
        for (int i = 0; i < a.nseg; ++i) n_out += a.seg[i].n_out;
        stamp = a.d_in * 65536 + n_out == ctx->dbg_shape && ctx->dbg_count++ == ctx->dbg_nth;
    }
    a.dbg = stamp ? ctx->dbg : nullptr;
    if (ctx->mode_force == 1) {  // debug key 8: gather the active rows whatever the density
        a.dense = 0;
        a.auto_dense = 0;
    } else if (ctx->mode_force == 2) {  // ... or stream every row
        a.dense = 1;
    }
    if (a.paired) {  // only the TMEM-operand kernel pairs gate and up; else UNSUPPORTED
        bool ok = impl != NMDLM_IMPL_SIMT && a.BT <= 128 && a.T <= 32 &&
                  words_of(a.d_in) <= 4096 && !(impl == NMDLM_IMPL_AUTO && a.BT <= 8);
        for (int i = 0; i < a.nseg; ++i) {
            const LinSeg& s = a.seg[i];
            if (s.n_out % 16 || s.ld_w % 16 || ((uintptr_t)s.wT & 15)) ok = false;
        }
        if (!ok) return NMDLM_ERR_UNSUPPORTED;
        return launch_ts(ctx, a, stream);
    }
    bool tc_ok = a.BT <= 256 && a.T <= 32 && words_of(a.d_in) <= 4096;
    for (int i = 0; i < a.nseg; ++i) {
        const LinSeg& s = a.seg[i];
        if (s.n_out % 16 || s.ld_w % 16 || ((uintptr_t)s.wT & 15)) tc_ok = false;
        if (i + 1 < a.nseg && s.n_out % 256) tc_ok = false;
    }
    if (impl == NMDLM_IMPL_TC && !tc_ok) return NMDLM_ERR_UNSUPPORTED;
    bool use_tc = impl == NMDLM_IMPL_TC || (impl == NMDLM_IMPL_AUTO && tc_ok);
    if (!use_tc) {
        for (int i = 0; i + 1 < a.nseg; ++i)
            if (a.seg[i].n_out % 32) return NMDLM_ERR_UNSUPPORTED;
        return launch_simt(a, stream);
    }
    if (a.BT <= 128) {
        const nmdlm_status st = launch_ts(ctx, a, stream);
        if (st != NMDLM_ERR_UNSUPPORTED || ctx->plan_tile || ctx->plan_ns) return st;
    }
    if (a.BT <= 16) return launch_tc_t<16, 256>(ctx, a, ws, stream);
    if (a.BT <= 32) return launch_tc_t<32, 256>(ctx, a, ws, stream);
    if (a.BT <= 64) return launch_tc_t<64, 256>(ctx, a, ws, stream);
    if (a.BT <= 128) return launch_tc_t<128, 256>(ctx, a, ws, stream);
    return launch_tc_t<256, 128>(ctx, a, ws, stream);
}

}  // namespace nmdlm

namespace nmdlm {

nmdlm_status weight_tensor_map(nmdlm_ctx* ctx, const int8_t* wT, int d_in, int n_out, int ld,
                               int box_rows, CUtensorMap* out, int box_w) {
    if (box_w != 128 && box_w != 96) return NMDLM_ERR_INVALID_ARG;
    for (const auto& e : ctx->tmaps)
        if (e.ptr == wT && e.d_in == d_in && e.n_out == n_out && e.ld == ld &&
            e.box_rows == box_rows && e.box_w == box_w) {
            *out = e.map;
            return NMDLM_OK;
        }
    static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    if (!encode) {
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", (void**)&encode, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !encode) {
            cudaGetLastError();
            encode = nullptr;
            return NMDLM_ERR_CUDA;
        }
    }
    cuuint64_t dims[2] = {(cuuint64_t)n_out, (cuuint64_t)d_in};
    cuuint64_t strides[1] = {(cuuint64_t)ld};
    // 128-channel boxes with the 128-byte swizzle, or 96-channel boxes unswizzled
    cuuint32_t box[2] = {(cuuint32_t)box_w, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUtensorMap m;
    const CUresult r = encode(&m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, (void*)wT, dims, strides, box,
                              estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                              box_w == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return NMDLM_ERR_CUDA;
    if (ctx->tmaps.size() > 4096) ctx->tmaps.clear();
    ctx->tmaps.push_back({wT, d_in, n_out, ld, box_rows, box_w, m});
    *out = m;
    return NMDLM_OK;
}

}  // namespace nmdlm
