// common.cuh -- device helpers shared by the N-MDLM kernels (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "nmdlm.h"

namespace nmdlm {

// ----------------------------------------------------------- error word ----
// Bits of the context's device error word.
enum : int { ERRBIT_VALUE = 1, ERRBIT_TIMEOUT = 2 };

__device__ __forceinline__ void raise_error(int* err, int bit) {
    if (err) atomicOr(err, bit);
}

// ------------------------------------------------- programmatic launches ----
// Every kernel of the library is launched as a programmatic dependent of the previous
// one on its stream.  pdl_wait blocks until the previous kernel has completed and its
// memory is visible; a kernel touches no global data that another kernel of the chain
// writes or reads before it.  Only the spiking linear's slot launches trigger their
// dependent (the small epilogue kernel) early, at their partial-sum stores, so that its
// blocks fill SMs as the linear's CTAs exit.  Elsewhere an early trigger, at kernel entry
// or after the linear's weight streaming, measured slower on GB300 than the implicit
// trigger at exit, which still hides launch latency and lets the spiking linear run its
// setup and first L2 prefetches before the wait.
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Transpose a 32 x 32 bit block held one row per lane: on entry bit i of lane j's x is
// element (j, i); on return bit j of lane i's result is that element.  Recursive block
// transposition, [A B; C D] -> [A C; B D] on 16-, 8-, 4-, 2- and 1-bit blocks, one
// shuffle per stage.  All 32 lanes must call it.
__device__ __forceinline__ uint32_t warp_transpose32(uint32_t x) {
    const int lane = threadIdx.x & 31;
    uint32_t m = 0x0000FFFFu;
#pragma unroll
    for (int s = 16; s >= 1; s >>= 1, m ^= m << s) {
        const uint32_t y = __shfl_xor_sync(0xffffffffu, x, s);
        x = (lane & s) ? ((x & ~m) | ((y >> s) & m)) : ((x & m) | ((y << s) & ~m));
    }
    return x;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__host__ __device__ __forceinline__ int words_of(int n) { return (n + 31) >> 5; }

// ------------------------------------------------------------- mbarrier ----
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Non-blocking probe of the phase with the given parity: never suspends the thread, so
// an issuer can ask ahead and use the answer later.
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait for the phase with the given parity to complete, for at most limit_ns.
// Returns false if the limit ran out (the caller records a timeout and unwinds).
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}

// Acquire load of a counter in global memory at GPU scope.
__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Waits until *p >= target, for at most limit_ns; false when the limit ran out.
__device__ __forceinline__ bool wait_count_bounded(const unsigned* p, unsigned target,
                                                   uint64_t limit_ns) {
    if (ld_acquire_gpu(p) >= target) return true;
    const uint64_t t0 = globaltimer_ns();
    while (ld_acquire_gpu(p) < target) {
        if (globaltimer_ns() - t0 > limit_ns) return false;
        __nanosleep(32);
    }
    return true;
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}
// Arrive on `bar` once every cp.async this thread issued so far has landed (the
// barrier's expected count includes this arrival).
__device__ __forceinline__ void cp_async_mbar_arrive(uint64_t* bar) {
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}
// 2-D TMA tile load (x = innermost coordinate), completion counted on `bar`.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
        "l"(map), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}

// The same load with an L2 eviction-priority hint (a policy made by createpolicy):
// weights stream through L2 once per pass, so they are marked first to go.
__device__ __forceinline__ void tma_load_2d_hint(void* dst, const CUtensorMap* map, int x, int y,
                                                 uint64_t* bar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
        "[%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_u32(dst)),
        "l"(map), "r"(x), "r"(y), "r"(smem_u32(bar)), "l"(policy)
        : "memory");
}

// L2 policy: every line the access touches is evicted before others.
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// Prefetch one box of a 2-D tensor into L2 (no shared-memory destination).
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap* map, int x, int y) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global [%0, {%1, %2}];" ::"l"(map), "r"(x),
                 "r"(y)
                 : "memory");
}

// Prefetch `bytes` (multiple of 16, 16-byte aligned address) of global memory into L2.
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// 1-D bulk copy global -> shared (16-byte aligned addresses, size a multiple of 16).
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes,
                                          uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// Address of the same shared-memory location in CTA `rank` of this cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t saddr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
    return r;
}

// Bulk element-wise 32-bit integer add of `bytes` (multiple of 16) of this CTA's shared
// memory into a peer's shared memory (cluster addresses from mapa_shared); completion is
// counted in bytes on the peer's mbarrier `bar_cluster`.  Integer addition is exact and
// commutative, so the order in which peers arrive does not change the result.
__device__ __forceinline__ void bulk_reduce_add_u32_peer(uint32_t dst_cluster, const void* src,
                                                         uint32_t bytes, uint32_t bar_cluster) {
    asm volatile(
        "cp.reduce.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes.add.u32 "
        "[%0], [%1], %2, [%3];" ::"r"(dst_cluster),
        "r"(smem_u32(src)), "r"(bytes), "r"(bar_cluster)
        : "memory");
}

// Split cluster barrier: arrive (release) now, wait (acquire) later.  Every thread of
// every CTA of the cluster takes part.
// Bulk element-wise 32-bit integer add of `bytes` (multiple of 16, both addresses 16-byte
// aligned) of this CTA's shared memory into global memory, performed at L2; tracked by
// the issuing thread's bulk groups (bulk_commit / bulk_wait_all).
__device__ __forceinline__ void bulk_reduce_add_s32_global(int32_t* dst, const void* src, uint32_t bytes) {
    asm volatile("cp.reduce.async.bulk.global.shared::cta.bulk_group.add.s32 [%0], [%1], %2;" ::"l"(dst),
                 "r"(smem_u32(src)), "r"(bytes)
                 : "memory");
}
// Bulk copy of `bytes` (multiple of 16, both addresses 16-byte aligned) of this CTA's
// shared memory to global memory; tracked like bulk_reduce_add_s32_global.
__device__ __forceinline__ void bulk_store_global(void* dst, const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
                 "r"(smem_u32(src)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void cluster_arrive() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// ------------------------------------------------------------- cp.async ----
// 16-byte global -> shared copy; src_bytes < 16 zero-fills the rest (0 = all zero).
__device__ __forceinline__ void cp_async16(void* dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)),
                 "l"(src), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(smem_u32(dst)), "l"(src),
                 "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// ------------------------------------------------------- tcgen05 / TMEM ----
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Warp-collective: allocate ncols TMEM columns, base address written to *dst (smem).
__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(dst)),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr),
                 "r"(ncols)
                 : "memory");
}
// D[tmem] (+)= A[smem] * B[smem], kind::f16, issued by one thread.
__device__ __forceinline__ void mma_f16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                        uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// D[tmem] (+)= A[tmem] * B[smem], kind::f16, issued by one thread (A: one row per TMEM
// lane, two 16-bit elements of K per 32-bit column).
__device__ __forceinline__ void mma_f16_ts(uint32_t tmem_d, uint32_t tmem_a, uint64_t bdesc,
                                           uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(tmem_d),
        "r"(tmem_a), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Warp-collective: lane i writes 16 consecutive 32-bit columns of TMEM lane (base + i).
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
        "%13,%14,%15,%16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15])
        : "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
// Warp-collective: lane i reads 32 consecutive 32-bit columns of TMEM lane (base + i).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),
          "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]),
          "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
          "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]),
          "=r"(v[31])
        : "r"(taddr)
        : "memory");
}

// Arrive once on `bar` when every tcgen05.mma issued so far by this thread completes.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_u32(bar))
        : "memory");
}
// Warp-collective: lane i reads 8 consecutive 32-bit columns of TMEM lane (base + i).
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&v)[8]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]),
          "=r"(v[6]), "=r"(v[7])
        : "r"(taddr)
        : "memory");
}

// Shared-memory matrix descriptor, no swizzle (canonical core matrices of 8 rows x
// 16 bytes).  lbo/sbo in bytes.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;  // descriptor version for tcgen05
    return d;                 // base offset 0, layout type 0 (no swizzle)
}

// Instruction descriptor, kind::f16: fp16 A and B (both MN-major), fp32 accumulate.
__host__ __device__ __forceinline__ uint32_t idesc_f16_mn(int M, int N) {
    return (1u << 4)                          // D format f32
           | (0u << 7) | (0u << 10)           // A, B = f16
           | (1u << 15) | (1u << 16)          // A, B MN-major
           | ((uint32_t)(N >> 3) << 17)       // N / 8
           | ((uint32_t)(M >> 4) << 24);      // M / 16
}

// kind::f16 instruction descriptor with A in tensor memory (K-major) and B MN-major in
// shared memory; f32 accumulation.
__host__ __device__ __forceinline__ uint32_t idesc_f16_tmemA_mnB(int M, int N) {
    return (1u << 4)                          // D format f32
           | (0u << 7) | (0u << 10)           // A, B = f16
           | (0u << 15) | (1u << 16)          // A K-major, B MN-major
           | ((uint32_t)(N >> 3) << 17)       // N / 8
           | ((uint32_t)(M >> 4) << 24);      // M / 16
}

// int8 x4 -> two fp16x2 holding 1152 + b exactly (the byte xor 0x80 as the low byte
// of 0x64xx); the constant is removed after the accumulation.
__device__ __forceinline__ void i8x4_to_f16x4_biased(uint32_t x, uint32_t& lo, uint32_t& hi) {
    const uint32_t xs = x ^ 0x80808080u;
    lo = __byte_perm(xs, 0x64646464u, 0x5150);
    hi = __byte_perm(xs, 0x64646464u, 0x5352);
}

// The 16 bit pairs (2c, 2c + 1), c = 0..15, of x as fp16x2 words of 0 / 2^-16 (0x0100,
// a subnormal that the tensor cores multiply exactly): pair c sits in byte c / 4 of x
// shifted by 2 (c % 4); one byte permute of x >> s and x >> (s + 1) puts its two bits
// at bits 8 and 24, and a mask keeps them.
__device__ __forceinline__ void bits_to_e16_pairs(uint32_t x, uint32_t (&out)[16]) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const uint32_t xs = x >> (2 * r), xs1 = x >> (2 * r + 1);
#pragma unroll
        for (int byte = 0; byte < 4; ++byte)
            out[4 * byte + r] = __byte_perm(xs, xs1, (byte << 4) | ((4 + byte) << 12)) & 0x01000100u;
    }
}

// Two 0/1 bits (bit 0, bit 1 of v) -> fp16x2 {bit0, bit1} of 0.0 / 1.0.
__device__ __forceinline__ uint32_t bitpair_to_f16x2(uint32_t v) {
    return (((v & 3u) * 0x8001u) & 0x10001u) * 0x3C00u;
}

// int8 x4 -> two fp16x2 (exact): (b ^ 0x80) as the low byte of 0x64xx is 1024+b+128.
__device__ __forceinline__ void i8x4_to_f16x4(uint32_t x, uint32_t& lo, uint32_t& hi) {
    const uint32_t xs = x ^ 0x80808080u;
    uint32_t a = __byte_perm(xs, 0x64646464u, 0x5150);
    uint32_t b = __byte_perm(xs, 0x64646464u, 0x5352);
    const __half2 magic = __halves2half2(__ushort_as_half(0x6480), __ushort_as_half(0x6480));
    __half2 ha = __hsub2(*reinterpret_cast<__half2*>(&a), magic);
    __half2 hb = __hsub2(*reinterpret_cast<__half2*>(&b), magic);
    lo = *reinterpret_cast<uint32_t*>(&ha);
    hi = *reinterpret_cast<uint32_t*>(&hb);
}

// Two spike bits -> fp16x2 of 0.0 / 1.0 (bit0 -> low half).
__device__ __forceinline__ uint32_t bits2_to_f16x2(uint32_t x) {
    return ((x & 1u) * 0x3C00u) | (((x >> 1) & 1u) * 0x3C000000u);
}

// ------------------------------------------------------- linear launch ----
enum : int { EPI_KIND_INT = 0, EPI_KIND_F32 = 1, EPI_KIND_LOGITS = 2 };

// One output segment of a spiking linear launch: channels [0, n_out) of this segment
// come from W^T rows of stride ld_w and feed their own epilogue destinations.
struct LinSeg {
    const int8_t* wT;
    const float* scale;
    int ld_w;
    int n_out;
    int tile_begin;           // first tile index (of the launching kernel's tile width)
    uint32_t* bits;           // row-bit destination
    long long sb, st;         // word strides for token b and timestep t
    uint32_t* cm;             // [n_out][words(BT)] or null
    uint32_t* mask;           // [words(n_out)] or null
    float* cur;               // [BT][n_out] (logits kind: [B][n_out]) or null
    const float* res;         // [BT][n_out] or null
    const uint32_t* gate;     // row bits [BT][words(n_out)] or null
    int32_t* acc_out;         // [BT][n_out] or null
    int col0;                 // first accumulator column (k_linear_ts / k_linear_epi)
};

struct LinArgs {
    CUtensorMap tmap[3];      // per segment: W^T as a 2-D int8 tensor, box 128 x 64, 128B swizzle
    CUtensorMap gmap[3];      // the same tensor with a one-row box, for tile::gather4
    const uint32_t* in_cm;    // [d_in][words(BT)]
    const uint32_t* in_mask;  // [words(d_in)]
    const uint32_t* in_rows;  // [BT][words(d_in)] row bits of the same block, or null
    int d_in, BT, T, B, BTW;
    int nseg;
    LinSeg seg[3];
    int n_tiles;
    int kind, theta_i;
    float theta_f;
    int dense;                // every row of W^T, in order (DENSE mode)
    int auto_dense;           // AUTO mode: stream every row when >= 1/4 of them are active
    unsigned long long* stats;  // {rows fetched, synaptic ops}
    unsigned long long sops_dout;  // output channels counted per spike
    int* err;
    unsigned long long wait_ns;
    float* ws;                // split-K partials [nsplit][BT][n_tot]
    unsigned int* counters;   // per-tile arrival counters (zero between launches)
    int nsplit, n_tot;
    int desc_swap;            // debug: swap the LBO/SBO roles of the MMA descriptors
    int paired;               // gated MLP in one launch: seg[0] = gate, seg[1] = up (see k_linear_ts)
    int32_t* acc_g;           // k_linear_ts: partial sums, one slot per split: [split][columns][btp]
    int btp;                  // BT rounded up to a multiple of 4
    int epi_rb;               // k_linear_epi: 32-row blocks per CTA (1 or 2)
    long long acc_stride;     // words per split slot (columns x btp)
    int slot_mode;            // k_linear_ts: 1 = splits write slots, k_linear_epi runs the IF;
                              // 0 = cluster split-K through shared memory, IF in the kernel
    int slot_sync;            // slot mode: the splits of a tile meet at a counter in global
                              // memory, then each sums its slice of the slots and runs the IF
    unsigned* tickets;        // slot_sync: [2 * tiles] arrival / departure counters (zero)
    unsigned long long* dbg;  // debug: phase timestamps of CTA (0,0), or null
};

// Debug phase timestamp (thread 0 of CTA (0,0) only, when a.dbg is set).
#define NMDLM_TSTAMP(a, slot)                                                       \
    do {                                                                            \
        if ((a).dbg && blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0 &&    \
            (slot) < 4096)                                                          \
            (a).dbg[(slot)] = clock64();                                            \
    } while (0)
// Same, recorded by lane 0 of warp `w` of CTA (0,0).
#define NMDLM_TSTAMP_W(a, w, slot)                                                  \
    do {                                                                            \
        if ((a).dbg && blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 32 * (w) && \
            (slot) < 4096)                                                          \
            (a).dbg[(slot)] = clock64();                                            \
    } while (0)

// Per-CTA wall-clock stamp (global timer, ns) of event `ev` (0..3), recorded by thread 0
// of every CTA into word base + 4 * (linear CTA index) + ev of the debug buffer.
#define NMDLM_CSTAMP(a, base, ev)                                                    \
    do {                                                                             \
        if ((a).dbg && threadIdx.x == 0 && threadIdx.y == 0) {                       \
            const int cta_ = blockIdx.y * gridDim.x + blockIdx.x;                    \
            if ((base) + 4 * cta_ + (ev) < 4096)                                     \
                (a).dbg[(base) + 4 * cta_ + (ev)] = globaltimer_ns();                \
        }                                                                            \
    } while (0)

__device__ __forceinline__ int seg_of_tile(const LinArgs& a, int tile) {
    int s = 0;
    for (int i = 1; i < a.nseg; ++i)
        if (tile >= a.seg[i].tile_begin) s = i;
    return s;
}

// Epilogue of one warp over 32 consecutive channels lo0..lo0+31 of segment `s` for
// token b.  get(t) returns the exact int32 synaptic sum of row b*T+t for this lane.
// Accumulates this lane's column-mask words and any-spike flag.
template <int MAXT, int MAXW, class Get>
__device__ __forceinline__ void epi_token(const LinArgs& a, const LinSeg& s, int lo,
                                          bool valid, int b, Get get, uint32_t (&cmw)[MAXW],
                                          bool& any) {
    const int T = a.T;
    const int lane = threadIdx.x & 31;
    const int nw = words_of(s.n_out);
    const float sc = (valid && s.scale) ? s.scale[lo] : 0.0f;
    if (a.kind == EPI_KIND_LOGITS) {
        int sum = 0;
#pragma unroll
        for (int t = 0; t < MAXT; ++t)
            if (t < T) sum += get(t);
        if (valid) s.cur[(size_t)b * s.n_out + lo] = __fdiv_rn(__fmul_rn((float)sum, sc), (float)T);
        return;
    }
    int vi = 0;
    float vf = 0.0f;
#pragma unroll
    for (int t = 0; t < MAXT; ++t) {
        if (t >= T) break;
        const int bt = b * T + t;
        const int acc = get(t);
        bool sp;
        if (a.kind == EPI_KIND_INT) {
            const int h = vi + acc;
            sp = valid && h >= a.theta_i;
            vi = sp ? h - a.theta_i : h;
            if (valid && s.cur) s.cur[(size_t)bt * s.n_out + lo] = __fmul_rn((float)acc, sc);
        } else {
            float I = __fmul_rn((float)acc, sc);
            if (s.res) I = __fadd_rn(I, valid ? s.res[(size_t)bt * s.n_out + lo] : 0.0f);
            if (s.gate && valid) {
                const uint32_t gw = s.gate[(size_t)bt * nw + (lo >> 5)];
                if (!((gw >> (lo & 31)) & 1u)) I = 0.0f;
            }
            if (valid && s.cur) s.cur[(size_t)bt * s.n_out + lo] = I;
            const float h = __fadd_rn(vf, I);
            sp = valid && h >= a.theta_f;
            vf = sp ? __fsub_rn(h, a.theta_f) : h;
        }
        if (valid && s.acc_out) s.acc_out[(size_t)bt * s.n_out + lo] = acc;
        const uint32_t word = __ballot_sync(0xffffffffu, sp);
        // lane 0 holds the group's first channel: a group wholly past n_out writes nothing
        if (lane == 0 && (lo >> 5) < nw)
            s.bits[(long long)b * s.sb + (long long)t * s.st + (lo >> 5)] = word;
        if (sp) {
            cmw[bt >> 5] |= 1u << (bt & 31);
            any = true;
        }
    }
}

// The same epilogue for NTOK consecutive tokens b0..b0+NTOK-1 at once (tokens beyond
// a.B are skipped): the T-step IF recurrences of different tokens are independent, so
// interleaving them hides the latency of each step.  get(i, t) returns the sum of row
// (b0+i)*T+t for this lane.
template <int NTOK, int MAXW, class Get>
__device__ __forceinline__ void epi_tokens(const LinArgs& a, const LinSeg& s, int lo, bool valid,
                                           int b0, Get get, uint32_t (&cmw)[MAXW], bool& any) {
    const int T = a.T;
    const int lane = threadIdx.x & 31;
    const int nw = words_of(s.n_out);
    const float sc = (valid && s.scale) ? s.scale[lo] : 0.0f;
    const bool lead = lane == 0 && (lo >> 5) < nw;
    if (a.kind == EPI_KIND_LOGITS) {
#pragma unroll
        for (int i = 0; i < NTOK; ++i) {
            const int b = b0 + i;
            if (b >= a.B) break;
            int sum = 0;
            for (int t = 0; t < T; ++t) sum += get(i, t);
            if (valid) s.cur[(size_t)b * s.n_out + lo] = __fdiv_rn(__fmul_rn((float)sum, sc), (float)T);
        }
        return;
    }
    int vi[NTOK];
    float vf[NTOK];
#pragma unroll
    for (int i = 0; i < NTOK; ++i) { vi[i] = 0; vf[i] = 0.0f; }
    for (int t = 0; t < T; ++t) {
#pragma unroll
        for (int i = 0; i < NTOK; ++i) {
            const int b = b0 + i;
            if (b >= a.B) break;
            const int bt = b * T + t;
            const int acc = get(i, t);
            bool sp;
            if (a.kind == EPI_KIND_INT) {
                const int h = vi[i] + acc;
                sp = valid && h >= a.theta_i;
                vi[i] = sp ? h - a.theta_i : h;
                if (valid && s.cur) s.cur[(size_t)bt * s.n_out + lo] = __fmul_rn((float)acc, sc);
            } else {
                float I = __fmul_rn((float)acc, sc);
                if (s.res) I = __fadd_rn(I, valid ? s.res[(size_t)bt * s.n_out + lo] : 0.0f);
                if (s.gate && valid) {
                    const uint32_t gw = s.gate[(size_t)bt * nw + (lo >> 5)];
                    if (!((gw >> (lo & 31)) & 1u)) I = 0.0f;
                }
                if (valid && s.cur) s.cur[(size_t)bt * s.n_out + lo] = I;
                const float h = __fadd_rn(vf[i], I);
                sp = valid && h >= a.theta_f;
                vf[i] = sp ? __fsub_rn(h, a.theta_f) : h;
            }
            if (valid && s.acc_out) s.acc_out[(size_t)bt * s.n_out + lo] = acc;
            const uint32_t word = __ballot_sync(0xffffffffu, sp);
            if (lead) s.bits[(long long)b * s.sb + (long long)t * s.st + (lo >> 5)] = word;
            if (sp) {
#pragma unroll
                for (int w = 0; w < MAXW; ++w)
                    if (w == (bt >> 5)) cmw[w] |= 1u << (bt & 31);
                any = true;
            }
        }
    }
}

}  // namespace nmdlm
