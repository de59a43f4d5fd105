// Shared device/host helpers of libkronq: status handling, bounded waits, and thin
// inline-PTX wrappers for mbarrier, TMA (cp.async.bulk.tensor) and tcgen05 (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "../../include/kronq.h"

namespace kq {

// ----------------------------------------------------------------------------- host side
void set_error(const char* fmt, ...);
kq_status cuda_status(cudaError_t e, const char* where);

#define KQ_CUDA(call)                                                   \
    do {                                                                \
        cudaError_t _e = (call);                                        \
        if (_e != cudaSuccess) return ::kq::cuda_status(_e, #call);    \
    } while (0)

// Every kernel launch is followed by this check, which also counts the launch.
void count_launch();
#define KQ_LAUNCH_CHECK(what)                                           \
    do {                                                                \
        ::kq::count_launch();                                           \
        cudaError_t _e = cudaGetLastError();                            \
        if (_e != cudaSuccess) return ::kq::cuda_status(_e, what);      \
    } while (0)

inline int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Returns from the enclosing function when a kq_status expression is not KQ_OK.
#define KQ_TRY(expr)                                                    \
    do {                                                                \
        const kq_status _s = (expr);                                    \
        if (_s != KQ_OK) return _s;                                     \
    } while (0)

// Runs the set-up f (returning kq_status) once for each device it is called with current:
// kernel attributes such as the dynamic shared-memory limit belong to the device they were
// set on, so a process that drives several GPUs sets them on each. A failed set-up is
// tried again on the next call; two threads may both run it (it only repeats idempotent
// settings).
template <typename F>
inline kq_status once_per_device(std::atomic<uint64_t>& done, F&& f) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return f();
    const uint64_t bit = uint64_t{1} << dev;
    if (done.load(std::memory_order_acquire) & bit) return KQ_OK;
    const kq_status s = f();
    if (s == KQ_OK) done.fetch_or(bit, std::memory_order_acq_rel);
    return s;
}

// Number of SMs of the current device (cached per device).
int num_sms();

// A library-owned stream for work that can run beside the caller's stream. An entry point
// forks to it with an event recorded on the caller's stream and joins back (the caller's
// stream waits on an event recorded on it) before returning, so the caller sees one
// ordered stream, and a CUDA graph captured from the caller's stream records both
// branches. One per host thread, device and caller stream (so concurrent calls on
// different caller streams fork to different side streams); its priority is one level below
// the caller's stream. side_stream returns nullptr (the caller then runs everything on its
// own stream) when the stream cannot be made, or when the caller's stream is being captured
// and its side stream does not exist yet.
struct SideStream {
    cudaStream_t s;
    cudaEvent_t ev[2];
    cudaStream_t s2;        // a second side stream (same priority) for long-running work
    cudaEvent_t ev2[4];
    bool tried;
};
SideStream* side_stream(cudaStream_t caller);

// ------------------------------------------------------------------ debug bounds checks
// In the debug build (libkronq_debug.so, compiled with -DKQ_DEBUG), KQ_IN_RANGE(i, n) checks
// 0 <= i < n for an index into a buffer of n elements before the kernel accesses it: a
// failed check records the source line in this translation unit's debug word (the first
// failure wins) and the guarded access is skipped, so a wrong index shows up as a status
// (kq_debug_status) instead of a fault. In the normal build it is `true` and costs
// nothing. Each .cu file ends with KQ_DEBUG_UNIT(name), which defines the host function
// that reads and clears that file's word.
#ifdef KQ_DEBUG
namespace {
__device__ int g_kq_debug_line;
}
__device__ __forceinline__ bool debug_in_range(long long i, long long n, int line) {
    if (i >= 0 && i < n) return true;
    atomicCAS(&g_kq_debug_line, 0, line);
    return false;
}
#define KQ_IN_RANGE(i, n) (::kq::debug_in_range(static_cast<long long>(i), static_cast<long long>(n), __LINE__))
#define KQ_DEBUG_UNIT(name)                                                                    \
    int debug_read_##name(int reset) {                                                         \
        int v = 0;                                                                             \
        if (cudaMemcpyFromSymbol(&v, g_kq_debug_line, sizeof(int)) != cudaSuccess) return -1;  \
        if (reset && v) {                                                                      \
            const int z = 0;                                                                   \
            if (cudaMemcpyToSymbol(g_kq_debug_line, &z, sizeof(int)) != cudaSuccess) return -1; \
        }                                                                                      \
        return v;                                                                              \
    }
#else
#define KQ_IN_RANGE(i, n) true
#define KQ_DEBUG_UNIT(name) \
    int debug_read_##name(int) { return 0; }
#endif

// ------------------------------------------------------------------------- device side
// Device error words: info == 0 ok; > 0 a 1-based pivot index (Cholesky); < 0 minus a
// kq_status recorded by a kernel (for example -KQ_ERR_TIMEOUT).
__device__ __forceinline__ void record_error(int* info, int code) {
    if (info) atomicCAS(info, 0, code);
}

// Correctly rounded a / b from y = __frcp_rn(b), after Markstein's theorem (P. W. Markstein,
// "Computation of elementary functions on the IBM RISC System/6000 processor", IBM J. Res.
// Dev. 34(1), 1990): when y is within half an ulp of 1/b and q within one ulp of a/b, the
// residual a - b q is exact under an fma and RN(q + (a - b q) y) = RN(a / b). q0 = RN(a y)
// can be 1.5 ulp off, so one correction brings it within one ulp and a second one rounds
// correctly; a = +-0 returns q0 (its sign is right). The theorem needs every intermediate
// normal: div_recip gives y = 0 for a divisor outside [2^-60, 2^60], and div_rn_fast_ok
// tells whether (a, y) is inside the range where div_rn_fast is exact; div_rn falls back to
// __fdiv_rn outside it. The OBS sweep runs div_rn_fast (two dependent fma pairs on its
// sequential chain, the reciprocal computed once per divisor) and redoes a row group with
// __fdiv_rn when div_rn_fast_ok failed anywhere in it.
__device__ __forceinline__ float div_recip(float b) {
    const float ab = fabsf(b);
    return (ab >= 0x1p-60f && ab <= 0x1p60f) ? __frcp_rn(b) : 0.0f;
}
__device__ __forceinline__ bool div_rn_fast_ok(float a, float y) {
    const float aa = fabsf(a);
    return y != 0.0f && (a == 0.0f || (aa >= 0x1p-60f && aa <= 0x1p60f));
}
__device__ __forceinline__ float div_rn_fast(float a, float b, float y) {
    const float q0 = __fmul_rn(a, y);
    const float q1 = __fmaf_rn(__fmaf_rn(-q0, b, a), y, q0);
    const float q2 = __fmaf_rn(__fmaf_rn(-q1, b, a), y, q1);
    return a == 0.0f ? q0 : q2;
}
__device__ __forceinline__ float div_rn(float a, float b, float y) {
    return div_rn_fast_ok(a, y) ? div_rn_fast(a, b, y) : __fdiv_rn(a, b);
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Every wait on an mbarrier gives up after this long and reports KQ_ERR_TIMEOUT.
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s
constexpr uint32_t kWaitLimitIters = 1u << 30;

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
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
// Bounded wait for the phase with the given parity. Returns false (and raises *abort)
// when the limit is reached or another thread has already raised *abort.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                          uint64_t limit_ns = kWaitLimitNs) {
    if (mbar_try_wait(bar, parity)) return true;
    uint64_t t0 = global_timer_ns();
    for (uint32_t it = 0; it < kWaitLimitIters; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
        if ((it & 255u) == 255u && global_timer_ns() - t0 > limit_ns) break;
    }
    *abort = 1;
    return false;
}

// --------------------------------------------------------------------------- TMA
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* m) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* m, uint64_t* bar, int x,
                                            int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(smem_u32(bar)), "r"(x), "r"(y)
        : "memory");
}

// ------------------------------------------------------------------ cp.async (LDGSTS)
// 16-byte asynchronous global->shared copy; bytes beyond src_bytes (0..16) are zero-filled.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem)), "l"(gmem),
                 "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// ------------------------------------------------------------------------- tcgen05
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(dst_smem)),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, fp32 accumulate).
__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                           uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrive once on `bar` when every tcgen05.mma issued so far by this thread completed.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_u32(bar))
        : "memory");
}
__device__ __forceinline__ void tc_wait_ld() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// 32 consecutive fp32 columns of the calling warp's 32 TMEM lanes (one row per thread).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// ------------------------------------------------------- pairs of CTAs (cta_group::2)
// A cluster of two CTAs whose tcgen05.mma (M = 256, issued by CTA 0) reads both CTAs'
// operands and writes each CTA's 128 rows of the accumulator into its own tensor memory.
// Every tcgen05 instruction of such a kernel uses cta_group::2.
__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// Address of the same shared variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
    uint32_t d;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(addr), "r"(rank));
    return d;
}
__device__ __forceinline__ void cluster_barrier() {
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cl(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait (as mbar_wait) with cluster scope, for barriers the peer CTA arrives on.
__device__ __forceinline__ bool mbar_wait_cl(uint64_t* bar, uint32_t parity, volatile int* abort) {
    if (mbar_try_wait_cl(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 0; it < kWaitLimitIters; ++it) {
        if (mbar_try_wait_cl(bar, parity)) return true;
        if (*abort) return false;
        if ((it & 255u) == 255u && global_timer_ns() - t0 > kWaitLimitNs) break;
    }
    *abort = 1;
    return false;
}
// TMA load into this CTA's shared memory whose transaction bytes land on the mbarrier at
// cluster address `bar` (this CTA's or the peer's).
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* m, uint32_t bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(x), "r"(y)
        : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// Arrive once on `bar` (same offset) in both CTAs of the pair when the pair's MMAs issued
// so far have completed.
__device__ __forceinline__ void tc_commit_pair(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            smem_u32(bar)),
        "h"(static_cast<uint16_t>(3))
        : "memory");
}

// Shared-memory matrix descriptor (tcgen05): start, leading/stride byte offsets, version 1,
// 128-byte swizzle. Addresses and offsets are in bytes.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
    d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
    d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
    d |= 1ull << 46;   // descriptor version for tcgen05
    d |= 2ull << 61;   // SWIZZLE_128B
    return d;
}

// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both MN-major.
__host__ __device__ constexpr uint32_t idesc_bf16_mn_major(int M, int N) {
    return (1u << 4)                               // D format: f32
           | (1u << 7)                             // A format: bf16
           | (1u << 10)                            // B format: bf16
           | (1u << 15)                            // A MN-major
           | (1u << 16)                            // B MN-major
           | (static_cast<uint32_t>(N >> 3) << 17) // N / 8
           | (static_cast<uint32_t>(M >> 4) << 24);// M / 16
}

}  // namespace kq
