// Host-side plumbing of libkronq: error strings, status mapping, device queries, and
// kq_check (reads the device error word written by kernels).
#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "kq_common.cuh"

namespace kq {

static thread_local char g_err[512] = "";
static std::atomic<uint64_t> g_launches{0};

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

void set_error(const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    std::vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
}

kq_status cuda_status(cudaError_t e, const char* where) {
    set_error("%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
    return KQ_ERR_CUDA;
}

int num_sms() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (!cache[dev]) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
        cache[dev] = n;
    }
    return cache[dev];
}

SideStream* side_stream(cudaStream_t caller) {
    // One side stream per (device, caller stream) and host thread, so calls on different
    // caller streams (concurrent layers) fork to different side streams.
    struct Entry {
        int dev;
        cudaStream_t caller;
        SideStream side;
    };
    constexpr int kMax = 64;
    static thread_local Entry table[kMax];
    static thread_local int used = 0;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
    for (int i = 0; i < used; ++i)
        if (table[i].dev == dev && table[i].caller == caller) return table[i].side.s ? &table[i].side : nullptr;
    if (used == kMax) return nullptr;   // beyond kMax caller streams: no fork, all work in order
    int prio = 0, least = 0, greatest = 0;
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamGetPriority(caller, &prio) != cudaSuccess ||
        cudaDeviceGetStreamPriorityRange(&least, &greatest) != cudaSuccess ||
        cudaStreamIsCapturing(caller, &cap) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    if (cap != cudaStreamCaptureStatusNone) return nullptr;   // made only outside a capture
    // Larger numbers are lower priorities: one level below the caller's.
    const int side_prio = prio < least ? prio + 1 : least;
    Entry& e = table[used++];
    e.dev = dev;
    e.caller = caller;
    e.side.tried = true;
    if (cudaStreamCreateWithPriority(&e.side.s, cudaStreamNonBlocking, side_prio) != cudaSuccess ||
        cudaStreamCreateWithPriority(&e.side.s2, cudaStreamNonBlocking, side_prio) != cudaSuccess ||
        cudaEventCreateWithFlags(&e.side.ev[0], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&e.side.ev[1], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&e.side.ev2[0], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&e.side.ev2[1], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&e.side.ev2[2], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&e.side.ev2[3], cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        e.side.s = nullptr;
    }
    return e.side.s ? &e.side : nullptr;
}

// Waits on an mbarrier that nothing ever arrives on, with the bounded wait every pipeline
// kernel uses, and reports the timeout the way those kernels do.
__global__ void selftest_timeout_kernel(int* info, uint64_t limit_ns) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0 && !mbar_wait(&bar, 0, &abort_flag, limit_ns)) record_error(info, -KQ_ERR_TIMEOUT);
}

}  // namespace kq

extern "C" kq_status kq_selftest_timeout(int* info, int64_t limit_us, kq_stream_t stream_) {
    if (!info || limit_us < 1 || limit_us > 2000000) {
        kq::set_error("kq_selftest_timeout: info must be a device int and 1 <= limit_us <= 2e6");
        return KQ_ERR_INVALID_ARG;
    }
    kq::selftest_timeout_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream_)>>>(
        info, static_cast<uint64_t>(limit_us) * 1000u);
    KQ_LAUNCH_CHECK("selftest_timeout_kernel");
    return KQ_OK;
}

namespace kq {
namespace {
// mismatches (+)= the number of i with div_rn(a_i, b_i, div_recip(b_i)) != __fdiv_rn(a_i, b_i)
// bit for bit.
__global__ void selftest_div_kernel(const float* __restrict__ a, const float* __restrict__ b, int64_t n,
                                    unsigned long long* __restrict__ mismatches) {
    unsigned long long bad = 0;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const float x = a[i], y = b[i];
        bad += __float_as_uint(div_rn(x, y, div_recip(y))) != __float_as_uint(__fdiv_rn(x, y));
    }
    for (int o = 16; o > 0; o >>= 1) bad += __shfl_xor_sync(0xffffffffu, bad, o);
    if ((threadIdx.x & 31) == 0 && bad) atomicAdd(mismatches, bad);
}
}  // namespace
}  // namespace kq

extern "C" kq_status kq_selftest_div(const float* a, const float* b, int64_t n, unsigned long long* mismatches,
                                     kq_stream_t stream_) {
    if (!a || !b || !mismatches || n < 0) {
        kq::set_error("kq_selftest_div: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (n == 0) return KQ_OK;
    const int64_t blocks = std::min<int64_t>(kq::cdiv(n, 256), static_cast<int64_t>(kq::num_sms()) * 8);
    kq::selftest_div_kernel<<<static_cast<unsigned>(blocks), 256, 0, reinterpret_cast<cudaStream_t>(stream_)>>>(
        a, b, n, mismatches);
    KQ_LAUNCH_CHECK("selftest_div_kernel");
    return KQ_OK;
}

extern "C" const char* kq_last_error(void) { return kq::g_err; }

extern "C" const char* kq_status_name(int s) {
    switch (s) {
        case KQ_OK: return "KQ_OK";
        case KQ_ERR_INVALID_ARG: return "KQ_ERR_INVALID_ARG";
        case KQ_ERR_UNSUPPORTED: return "KQ_ERR_UNSUPPORTED";
        case KQ_ERR_NOT_PD: return "KQ_ERR_NOT_PD";
        case KQ_ERR_CUDA: return "KQ_ERR_CUDA";
        case KQ_ERR_TIMEOUT: return "KQ_ERR_TIMEOUT";
        case KQ_ERR_WORKSPACE: return "KQ_ERR_WORKSPACE";
        case KQ_ERR_NONFINITE: return "KQ_ERR_NONFINITE";
        default: return "KQ_ERR_UNKNOWN";
    }
}

extern "C" int kq_version(void) { return 100; }

extern "C" uint64_t kq_launch_count(void) { return kq::g_launches.load(std::memory_order_relaxed); }

extern "C" kq_status kq_graph_instantiate(void* graph, int use_node_priority, void** exec) {
    if (!graph || !exec) {
        kq::set_error("kq_graph_instantiate: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    cudaGraphExec_t e = nullptr;
    const unsigned long long flags = use_node_priority ? cudaGraphInstantiateFlagUseNodePriority : 0ull;
    KQ_CUDA(cudaGraphInstantiateWithFlags(&e, static_cast<cudaGraph_t>(graph), flags));
    *exec = e;
    return KQ_OK;
}

extern "C" kq_status kq_graph_launch(void* exec, kq_stream_t stream) {
    if (!exec) {
        kq::set_error("kq_graph_launch: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    KQ_CUDA(cudaGraphLaunch(static_cast<cudaGraphExec_t>(exec), reinterpret_cast<cudaStream_t>(stream)));
    return KQ_OK;
}

extern "C" kq_status kq_graph_exec_destroy(void* exec) {
    if (exec) KQ_CUDA(cudaGraphExecDestroy(static_cast<cudaGraphExec_t>(exec)));
    return KQ_OK;
}

extern "C" kq_status kq_check(int* info, int reset, int* pivot_out, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    KQ_CUDA(cudaStreamSynchronize(stream));
    int v = 0;
    if (info) {
        KQ_CUDA(cudaMemcpy(&v, info, sizeof(int), cudaMemcpyDeviceToHost));
        if (reset && v != 0) KQ_CUDA(cudaMemset(info, 0, sizeof(int)));
    }
    if (pivot_out) *pivot_out = v;
    if (v == 0) return KQ_OK;
    if (v > 0) {
        kq::set_error("non-positive pivot at index %d", v);
        return KQ_ERR_NOT_PD;
    }
    kq::set_error("kernel reported %s", kq_status_name(-v));
    return static_cast<kq_status>(-v);
}

// ------------------------------------------------------------------ debug build
namespace kq {
namespace {
// buf[i] = i for i in [0, n] under a bounds check against n: buf holds n + 1 floats, so the
// last write stays inside it in every build; the debug build's check skips it and records
// this line.
__global__ void selftest_bounds_kernel(float* __restrict__ buf, int64_t n) {
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i <= n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x)
        if (KQ_IN_RANGE(i, n)) buf[i] = static_cast<float>(i);
}
}  // namespace

KQ_DEBUG_UNIT(api)
int debug_read_syrk(int);
int debug_read_biip(int);
int debug_read_chol(int);
int debug_read_obs(int);
int debug_read_trail_tc(int);
int debug_read_gptaq(int);
int debug_read_infer(int);
int debug_read_check(int);
}  // namespace kq

extern "C" int kq_debug_build(void) {
#ifdef KQ_DEBUG
    return 1;
#else
    return 0;
#endif
}

extern "C" kq_status kq_debug_status(int* unit, int* line, int reset) {
    using Reader = int (*)(int);
    static const Reader readers[] = {kq::debug_read_api,      kq::debug_read_syrk,  kq::debug_read_biip,
                                     kq::debug_read_chol,     kq::debug_read_obs,   kq::debug_read_trail_tc,
                                     kq::debug_read_gptaq,    kq::debug_read_infer, kq::debug_read_check};
    KQ_CUDA(cudaDeviceSynchronize());
    int u = -1, l = 0;
    for (int k = 0; k < static_cast<int>(sizeof(readers) / sizeof(readers[0])); ++k) {
        const int v = readers[k](reset);
        if (v < 0) {
            kq::set_error("kq_debug_status: cannot read the debug word of unit %d", k);
            return KQ_ERR_CUDA;
        }
        if (v > 0 && u < 0) {
            u = k;
            l = v;
        }
    }
    if (unit) *unit = u;
    if (line) *line = l;
    return KQ_OK;
}

extern "C" kq_status kq_selftest_bounds(float* buf, int64_t n, kq_stream_t stream_) {
    if (!buf || n < 1) {
        kq::set_error("kq_selftest_bounds: buf must hold n + 1 floats, n >= 1");
        return KQ_ERR_INVALID_ARG;
    }
    const int64_t blocks = std::min<int64_t>(kq::cdiv(n + 1, 256), 1024);
    kq::selftest_bounds_kernel<<<static_cast<unsigned>(blocks), 256, 0, reinterpret_cast<cudaStream_t>(stream_)>>>(
        buf, n);
    KQ_LAUNCH_CHECK("selftest_bounds_kernel");
    return KQ_OK;
}
