// GPTAQ drift correction: the matrix P of Proposition 1 and Algorithm 2,
//   P = alpha ((D' L) o M_U) L^T,
// with D' the rescaled, rotated drift statistic (Algorithm 1), L the lower factor of the
// damped H^-1 = L L^T (kq_chol_inv) and M_U the strictly upper-triangular mask. The output
// is Pt = P^T (row-major, strictly lower triangular), the layout the sweep reads.
//
// Two triangular GEMMs on the 5th-generation tensor cores with fp32-accurate products from
// the 3xTF32 split (x = x_hi + x_lo, x_hi rounded to tf32; a b ~= a_lo b_hi + a_hi b_lo +
// a_hi b_hi, fp32 accumulation in TMEM):
//   GEMM 1  A1[i][k] = sum_m D'[i][m] L[m][k] for k > i (else 0). Only the tiles on or above
//           the diagonal exist, and since L[m][k] = 0 for m < k the sum starts at the
//           tile's first column: m in [128 kt, n). Operands K-major: D' rows, and rows of
//           R = L^T (a transposing split). The epilogue writes A1 already split.
//   GEMM 2  Pt[j][i] = alpha sum_k L[j][k] A1[i][k] over k in (i, j]; tiles on or below
//           the diagonal, k in [128 it, 128 jt + 128). Operands: L rows and A1 rows.
// One CTA per 128 x 128 tile, the tiles with the longest K first. Warp 0 issues the TMA
// loads (hi and lo of both operands, 32-wide k slabs, 128-byte swizzle) into a 3-stage
// ring, warp 1 the MMAs (M 128, N 128, K 8, three per k step) into one TMEM accumulator,
// warps 2..5 read it back (one row per thread) and write the tile. Every mbarrier wait is
// bounded; a timeout sets -KQ_ERR_TIMEOUT in *info and the CTA drains before it exits.
#include <algorithm>
#include <cstring>

#include "trail_tc.cuh"

namespace kq {
namespace {

constexpr int PBM = 128;                 // tile rows and columns
constexpr int PBK = 32;                  // k per slab
constexpr int P_STAGES = 3;
constexpr int P_SLAB = PBM * PBK * 4;    // 16 KB: one operand part (hi or lo) of one slab
constexpr int P_STAGE = 4 * P_SLAB;      // A hi, A lo, B hi, B lo
constexpr int P_THREADS = 192;           // TMA, MMA, 4 epilogue warps
constexpr int P_SMEM = P_STAGES * P_STAGE + 1024 + 256;

// Tile t of GEMM 1 (upper tiles, longest K first): column tile kt ascending, row tile it <= kt.
__device__ __forceinline__ void upper_tile(int t, int* it, int* kt) {
    int k = 0;
    while (t >= k + 1) {
        t -= k + 1;
        ++k;
    }
    *kt = k;
    *it = t;
}

// Tile t of GEMM 2 (lower tiles, longest K first): offset jt - it from N - 1 down to 0.
__device__ __forceinline__ void lower_tile(int t, int N, int* jt, int* it) {
    int dlt = N - 1;
    while (t >= N - dlt) {
        t -= N - dlt;
        --dlt;
    }
    *it = t;
    *jt = t + dlt;
}

__device__ __forceinline__ bool wait_quiet(uint64_t* bar, uint32_t parity) {
    int dummy = 0;
    return mbar_wait(bar, parity, &dummy);
}

// SECOND = false: GEMM 1 (writes Ah, Al). SECOND = true: GEMM 2 (writes Pt).
template <bool SECOND>
__global__ void __launch_bounds__(P_THREADS, 1)
gptaq_gemm_kernel(const __grid_constant__ CUtensorMap mAh, const __grid_constant__ CUtensorMap mAl,
                  const __grid_constant__ CUtensorMap mBh, const __grid_constant__ CUtensorMap mBl, int n,
                  float alpha, float* __restrict__ out_hi, float* __restrict__ out_lo, int* info) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + P_STAGES * P_STAGE);
    uint64_t* empty = full + P_STAGES;
    uint64_t* tfull = empty + P_STAGES;
    uint64_t* mma_done = tfull + 1;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int N = (n + PBM - 1) / PBM;
    int rt, ct;   // output row tile, column tile
    int k_lo, k_hi;
    if (!SECOND) {
        upper_tile(blockIdx.x, &rt, &ct);
        k_lo = ct * PBM;
        k_hi = n;
    } else {
        lower_tile(blockIdx.x, N, &rt, &ct);
        k_lo = ct * PBM;
        k_hi = min(n, rt * PBM + PBM);
    }
    const int r0 = rt * PBM, c0 = ct * PBM;
    const int nslab = (k_hi - k_lo + PBK - 1) / PBK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < P_STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(tfull, 1);
        mbar_init(mma_done, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, PBM);
        tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&mAh);
        tma_prefetch_desc(&mAl);
        tma_prefetch_desc(&mBh);
        tma_prefetch_desc(&mBl);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            int issued = 0;
            for (int s = 0; s < nslab; ++s) {
                const int st = s % P_STAGES;
                const uint32_t u = static_cast<uint32_t>(s / P_STAGES);
                if (!mbar_wait(&empty[st], (u & 1u) ^ 1u, abort_flag)) break;
                mbar_arrive_expect_tx(&full[st], P_STAGE);
                uint8_t* base = smem + st * P_STAGE;
                const int x = k_lo + s * PBK;
                tma_load_2d(base, &mAh, &full[st], x, r0);
                tma_load_2d(base + P_SLAB, &mAl, &full[st], x, r0);
                tma_load_2d(base + 2 * P_SLAB, &mBh, &full[st], x, c0);
                tma_load_2d(base + 3 * P_SLAB, &mBl, &full[st], x, c0);
                issued = s + 1;
            }
            for (int s = (issued > P_STAGES ? issued - P_STAGES : 0); s < issued; ++s)
                wait_quiet(&full[s % P_STAGES], static_cast<uint32_t>(s / P_STAGES) & 1u);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_tf32_k_major(PBM, PBM);
            bool ok = true;
            for (int s = 0; s < nslab; ++s) {
                const int st = s % P_STAGES;
                if (!mbar_wait(&full[st], static_cast<uint32_t>(s / P_STAGES) & 1u, abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a_hi = smem_u32(smem + st * P_STAGE);
                const uint32_t a_lo = a_hi + P_SLAB;
                const uint32_t b_hi = a_hi + 2 * P_SLAB;
                const uint32_t b_lo = a_hi + 3 * P_SLAB;
#pragma unroll
                for (int kk = 0; kk < PBK / 8; ++kk) {
                    const uint32_t ko = static_cast<uint32_t>(kk * 32);
                    const uint64_t dah = smem_desc_sw128(a_hi + ko, 16, 1024);
                    const uint64_t dal = smem_desc_sw128(a_lo + ko, 16, 1024);
                    const uint64_t dbh = smem_desc_sw128(b_hi + ko, 16, 1024);
                    const uint64_t dbl = smem_desc_sw128(b_lo + ko, 16, 1024);
                    tc_mma_tf32(tmem, dal, dbh, idesc, (s > 0 || kk > 0) ? 1u : 0u);
                    tc_mma_tf32(tmem, dah, dbl, idesc, 1u);
                    tc_mma_tf32(tmem, dah, dbh, idesc, 1u);
                }
                tc_commit(&empty[st]);
            }
            if (ok && nslab > 0) tc_commit(tfull);
            tc_commit(mma_done);
            wait_quiet(mma_done, 0);
        }
    } else {
        // epilogue: warp w reads TMEM lanes 32 (w & 3) .. + 31, thread = one output row
        const int q = warp & 3;
        const int rloc = q * 32 + lane;
        const int row = r0 + rloc;
        bool ok = nslab == 0 || mbar_wait(tfull, 0, abort_flag);
        ok = __all_sync(0xffffffffu, ok) && !*abort_flag;
        if (ok) {
            tc_fence_after();
#pragma unroll 1
            for (int p = 0; p < PBM / 32; ++p) {
                float v[32];
                if (nslab > 0) {
                    tmem_ld32(tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(p * 32), v);
                    tc_wait_ld();
                } else {
#pragma unroll
                    for (int c = 0; c < 32; ++c) v[c] = 0.0f;
                }
                const int cbase = c0 + p * 32;
                if (row < n) {
                    if (!SECOND) {
                        // A1 = (D' L) o M_U, kept where column > row, written as tf32 hi / lo
                        float* ph = out_hi + static_cast<int64_t>(row) * n + cbase;
                        float* pl = out_lo + static_cast<int64_t>(row) * n + cbase;
#pragma unroll
                        for (int c = 0; c < 32; ++c) {
                            if (cbase + c < n) {
                                const float x = (cbase + c > row) ? v[c] : 0.0f;
                                const float h = tf32_hi(x);
                                ph[c] = h;
                                pl[c] = x - h;
                            }
                        }
                    } else {
                        // Pt[j][i] = alpha (L A1^T)[j][i], kept where i < j
                        float* pp = out_hi + static_cast<int64_t>(row) * n + cbase;
#pragma unroll
                        for (int c = 0; c < 32; ++c)
                            if (cbase + c < n) pp[c] = (cbase + c < row) ? alpha * v[c] : 0.0f;
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) record_error(info, -KQ_ERR_TIMEOUT);
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, PBM);
    }
}

// Rh[k][m] = tf32(L[m][k]), Rl = L[m][k] - Rh[k][m]: the split of R = L^T, transposed
// through a 32 x 33 shared tile. Block (32, 8).
__global__ void split_transpose_kernel(const float* __restrict__ L, int64_t n, float* __restrict__ Rh,
                                       float* __restrict__ Rl) {
    __shared__ float t[32][33];
    const int64_t m0 = static_cast<int64_t>(blockIdx.y) * 32, k0 = static_cast<int64_t>(blockIdx.x) * 32;
    for (int r = threadIdx.y; r < 32; r += 8) {
        const int64_t m = m0 + r, k = k0 + threadIdx.x;
        t[r][threadIdx.x] = (m < n && k < n) ? L[m * n + k] : 0.0f;
    }
    __syncthreads();
    for (int r = threadIdx.y; r < 32; r += 8) {
        const int64_t k = k0 + r, m = m0 + threadIdx.x;
        if (k < n && m < n) {
            const float x = t[threadIdx.x][r];
            const float h = tf32_hi(x);
            Rh[k * n + m] = h;
            Rl[k * n + m] = x - h;
        }
    }
}

inline size_t mat_bytes(int64_t n) { return (static_cast<size_t>(n) * n * sizeof(float) + 255) & ~static_cast<size_t>(255); }

}  // namespace

KQ_DEBUG_UNIT(gptaq)
}  // namespace kq

using namespace kq;

extern "C" size_t kq_gptaq_p_workspace(int64_t n) {
    if (n < 1) return 0;
    return 6 * mat_bytes(n) + 256;
}

extern "C" kq_status kq_gptaq_p(const float* Dp, const float* Lt, int64_t n, float alpha, float* Pt, int* info,
                                void* ws, size_t ws_bytes, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!Dp || !Lt || !Pt || n < 1 || n > 65536) {
        set_error("kq_gptaq_p: invalid arguments (n=%lld)", (long long)n);
        return KQ_ERR_INVALID_ARG;
    }
    if ((n % 4) != 0 || (reinterpret_cast<uintptr_t>(Dp) & 15u) || (reinterpret_cast<uintptr_t>(Lt) & 15u)) {
        set_error("kq_gptaq_p: n must be a multiple of 4 and D', Lt 16-byte aligned");
        return KQ_ERR_UNSUPPORTED;
    }
    if (!ws || ws_bytes < kq_gptaq_p_workspace(n) || (reinterpret_cast<uintptr_t>(ws) & 255u)) {
        set_error("kq_gptaq_p: workspace must be 256-byte aligned and hold %zu bytes", kq_gptaq_p_workspace(n));
        return KQ_ERR_WORKSPACE;
    }
    const size_t mb = mat_bytes(n);
    uint8_t* w8 = static_cast<uint8_t*>(ws);
    float* X0 = reinterpret_cast<float*>(w8);            // D'_hi, later L_hi
    float* X1 = reinterpret_cast<float*>(w8 + mb);       // D'_lo, later L_lo
    float* Rh = reinterpret_cast<float*>(w8 + 2 * mb);
    float* Rl = reinterpret_cast<float*>(w8 + 3 * mb);
    float* Ah = reinterpret_cast<float*>(w8 + 4 * mb);   // A1 = (D' L) o M_U, split
    float* Al = reinterpret_cast<float*>(w8 + 5 * mb);
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(gptaq_gemm_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, P_SMEM));
        KQ_CUDA(cudaFuncSetAttribute(gptaq_gemm_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, P_SMEM));
        return KQ_OK;
    }));
    const int64_t N = cdiv(n, PBM);
    const int64_t ntiles = N * (N + 1) / 2;
    kq_status st = split_tf32(Dp, n * n, X0, X1, stream);
    if (st != KQ_OK) return st;
    split_transpose_kernel<<<dim3(static_cast<unsigned>(cdiv(n, 32)), static_cast<unsigned>(cdiv(n, 32))), dim3(32, 8),
                             0, stream>>>(Lt, n, Rh, Rl);
    KQ_LAUNCH_CHECK("split_transpose_kernel");
    CUtensorMap ma, mal, mb_, mbl;
    if ((st = make_f32_map(&ma, X0, n, n, PBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&mal, X1, n, n, PBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&mb_, Rh, n, n, PBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&mbl, Rl, n, n, PBM)) != KQ_OK) return st;
    gptaq_gemm_kernel<false><<<static_cast<unsigned>(ntiles), P_THREADS, P_SMEM, stream>>>(ma, mal, mb_, mbl,
                                                                                           static_cast<int>(n), 1.0f,
                                                                                           Ah, Al, info);
    KQ_LAUNCH_CHECK("gptaq_gemm_kernel<1>");
    // GEMM 2: A = L rows (split into the buffers D' used), B = A1 rows
    if ((st = split_tf32(Lt, n * n, X0, X1, stream)) != KQ_OK) return st;
    if ((st = make_f32_map(&mb_, Ah, n, n, PBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&mbl, Al, n, n, PBM)) != KQ_OK) return st;
    KQ_CUDA(cudaMemsetAsync(Pt, 0, sizeof(float) * n * n, stream));
    gptaq_gemm_kernel<true><<<static_cast<unsigned>(ntiles), P_THREADS, P_SMEM, stream>>>(ma, mal, mb_, mbl,
                                                                                          static_cast<int>(n), alpha,
                                                                                          Pt, nullptr, info);
    KQ_LAUNCH_CHECK("gptaq_gemm_kernel<2>");
    return KQ_OK;
}
