// Stage 1: Kronecker-factor accumulation H (+)= A^T A on the 5th-generation tensor cores.
//
// Paper: Sec. 2.1 Eq. (ptq_obj) (H_X = X X^T, tokens as columns there), Sec. 3.1 Eq. (kfac)
// (H = H_X (x) H_G), Algorithm 1 ("online statistics"). Tokens are rows here, so the
// factor is A^T A for A [T x d].
//
// Design (sm_103a):
//   * one CTA per 128 x 256 output tile of the lower triangle (row tile i, column tile j,
//     128 i + 127 >= 256 j); the tile is mirrored into the upper triangle on write-out;
//   * warp 0 issues TMA loads of 64-token x 64-feature boxes (128-byte swizzle) into a
//     4-stage ring; both operands are slices of the same A, read MN-major (features
//     contiguous), so no transpose pass is needed;
//   * warp 1 allocates 512 TMEM columns and issues tcgen05.mma kind::f16 (bf16 x bf16 ->
//     fp32, M = 128, N = 256, K = 16) into one of two 256-column accumulators;
//   * warps 2..9 drain an accumulator every KQ_SYRK_CHUNK_TOKENS tokens into an fp32
//     running sum held in registers (each thread owns 128 columns of one row), while the
//     MMAs continue into the other accumulator. This bounds how many tensor-core
//     additions any fp32 partial sum sees;
//   * every mbarrier wait is bounded (kq::mbar_wait); a timeout is reported as
//     -KQ_ERR_TIMEOUT in *info and the CTA drains its own copies and MMAs before exit.
#include <cstdio>
#include <cstdlib>
#include <cstring>

#include "kq_common.cuh"

namespace kq {
namespace {

constexpr int BM = 128;   // output rows per tile (MMA M, TMEM lanes)
constexpr int BN = 256;   // output columns per tile (MMA N)
constexpr int BK = 64;    // tokens per pipeline stage
constexpr int STAGES = 4;
constexpr int BOX_BYTES = BK * 64 * 2;          // one 64-token x 64-feature bf16 box
constexpr int A_BYTES = BK * BM * 2;            // 16 KB
constexpr int B_BYTES = BK * BN * 2;            // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;  // 48 KB
constexpr int NUM_THREADS = 320;                // 10 warps
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256;
constexpr uint32_t TMEM_COLS = 512;
// Canonical MN-major SW128 layout: atoms of 64 features x 8 tokens (1 KB). Along the MN
// dimension atoms are one TMA box apart; along K they are 1 KB apart.
constexpr uint32_t LBO = BOX_BYTES;   // next 64 features
constexpr uint32_t SBO = 1024;        // next 8 tokens

// Tile order of the lower triangle (tile (i, j) needs i >= 2 j): bands of BAND column tiles,
// each band row by row, BAND tiles per row once past the diagonal. The CTAs resident at
// one time (about one per SM) then cover ~19 row panels x 8 column panels, i.e. ~4.5k of
// the d features, instead of one column panel and ~150 row panels (~20k features): every
// resident set streams all T tokens of its features from HBM, so this is what keeps a
// large factor (d = 14336, 28672) from re-reading X several times over.
constexpr int BAND = 8;
// Tiles of a band's first r rows past its start (row k of the band holds min(w, k / 2 + 1)).
__host__ __device__ constexpr int band_tiles(int r, int w) {
    return r <= 2 * w ? (r / 2) * (r / 2 + 1) + (r & 1) * (r / 2 + 1) : w * (w + 1) + (r - 2 * w) * w;
}
__device__ __forceinline__ void tile_of(int bid, int n_row_tiles, int n_col_tiles, int* ti, int* tj) {
    for (int j0 = 0; j0 < n_col_tiles; j0 += BAND) {
        const int w = min(BAND, n_col_tiles - j0);
        const int rows = n_row_tiles - 2 * j0;
        const int cnt = band_tiles(rows, w);
        if (bid >= cnt) {
            bid -= cnt;
            continue;
        }
        int k = 0;
        if (bid >= w * (w + 1) && rows > 2 * w) {   // past the triangle: w tiles a row
            k = 2 * w + (bid - w * (w + 1)) / w;
            bid = (bid - w * (w + 1)) % w;
        } else {
            while (bid >= min(w, k / 2 + 1)) bid -= min(w, k++ / 2 + 1);
        }
        *ti = 2 * j0 + k;
        *tj = j0 + bid;
        return;
    }
    *ti = 0;   // not reached for bid < the number of lower tiles
    *tj = 0;
}

__device__ __forceinline__ bool wait_noabort(uint64_t* bar, uint32_t parity) {
    int dummy = 0;
    return mbar_wait(bar, parity, &dummy);
}

// The body shared by the two Gram products.
//   CROSS = false (SYRK): H (+)= A^T A, lower 128 x 256 tiles mirrored on write-out; every
//     operand box comes from map a0.
//   CROSS = true: D (+)= (A_hi + A_lo)^T B over all tiles, no symmetry: the K loop runs over
//     the T tokens of the pair (a0 = A_hi, b) and then over the pair (a1 = A_lo, b).
template <bool CROSS>
__device__ __forceinline__ void gram_tc_body(const CUtensorMap* a0, const CUtensorMap* a1,
                                             const CUtensorMap* bmap, float* __restrict__ H, int d,
                                             int T, int n_row_tiles, int chunk_stages, int accumulate,
                                             int* info) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* mma_done = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    int ti, tj;
    if (CROSS) {
        ti = static_cast<int>(blockIdx.x) % n_row_tiles;
        tj = static_cast<int>(blockIdx.x) / n_row_tiles;
    } else {
        tile_of(blockIdx.x, n_row_tiles, (d + BN - 1) / BN, &ti, &tj);
    }
    const int i0 = ti * BM;
    const int j0 = tj * BN;
    const int nk1 = (T + BK - 1) / BK;          // stages per pass over the tokens
    const int nk = CROSS ? 2 * nk1 : nk1;
    const int nchunks = (nk + chunk_stages - 1) / chunk_stages;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&tfull[b], 1);
            mbar_init(&tempty[b], 8);
        }
        mbar_init(mma_done, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, TMEM_COLS);
        tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(a0);
        if (CROSS) {
            tma_prefetch_desc(a1);
            tma_prefetch_desc(bmap);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int issued = 0;
            for (int k = 0; k < nk; ++k) {
                const int s = k % STAGES;
                const uint32_t u = static_cast<uint32_t>(k / STAGES);
                if (!mbar_wait(&empty[s], (u & 1u) ^ 1u, abort_flag)) break;
                mbar_arrive_expect_tx(&full[s], STAGE_BYTES);
                uint8_t* a = smem + s * STAGE_BYTES;
                uint8_t* b = a + A_BYTES;
                const bool second = CROSS && k >= nk1;
                const int y = (second ? k - nk1 : k) * BK;
                const CUtensorMap* am = second ? a1 : a0;
                const CUtensorMap* bm = CROSS ? bmap : a0;
                tma_load_2d(a, am, &full[s], i0, y);
                tma_load_2d(a + BOX_BYTES, am, &full[s], i0 + 64, y);
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    tma_load_2d(b + q * BOX_BYTES, bm, &full[s], j0 + 64 * q, y);
                issued = k + 1;
            }
            // Drain: every issued load must have landed before the CTA may exit.
            for (int k = (issued > STAGES ? issued - STAGES : 0); k < issued; ++k)
                wait_noabort(&full[k % STAGES], static_cast<uint32_t>(k / STAGES) & 1u);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_mn_major(BM, BN);
            int k = 0;
            bool ok = true;
            for (int c = 0; c < nchunks && ok; ++c) {
                const int buf = c & 1;
                const uint32_t u = static_cast<uint32_t>(c >> 1);
                if (!mbar_wait(&tempty[buf], (u & 1u) ^ 1u, abort_flag)) break;
                tc_fence_after();
                const uint32_t dt = tmem + static_cast<uint32_t>(buf * BN);
                const int kend = min(nk, (c + 1) * chunk_stages);
                for (int kk = 0; k < kend; ++k, ++kk) {
                    const int s = k % STAGES;
                    if (!mbar_wait(&full[s], static_cast<uint32_t>(k / STAGES) & 1u, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a = smem_u32(smem + s * STAGE_BYTES);
                    const uint32_t b = a + A_BYTES;
#pragma unroll
                    for (int k16 = 0; k16 < BK / 16; ++k16) {
                        const uint64_t ad = smem_desc_sw128(a + k16 * 2048, LBO, SBO);
                        const uint64_t bd = smem_desc_sw128(b + k16 * 2048, LBO, SBO);
                        tc_mma_f16(dt, ad, bd, idesc, (kk > 0 || k16 > 0) ? 1u : 0u);
                    }
                    tc_commit(&empty[s]);
                }
                if (ok) tc_commit(&tfull[buf]);
            }
            // All MMAs must be complete before TMEM is released.
            tc_commit(mma_done);
            wait_noabort(mma_done, 0);
        }
    } else {
        // ------------------------------------------------------------ epilogue (8 warps)
        const int q = warp & 3;                 // TMEM lane quadrant this warp may access
        const int half = (warp - 2) >> 2;       // which 128 of the 256 columns
        const int row = i0 + q * 32 + lane;
        float acc[128];
#pragma unroll
        for (int i = 0; i < 128; ++i) acc[i] = 0.0f;
        bool ok = true;
        for (int c = 0; c < nchunks; ++c) {
            const int buf = c & 1;
            const uint32_t u = static_cast<uint32_t>(c >> 1);
            ok = mbar_wait(&tfull[buf], u & 1u, abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc_fence_after();
            const uint32_t base = tmem + (static_cast<uint32_t>(q * 32) << 16) +
                                  static_cast<uint32_t>(buf * BN + half * 128);
#pragma unroll
            for (int p = 0; p < 4; ++p) {
                float v[32];
                tmem_ld32(base + p * 32, v);
                tc_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) acc[p * 32 + i] += v[i];
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[buf]);
        }
        // Write-out through shared memory (the pipeline stages are idle now): each warp stages
        // its 32 rows x 128 columns, then updates the lower tile one 128-byte row segment at a
        // time (coalesced, also for the accumulate read) and writes the mirror from the staged
        // results (lanes on consecutive rows of H^T: coalesced too).
        ok = __all_sync(0xffffffffu, ok && !*abort_flag);
        if (ok) {
            constexpr int SLD = 129;
            float* st = reinterpret_cast<float*>(smem) + (warp - 2) * 32 * SLD;
#pragma unroll
            for (int i = 0; i < 128; ++i) st[lane * SLD + i] = acc[i];
            __syncwarp();
            const int cbase = j0 + half * 128;
            const int rbase = i0 + q * 32;
            // eight rows at a time, so 32 loads per lane are in flight (accumulate mode)
#pragma unroll 1
            for (int r8 = 0; r8 < 32; r8 += 8) {
                float old[8][4];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int rr = rbase + r8 + u;
#pragma unroll
                    for (int m = 0; m < 4; ++m) {
                        const int col = cbase + lane + 32 * m;
                        old[u][m] = (accumulate && rr < d && col < d && (CROSS || col <= rr))
                                        ? H[static_cast<int64_t>(rr) * d + col] : 0.0f;
                    }
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int rr = rbase + r8 + u;
#pragma unroll
                    for (int m = 0; m < 4; ++m) {
                        const int col = cbase + lane + 32 * m;
                        if (rr < d && col < d && (CROSS || col <= rr) &&
                            KQ_IN_RANGE(static_cast<int64_t>(rr) * d + col, static_cast<int64_t>(d) * d)) {
                            const float v = st[(r8 + u) * SLD + lane + 32 * m] + old[u][m];
                            H[static_cast<int64_t>(rr) * d + col] = v;
                            st[(r8 + u) * SLD + lane + 32 * m] = v;
                        }
                    }
                }
            }
            __syncwarp();
            if (!CROSS && row < d) {
#pragma unroll 4
                for (int i = 0; i < 128; ++i) {
                    const int col = cbase + i;
                    if (col < d && col < row && KQ_IN_RANGE(static_cast<int64_t>(col) * d + row, static_cast<int64_t>(d) * d))
                        H[static_cast<int64_t>(col) * d + row] = st[lane * SLD + i];
                }
            }
        }
    }

    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) record_error(info, -KQ_ERR_TIMEOUT);
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

__global__ void __launch_bounds__(NUM_THREADS, 1)
syrk_tc_kernel(const __grid_constant__ CUtensorMap tmap, float* __restrict__ H, int d, int T,
               int n_row_tiles, int chunk_stages, int accumulate, int* info) {
    gram_tc_body<false>(&tmap, &tmap, &tmap, H, d, T, n_row_tiles, chunk_stages, accumulate, info);
}

__global__ void __launch_bounds__(NUM_THREADS, 1)
drift_tc_kernel(const __grid_constant__ CUtensorMap a_hi, const __grid_constant__ CUtensorMap a_lo,
                const __grid_constant__ CUtensorMap b, float* __restrict__ D, int d, int T,
                int n_row_tiles, int chunk_stages, int accumulate, int* info) {
    gram_tc_body<true>(&a_hi, &a_lo, &b, D, d, T, n_row_tiles, chunk_stages, accumulate, info);
}

// Round a finite fp32 value to the nearest bf16, ties to even; returns the 16 bf16 bits.
__device__ __forceinline__ uint32_t bf16_rn_bits(float f) {
    const uint32_t u = __float_as_uint(f);
    return (u + 0x7fffu + ((u >> 16) & 1u)) >> 16;
}

// Exact split of the drift X~ - X into a bf16 pair: hi = bf16(x~ - x), lo = bf16((x~ - x) - hi).
// x~ - x of two bf16 values is exact in fp32 (their significands have 8 bits), and hi + lo
// carries 16 significant bits, which holds the difference exactly unless the two exponents
// are more than 8 apart (then the pair is within 2^-17 of it). Eight elements per thread.
__global__ void drift_split_kernel(const uint16_t* __restrict__ Xt, const uint16_t* __restrict__ X,
                                   int64_t T, int64_t d, int64_t ld, uint16_t* __restrict__ hi,
                                   uint16_t* __restrict__ lo) {
    const int64_t per_row = d >> 3;
    const int64_t total = T * per_row;
    for (int64_t v = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; v < total;
         v += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t t = v / per_row;
        const int64_t c = (v - t * per_row) << 3;
        const uint4 a = __ldg(reinterpret_cast<const uint4*>(Xt + t * ld + c));
        const uint4 b = __ldg(reinterpret_cast<const uint4*>(X + t * ld + c));
        const uint32_t aw[4] = {a.x, a.y, a.z, a.w};
        const uint32_t bw[4] = {b.x, b.y, b.z, b.w};
        uint32_t hw[4], lw[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint32_t h2 = 0, l2 = 0;
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const float xa = __uint_as_float(((aw[q] >> (16 * e)) & 0xffffu) << 16);
                const float xb = __uint_as_float(((bw[q] >> (16 * e)) & 0xffffu) << 16);
                const float df = xa - xb;
                const uint32_t h = bf16_rn_bits(df);
                const uint32_t l = bf16_rn_bits(df - __uint_as_float(h << 16));
                h2 |= h << (16 * e);
                l2 |= l << (16 * e);
            }
            hw[q] = h2;
            lw[q] = l2;
        }
        *reinterpret_cast<uint4*>(hi + t * d + c) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        *reinterpret_cast<uint4*>(lo + t * d + c) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
    }
}

// tr(H) in fp64 from the diagonal (one CTA).
__global__ void trace_kernel(const float* __restrict__ H, int64_t n, double* out) {
    __shared__ double part[32];
    double s = 0.0;
    for (int64_t j = threadIdx.x; j < n; j += blockDim.x) s += static_cast<double>(H[j * n + j]);
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x < 32) {
        s = threadIdx.x < blockDim.x / 32 ? part[threadIdx.x] : 0.0;
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (threadIdx.x == 0) *out = s;
    }
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// 2D map over a [rows x d] bf16 matrix (row stride ld elements): 64-feature x BK-token
// boxes, 128-byte swizzle, zero fill past the last row.
kq_status make_bf16_map(CUtensorMap* m, const uint16_t* base, int64_t d, int64_t rows, int64_t ld,
                        const char* who) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) {
        set_error("%s: cuTensorMapEncodeTiled is unavailable", who);
        return KQ_ERR_CUDA;
    }
    std::memset(m, 0, sizeof(*m));
    cuuint64_t gdim[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
    cuuint64_t gstride[1] = {static_cast<cuuint64_t>(ld) * 2};
    cuuint32_t box[2] = {64, static_cast<cuuint32_t>(BK)};
    cuuint32_t estride[2] = {1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(base), gdim, gstride,
                     box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("%s: cuTensorMapEncodeTiled failed (%d)", who, static_cast<int>(r));
        return KQ_ERR_CUDA;
    }
    return KQ_OK;
}

// Stages (64 tokens each) between drains of the SYRK accumulator. Drains every 512 tokens
// keep the relative error of H_X at T = 262144 near 9e-7; every 1024 or 2048 tokens it grows
// to 2.4e-6 or 5.3e-6 (a downward bias of the tensor-core sums), for 2.5 % less time at 2048.
constexpr int syrk_chunk_stages() { return KQ_SYRK_CHUNK_TOKENS / BK; }

}  // namespace

kq_status launch_trace(const float* H, int64_t n, double* out, cudaStream_t stream) {
    trace_kernel<<<1, 1024, 0, stream>>>(H, n, out);
    KQ_LAUNCH_CHECK("trace_kernel");
    return KQ_OK;
}

KQ_DEBUG_UNIT(syrk)
}  // namespace kq

extern "C" kq_status kq_accum_factor(const uint16_t* A, int64_t T, int64_t d, int64_t lda,
                                     float* H, int accumulate, double* trace, int* info,
                                     kq_stream_t stream_) {
    using namespace kq;
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!H || d < 1 || d > 65536 || T < 0 || (T > 0 && !A) || lda < d) {
        set_error("kq_accum_factor: invalid arguments (d=%lld T=%lld lda=%lld)", (long long)d,
                  (long long)T, (long long)lda);
        return KQ_ERR_INVALID_ARG;
    }
    if (T > 0 && ((reinterpret_cast<uintptr_t>(A) & 15u) != 0 || (lda % 8) != 0 || T > (1ll << 31) - 64)) {
        set_error("kq_accum_factor: A must be 16-byte aligned with lda %% 8 == 0 and T < 2^31");
        return KQ_ERR_INVALID_ARG;
    }
    if (T == 0) {
        if (!accumulate) KQ_CUDA(cudaMemsetAsync(H, 0, sizeof(float) * d * d, stream));
    } else {
        CUtensorMap tmap;
        kq_status st = make_bf16_map(&tmap, A, d, T, lda, "kq_accum_factor");
        if (st != KQ_OK) return st;
        static std::atomic<uint64_t> attr_set{0};
        KQ_TRY(once_per_device(attr_set, [&]() -> kq_status {
            KQ_CUDA(cudaFuncSetAttribute(syrk_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         SMEM_BYTES));
            return KQ_OK;
        }));
        const int n_row = static_cast<int>(cdiv(d, BM));
        const int n_col = static_cast<int>(cdiv(d, BN));
        int64_t tiles = 0;
        for (int j = 0; j < n_col; ++j) tiles += (n_row - 2 * j > 0) ? n_row - 2 * j : 0;
        const int chunk_stages = syrk_chunk_stages();
        syrk_tc_kernel<<<static_cast<unsigned>(tiles), NUM_THREADS, SMEM_BYTES, stream>>>(
            tmap, H, static_cast<int>(d), static_cast<int>(T), n_row, chunk_stages, accumulate, info);
        KQ_LAUNCH_CHECK("syrk_tc_kernel");
    }
    if (trace) return launch_trace(H, d, trace, stream);
    return KQ_OK;
}

// ---------------------------------------------------------------------------- drift statistic
extern "C" size_t kq_accum_drift_workspace(int64_t T, int64_t d) {
    using namespace kq;
    if (T < 1 || d < 1) return 0;
    const int64_t Tr = cdiv(T, BK) * BK;
    return 2 * static_cast<size_t>(Tr) * static_cast<size_t>(d) * sizeof(uint16_t);
}

extern "C" kq_status kq_accum_drift(const uint16_t* Xt, const uint16_t* X, int64_t T, int64_t d, int64_t ld,
                                    float* D, int accumulate, int* info, void* ws, size_t ws_bytes,
                                    kq_stream_t stream_) {
    using namespace kq;
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!D || d < 1 || d > 65536 || T < 0 || (T > 0 && (!Xt || !X)) || ld < d) {
        set_error("kq_accum_drift: invalid arguments (d=%lld T=%lld ld=%lld)", (long long)d, (long long)T,
                  (long long)ld);
        return KQ_ERR_INVALID_ARG;
    }
    if (T > 0 && ((reinterpret_cast<uintptr_t>(Xt) & 15u) || (reinterpret_cast<uintptr_t>(X) & 15u) ||
                  (ld % 8) != 0 || (d % 8) != 0 || T > (1ll << 31) - 64)) {
        set_error("kq_accum_drift: X~ and X must be 16-byte aligned, d and ld multiples of 8, T < 2^31");
        return KQ_ERR_INVALID_ARG;
    }
    if (T == 0) {
        if (!accumulate) KQ_CUDA(cudaMemsetAsync(D, 0, sizeof(float) * d * d, stream));
        return KQ_OK;
    }
    // token chunk: what the workspace holds (a multiple of BK tokens), at most all of T
    const int64_t per_token = 2 * d * static_cast<int64_t>(sizeof(uint16_t));
    int64_t Tc = ws ? static_cast<int64_t>(ws_bytes / per_token) / BK * BK : 0;
    if (Tc > cdiv(T, BK) * BK) Tc = cdiv(T, BK) * BK;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || Tc < BK) {
        set_error("kq_accum_drift: workspace must be 256-byte aligned and hold at least %lld bytes "
                  "(%zu for one pass)", (long long)(per_token * BK), kq_accum_drift_workspace(T, d));
        return KQ_ERR_WORKSPACE;
    }
    uint16_t* hi = static_cast<uint16_t*>(ws);
    uint16_t* lo = hi + Tc * d;
    static std::atomic<uint64_t> attr_set{0};
    KQ_TRY(once_per_device(attr_set, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(drift_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES));
        return KQ_OK;
    }));
    const int n_row = static_cast<int>(cdiv(d, BM));
    const int n_col = static_cast<int>(cdiv(d, BN));
    const int chunk_stages = syrk_chunk_stages();
    for (int64_t t0 = 0; t0 < T; t0 += Tc) {
        const int64_t tn = std::min<int64_t>(Tc, T - t0);
        const int64_t vecs = tn * (d / 8);
        const int64_t grid = std::min<int64_t>(cdiv(vecs, 256), static_cast<int64_t>(num_sms()) * 16);
        drift_split_kernel<<<static_cast<unsigned>(grid), 256, 0, stream>>>(Xt + t0 * ld, X + t0 * ld, tn, d, ld,
                                                                            hi, lo);
        KQ_LAUNCH_CHECK("drift_split_kernel");
        CUtensorMap mh, ml, mb;
        kq_status st = make_bf16_map(&mh, hi, d, tn, d, "kq_accum_drift");
        if (st == KQ_OK) st = make_bf16_map(&ml, lo, d, tn, d, "kq_accum_drift");
        if (st == KQ_OK) st = make_bf16_map(&mb, X + t0 * ld, d, tn, ld, "kq_accum_drift");
        if (st != KQ_OK) return st;
        drift_tc_kernel<<<static_cast<unsigned>(n_row * n_col), NUM_THREADS, SMEM_BYTES, stream>>>(
            mh, ml, mb, D, static_cast<int>(d), static_cast<int>(tn), n_row, chunk_stages,
            (accumulate || t0 > 0) ? 1 : 0, info);
        KQ_LAUNCH_CHECK("drift_tc_kernel");
    }
    return KQ_OK;
}
