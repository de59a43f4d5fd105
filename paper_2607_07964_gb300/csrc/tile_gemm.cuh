// SIMT fp32 tile GEMM used by the OBS trailing update and the blocked inverse Cholesky:
// acc[i][j] (+)= sum_k A[r_i][k] * B(k, c_j) over a 128 x 128 output tile, K <= 128,
// 256 threads, 8 x 8 outputs per thread. Every output's products are accumulated with one
// fused multiply-add per k in ascending k (acc = fma(a, b, acc)), which is the order the
// OBS sweep fixes for bit-exact results.
//
// A is K-contiguous (row r at A + r * lda). B is either K-contiguous (BN = false, "B^T":
// row c at B + c * ldb) or N-contiguous (BN = true: row k at B + k * ldb). K is staged in
// chunks of 32 through a 3-stage cp.async ring; shared rows are padded so every 128-bit
// read is bank-conflict free. Rows/columns/k beyond the valid range are zero-filled.
#pragma once

#include "kq_common.cuh"

namespace kq {

constexpr int GT = 128;          // tile rows and columns
constexpr int GK = 32;           // k per chunk
constexpr int GLD = GK + 4;      // row stride of K-contiguous chunks [GT][GK]
constexpr int GLDN = GT + 4;     // row stride of N-contiguous chunks [GK][GT]
constexpr int GSTAGES = 3;
constexpr int G_A_FLOATS = GT * GLD;                  // 4608
constexpr int G_B_FLOATS = GT * GLD;                  // >= GK * GLDN = 4224
constexpr int G_STAGE_FLOATS = G_A_FLOATS + G_B_FLOATS;
constexpr size_t G_SMEM = static_cast<size_t>(GSTAGES) * G_STAGE_FLOATS * sizeof(float);   // 110592
constexpr int G_THREADS = 256;

// Output row of register row i for thread row ty: {4ty..4ty+3, 64+4ty..64+4ty+3}.
__device__ __forceinline__ int gt_row(int ty, int i) { return i < 4 ? 4 * ty + i : 64 + 4 * ty + (i - 4); }
// Output column of register column j for thread column tx.
template <bool BN>
__device__ __forceinline__ int gt_col(int tx, int j) {
    return BN ? (j < 4 ? 4 * tx + j : 64 + 4 * tx + (j - 4)) : tx + 16 * j;
}

template <bool VEC>
__device__ __forceinline__ void g_copy16(float* dst, const float* src_row, int64_t k, int valid_floats) {
    // valid_floats in [0, 4]: how many of src_row[k .. k+3] exist
    if (VEC) {
        cp_async16(dst, valid_floats > 0 ? static_cast<const void*>(src_row + k) : static_cast<const void*>(src_row),
                   4 * valid_floats);
    } else {
        float4 v;
        v.x = valid_floats > 0 ? src_row[k] : 0.0f;
        v.y = valid_floats > 1 ? src_row[k + 1] : 0.0f;
        v.z = valid_floats > 2 ? src_row[k + 2] : 0.0f;
        v.w = valid_floats > 3 ? src_row[k + 3] : 0.0f;
        *reinterpret_cast<float4*>(dst) = v;
    }
}

template <bool BN, bool VEC>
__device__ __forceinline__ void g_load_chunk(float* smem, int stage, int ch, const float* A, int64_t lda, int arows,
                                             const float* B, int64_t ldb, int bcols, int kb) {
    float* As = smem + stage * G_STAGE_FLOATS;
    float* Bs = As + G_A_FLOATS;
    const int k0 = ch * GK;
    for (int q = threadIdx.x; q < GT * (GK / 4); q += G_THREADS) {
        const int r = q >> 3, k4 = q & 7;
        const int k = k0 + 4 * k4;
        const int va = r < arows ? max(0, min(4, kb - k)) : 0;
        g_copy16<VEC>(As + r * GLD + 4 * k4, A + static_cast<int64_t>(r < arows ? r : 0) * lda, k, va);
        if (!BN) {
            const int vb = r < bcols ? max(0, min(4, kb - k)) : 0;
            g_copy16<VEC>(Bs + r * GLD + 4 * k4, B + static_cast<int64_t>(r < bcols ? r : 0) * ldb, k, vb);
        }
    }
    if (BN) {
        for (int q = threadIdx.x; q < GK * (GT / 4); q += G_THREADS) {
            const int kk = q >> 5, c4 = q & 31;
            const int k = k0 + kk, c = 4 * c4;
            const int vb = k < kb ? max(0, min(4, bcols - c)) : 0;
            g_copy16<VEC>(Bs + kk * GLDN + c, B + static_cast<int64_t>(k < kb ? k : 0) * ldb, c, vb);
        }
    }
}

template <bool BN>
__device__ __forceinline__ void g_compute_chunk(const float* smem, int stage, int ty, int tx, float (&acc)[8][8]) {
    const float* As = smem + stage * G_STAGE_FLOATS;
    const float* Bs = As + G_A_FLOATS;
#pragma unroll 1
    for (int k4 = 0; k4 < GK / 4; ++k4) {
        float4 a[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) a[i] = *reinterpret_cast<const float4*>(As + gt_row(ty, i) * GLD + 4 * k4);
        if (!BN) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float4 b = *reinterpret_cast<const float4*>(Bs + gt_col<false>(tx, j) * GLD + 4 * k4);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    acc[i][j] = __fmaf_rn(a[i].x, b.x, acc[i][j]);
                    acc[i][j] = __fmaf_rn(a[i].y, b.y, acc[i][j]);
                    acc[i][j] = __fmaf_rn(a[i].z, b.z, acc[i][j]);
                    acc[i][j] = __fmaf_rn(a[i].w, b.w, acc[i][j]);
                }
            }
        } else {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
                const float* brow = Bs + (4 * k4 + kk) * GLDN;
                const float4 b0 = *reinterpret_cast<const float4*>(brow + 4 * tx);
                const float4 b1 = *reinterpret_cast<const float4*>(brow + 64 + 4 * tx);
                const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float av = kk == 0 ? a[i].x : kk == 1 ? a[i].y : kk == 2 ? a[i].z : a[i].w;
#pragma unroll
                    for (int j = 0; j < 8; ++j) acc[i][j] = __fmaf_rn(av, bv[j], acc[i][j]);
                }
            }
        }
    }
}

// acc = sum over k < kb of A-tile x B-tile, in ascending k (INIT = false: the sum continues
// from the acc passed in). smem: G_SMEM bytes, 16-aligned.
template <bool BN, bool VEC, bool INIT = true>
__device__ __forceinline__ void gemm_tile(const float* A, int64_t lda, int arows, const float* B, int64_t ldb, int bcols,
                                          int kb, float (&acc)[8][8], float* smem) {
    const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
    if (INIT) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[i][j] = 0.0f;
    }
    const int nch = (kb + GK - 1) / GK;
    for (int c = 0; c < GSTAGES - 1; ++c) {
        if (c < nch) g_load_chunk<BN, VEC>(smem, c, c, A, lda, arows, B, ldb, bcols, kb);
        cp_async_commit();
    }
    for (int c = 0; c < nch; ++c) {
        cp_async_wait<GSTAGES - 2>();
        __syncthreads();
        const int nxt = c + GSTAGES - 1;
        if (nxt < nch) g_load_chunk<BN, VEC>(smem, nxt % GSTAGES, nxt, A, lda, arows, B, ldb, bcols, kb);
        cp_async_commit();
        g_compute_chunk<BN>(smem, c % GSTAGES, ty, tx, acc);
    }
    cp_async_wait<0>();
    __syncthreads();
}

}  // namespace kq
