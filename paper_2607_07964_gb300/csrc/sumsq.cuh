// Sums of squares along rows and along columns of a row-major fp32 matrix, in a fixed
// order (deterministic): fp32 partials over short runs, fp64 across runs and lanes.
//
// Both are HBM-bound single passes. They keep many independent loads in flight per thread
// (the runs are unrolled, loads first, then the FMA chain), which a one-load-per-iteration
// loop does not: with ~1 us DRAM latency that loop ran at a tenth of the copy bandwidth.
#pragma once

#include <stdint.h>

namespace kq {

// Column sums: block (CS_X, CS_Y); column j = blockIdx.x * CS_X + threadIdx.x; thread row y
// reads the CS_U-row runs starting at y * CS_U, stepping CS_Y * CS_U rows.
constexpr int CS_X = 32, CS_Y = 16, CS_U = 16;

// sum over r of M[r][j]^2; the result is valid in threadIdx.y == 0 (all threads must call).
__device__ __forceinline__ double col_sumsq(const float* __restrict__ M, int64_t rows, int64_t cols, int64_t j) {
    __shared__ double part[CS_Y][CS_X + 1];
    double acc = 0.0;
    if (j < cols) {
        for (int64_t r0 = static_cast<int64_t>(threadIdx.y) * CS_U; r0 < rows; r0 += CS_Y * CS_U) {
            float v[CS_U];
#pragma unroll
            for (int k = 0; k < CS_U; ++k) v[k] = (r0 + k < rows) ? __ldg(M + (r0 + k) * cols + j) : 0.0f;
            float p = 0.0f;
#pragma unroll
            for (int k = 0; k < CS_U; ++k) p = fmaf(v[k], v[k], p);
            acc += p;
        }
    }
    part[threadIdx.y][threadIdx.x] = acc;
    __syncthreads();
    double a = 0.0;
    if (threadIdx.y == 0)
        for (int y = 0; y < CS_Y; ++y) a += part[y][threadIdx.x];
    return a;
}

// Row sums: one warp per row. Lane l reads 4-float groups l, l + 32, ... (float4 when the
// row start is 16-byte aligned and the length a multiple of 4), RS_U groups per run.
constexpr int RS_U = 4;

// sum over j of row[j]^2, valid in every lane of the warp.
__device__ __forceinline__ double row_sumsq(const float* __restrict__ row, int64_t n) {
    const int lane = threadIdx.x & 31;
    double acc = 0.0;
    if ((n & 3) == 0 && (reinterpret_cast<uintptr_t>(row) & 15) == 0) {
        const float4* r4 = reinterpret_cast<const float4*>(row);
        const int64_t n4 = n >> 2;
        for (int64_t g0 = lane; g0 < n4; g0 += 32 * RS_U) {
            float4 v[RS_U];
#pragma unroll
            for (int u = 0; u < RS_U; ++u)
                v[u] = (g0 + 32 * u < n4) ? __ldg(r4 + g0 + 32 * u) : make_float4(0.f, 0.f, 0.f, 0.f);
            float p = 0.0f;
#pragma unroll
            for (int u = 0; u < RS_U; ++u) {
                p = fmaf(v[u].x, v[u].x, p);
                p = fmaf(v[u].y, v[u].y, p);
                p = fmaf(v[u].z, v[u].z, p);
                p = fmaf(v[u].w, v[u].w, p);
            }
            acc += p;
        }
    } else {
        for (int64_t j0 = lane; j0 < n; j0 += 32 * 4 * RS_U) {
            float v[4 * RS_U];
#pragma unroll
            for (int u = 0; u < 4 * RS_U; ++u) v[u] = (j0 + 32 * u < n) ? __ldg(row + j0 + 32 * u) : 0.0f;
            float p = 0.0f;
#pragma unroll
            for (int u = 0; u < 4 * RS_U; ++u) p = fmaf(v[u], v[u], p);
            acc += p;
        }
    }
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    return acc;
}

}  // namespace kq
