// Stage 4: the column-wise OBS sweep with b-bit asymmetric grids (GPTQ mode).
//
// Paper: Sec. 2.1 Eq. (obs_update) (compensation -(w_p - q_p)/[H^-1]_pp [H^-1]_{p,p+1:}),
// Algorithm 2 (inner column loop over a block of B columns with error E, then the lazy
// trailing update W[:, i+B:] -= E R[i:i+B, i+B:]), Proposition 1 (H_G cancels, so only
// L = R^T enters). The GPTAQ drift term P is zero here (one input set, X-tilde = X).
//
// Every fp32 operation is written with an explicit round-to-nearest intrinsic so the
// compiler cannot contract or reorder it; the order is:
//   grid      scale = (xmax - xmin) / (2^b - 1), zero = rint(-xmin / scale)
//   column j  q = clamp(rint(w / scale) + zero, 0, 2^b - 1); what = scale * (q - zero)
//             E = (w - what) / R_jj;  w_k = fma(-E, R_jk, w_k) for k in (j, block end)
//   trailing  acc = fma(E_k, R_kc, acc) over ascending k; w_c = w_c - acc
// Kernels:
//   rowgrid_kernel   per-row grid (group = 0) from the whole row before the sweep
//   obs_block_kernel four rows per warp; the block's R (128 x 128) in shared memory
//   trailing_kernel  128 x 128 output tiles of the shared tile GEMM (tile_gemm.cuh)
//   colloss_kernel   col_loss[j] = sum over rows of E_j^2, fixed order, fp64
#include <math.h>

#include "kq_common.cuh"
#include "tile_gemm.cuh"

namespace kq {
namespace {

constexpr int BLK = 128;          // block size B (Algorithm 2); the only supported value
constexpr int RTLD = BLK + 4;     // row stride of the staged L block (16-byte rows)
constexpr int kRowsPerLane = 1;   // rows per lane group in the block kernel

struct Grid {
    float scale, zero;
};

__device__ __forceinline__ Grid make_grid(float xmin, float xmax, float maxq) {
    xmin = fminf(xmin, 0.0f);
    xmax = fmaxf(xmax, 0.0f);
    if (xmin == 0.0f && xmax == 0.0f) {
        xmin = -1.0f;
        xmax = 1.0f;
    }
    Grid g;
    g.scale = __fdiv_rn(__fsub_rn(xmax, xmin), maxq);
    g.zero = rintf(__fdiv_rn(-xmin, g.scale));
    return g;
}

__device__ __forceinline__ float warp_min(float v) {
    for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Per-row grid from the whole row (group = 0). Warp per row.
__global__ void rowgrid_kernel(const float* __restrict__ W, int64_t d_out, int64_t d_in, int bits,
                               float* __restrict__ scale, int32_t* __restrict__ zero,
                               float* __restrict__ gscale, float* __restrict__ gzero) {
    const int64_t r = static_cast<int64_t>(blockIdx.x) * (blockDim.x / 32) + threadIdx.x / 32;
    const int lane = threadIdx.x & 31;
    if (r >= d_out) return;
    float mn = 0.0f, mx = 0.0f;
    for (int64_t j = lane; j < d_in; j += 32) {
        const float v = W[r * d_in + j];
        mn = fminf(mn, v);
        mx = fmaxf(mx, v);
    }
    mn = warp_min(mn);
    mx = warp_max(mx);
    const Grid g = make_grid(mn, mx, static_cast<float>((1 << bits) - 1));
    if (lane == 0) {
        scale[r] = g.scale;
        zero[r] = static_cast<int32_t>(g.zero);
        gscale[r] = g.scale;
        gzero[r] = g.zero;
    }
}

// One block [i0, e) of the sweep for all rows. A group of LPR = 4 lanes handles RPL rows;
// lane position lp holds columns i0 + 4 t + lp (t = 0..31) of each of its rows in registers.
// Per column j the owner lane broadcasts w_j inside its group; every lane of the group
// computes the (identical) quantization, then updates its own later columns. The RPL rows
// of a lane share the loads of R and give independent instruction chains.
#ifndef KQ_OBS_LANES_PER_ROW
#define KQ_OBS_LANES_PER_ROW 8
#endif
constexpr int LPR = KQ_OBS_LANES_PER_ROW;   // lanes per row group (4 or 8)
constexpr int CPL = BLK / LPR;         // columns per lane

__device__ __forceinline__ float group_min(float v) {
    for (int o = LPR / 2; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float group_max(float v) {
    for (int o = LPR / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

template <int RPL>
__global__ void __launch_bounds__(128, 3) obs_block_kernel(
    const float* __restrict__ W, int64_t d_out, int64_t d_in, const float* __restrict__ Lt, int64_t i0,
    int bits, int group, const float* __restrict__ gscale, const float* __restrict__ gzero,
    uint8_t* __restrict__ codes, float* __restrict__ scale, int32_t* __restrict__ zero,
    float* __restrict__ E, float* __restrict__ pre_q, bool vec) {
    // The block of L = R^T in its own layout: Rt[k][j] = Lt[i0 + k][i0 + j] = R[i0 + j][i0 + k],
    // staged with 16-byte cp.async copies (scalar loads when rows are not 16-byte aligned).
    extern __shared__ __align__(16) float Rt[];   // [BLK][RTLD]
    const int nb = static_cast<int>(min(static_cast<int64_t>(BLK), d_in - i0));
    if (vec) {
        for (int e = threadIdx.x; e < BLK * (BLK / 4); e += blockDim.x) {
            const int k = e >> 5, j4 = (e & 31) * 4;
            const int valid = k < nb ? max(0, min(4, nb - j4)) : 0;
            cp_async16(Rt + k * RTLD + j4,
                       valid ? static_cast<const void*>(Lt + (i0 + k) * d_in + i0 + j4) : static_cast<const void*>(Lt),
                       4 * valid);
        }
        cp_async_commit();
        cp_async_wait<0>();
    } else {
        for (int e = threadIdx.x; e < BLK * BLK; e += blockDim.x) {
            const int k = e / BLK, j = e % BLK;
            Rt[k * RTLD + j] = (j < nb && k < nb) ? Lt[(i0 + k) * d_in + i0 + j] : 0.0f;
        }
    }
    __syncthreads();
    const float maxq = static_cast<float>((1 << bits) - 1);
    const int lane = threadIdx.x & 31;
    const int lp = lane & (LPR - 1);
    const int gbase = lane & ~(LPR - 1);
    const int64_t ngroups = group ? (d_in + group - 1) / group : 1;
    const int warps = blockDim.x / 32;
    constexpr int RPW = (32 / LPR) * RPL;   // rows per warp
    for (int64_t rw = (static_cast<int64_t>(blockIdx.x) * warps + threadIdx.x / 32) * RPW; rw < d_out;
         rw += static_cast<int64_t>(gridDim.x) * warps * RPW) {
        int64_t r[RPL];
        bool live[RPL];
        float w[RPL][CPL];
        Grid g[RPL];
#pragma unroll
        for (int u = 0; u < RPL; ++u) {
            r[u] = rw + (lane / LPR) * RPL + u;
            live[u] = r[u] < d_out;
            const float* wr = W + r[u] * d_in + i0;
#pragma unroll
            for (int t = 0; t < CPL; ++t) {
                const int c = LPR * t + lp;
                w[u][t] = (live[u] && c < nb) ? wr[c] : 0.0f;
            }
            if (group) {
                float mn = 0.0f, mx = 0.0f;
#pragma unroll
                for (int t = 0; t < CPL; ++t)
                    if (LPR * t + lp < nb) {
                        mn = fminf(mn, w[u][t]);
                        mx = fmaxf(mx, w[u][t]);
                    }
                g[u] = make_grid(group_min(mn), group_max(mx), maxq);
                if (live[u] && lp == 0) {
                    const int64_t gi = r[u] * ngroups + i0 / group;
                    scale[gi] = g[u].scale;
                    zero[gi] = static_cast<int32_t>(g[u].zero);
                }
            } else {
                g[u].scale = live[u] ? gscale[r[u]] : 1.0f;
                g[u].zero = live[u] ? gzero[r[u]] : 0.0f;
            }
        }
        // Slot q of the block is always w[.][0]: after its 8 columns the registers shift
        // down by one, which keeps the loop rolled (compact code) with register indexing.
#pragma unroll 1
        for (int q = 0; q < CPL; ++q) {
            float e_cur[RPL], pq_cur[RPL];
            uint32_t q_cur[RPL];
#pragma unroll
            for (int u = 0; u < RPL; ++u) {
                e_cur[u] = 0.0f;
                pq_cur[u] = 0.0f;
                q_cur[u] = 0;
            }
#pragma unroll
            for (int jl = 0; jl < LPR; ++jl) {
                const int j = LPR * q + jl;
                if (j < nb) {   // uniform across the warp
                    const float dj = Rt[j * RTLD + j];
                    float err[RPL];
#pragma unroll
                    for (int u = 0; u < RPL; ++u) {
                        const float wj = __shfl_sync(0xffffffffu, w[u][0], gbase | jl);
                        float qq = __fadd_rn(rintf(__fdiv_rn(wj, g[u].scale)), g[u].zero);
                        qq = fminf(fmaxf(qq, 0.0f), maxq);
                        const float what = __fmul_rn(g[u].scale, __fsub_rn(qq, g[u].zero));
                        err[u] = __fdiv_rn(__fsub_rn(wj, what), dj);
                        if (lp == jl) {
                            e_cur[u] = err[u];
                            q_cur[u] = static_cast<uint32_t>(qq);
                            pq_cur[u] = wj;
                        }
                    }
                    const float* rcol = Rt + (LPR * q + lp) * RTLD + j;   // R[j][k] = Rt[k][j]
#pragma unroll
                    for (int t = 0; t < CPL; ++t) {
                        if (t < CPL - q && LPR * (q + t) + lp > j) {
                            const float rv = rcol[LPR * t * RTLD];
#pragma unroll
                            for (int u = 0; u < RPL; ++u) w[u][t] = __fmaf_rn(-err[u], rv, w[u][t]);
                        }
                    }
                }
            }
            const int c = LPR * q + lp;
#pragma unroll
            for (int u = 0; u < RPL; ++u) {
                if (live[u] && c < nb) {
                    codes[r[u] * d_in + i0 + c] = static_cast<uint8_t>(q_cur[u]);
                    E[r[u] * d_in + i0 + c] = e_cur[u];
                    if (pre_q) pre_q[r[u] * d_in + i0 + c] = pq_cur[u];
                }
#pragma unroll
                for (int t = 0; t + 1 < CPL; ++t) w[u][t] = w[u][t + 1];
                w[u][CPL - 1] = 0.0f;
            }
        }
    }
}

// W[:, e0:] -= E[:, i0:e0] R[i0:e0, e0:] with R[k][c] = Lt[c][k]: 128 x 128 output tiles
// of the shared tile GEMM (acc = fma(E_k, R_kc, acc) over ascending k), then w = w - acc.
template <bool VEC>
__global__ void __launch_bounds__(G_THREADS, 2) trailing_kernel(float* __restrict__ W, const float* __restrict__ E,
                                                                const float* __restrict__ Lt, int64_t d_out,
                                                                int64_t d_in, int64_t i0, int kb) {
    extern __shared__ __align__(16) float sm[];
    const int64_t e0 = i0 + kb;
    const int64_t r0 = static_cast<int64_t>(blockIdx.y) * GT;
    const int64_t c0 = e0 + static_cast<int64_t>(blockIdx.x) * GT;
    const int arows = static_cast<int>(min(static_cast<int64_t>(GT), d_out - r0));
    const int bcols = static_cast<int>(min(static_cast<int64_t>(GT), d_in - c0));
    float acc[8][8];
    gemm_tile<false, VEC>(E + r0 * d_in + i0, d_in, arows, Lt + c0 * d_in + i0, d_in, bcols, kb, acc, sm);
    const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
    // Read-modify-write of W in two halves of 32 values, all loads of a half issued before
    // its stores, so the memory latency is paid twice rather than 64 times.
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        float wv[4][8];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int rr = gt_row(ty, 4 * h + i), cc = gt_col<false>(tx, j);
                wv[i][j] = (rr < arows && cc < bcols) ? W[(r0 + rr) * d_in + c0 + cc] : 0.0f;
            }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int rr = gt_row(ty, 4 * h + i), cc = gt_col<false>(tx, j);
                if (rr < arows && cc < bcols) W[(r0 + rr) * d_in + c0 + cc] = __fsub_rn(wv[i][j], acc[4 * h + i][j]);
            }
    }
}

// col_loss[j] = sum over rows of E[r][j]^2: fp32 partials over 32 rows, fp64 across them,
// fixed order. Block (32, 8): 32 columns, 8 row lanes.
__global__ void colloss_kernel(const float* __restrict__ E, int64_t d_out, int64_t d_in,
                               float* __restrict__ col_loss) {
    __shared__ double part[8][33];
    const int64_t j = static_cast<int64_t>(blockIdx.x) * 32 + threadIdx.x;
    double acc = 0.0;
    if (j < d_in) {
        float p = 0.0f;
        int cnt = 0;
        for (int64_t r = threadIdx.y; r < d_out; r += 8) {
            const float v = E[r * d_in + j];
            p = fmaf(v, v, p);
            if (++cnt == 32) {
                acc += p;
                p = 0.0f;
                cnt = 0;
            }
        }
        acc += p;
    }
    part[threadIdx.y][threadIdx.x] = acc;
    __syncthreads();
    if (threadIdx.y == 0 && j < d_in) {
        double a = 0.0;
        for (int y = 0; y < 8; ++y) a += part[y][threadIdx.x];
        col_loss[j] = static_cast<float>(a);
    }
}

struct ObsWs {
    float* E;
    float* gscale;
    float* gzero;
};

ObsWs carve(void* ws, int64_t d_out, int64_t d_in) {
    ObsWs o;
    o.E = static_cast<float*>(ws);
    o.gscale = o.E + d_out * d_in;
    o.gzero = o.gscale + d_out;
    return o;
}

}  // namespace
}  // namespace kq

using namespace kq;

extern "C" size_t kq_obs_quantize_workspace(int64_t d_out, int64_t d_in, int block) {
    (void)block;
    if (d_out < 1 || d_in < 1) return 0;
    return static_cast<size_t>(d_out) * d_in * sizeof(float) + 2 * static_cast<size_t>(d_out) * sizeof(float) + 256;
}

extern "C" kq_status kq_obs_quantize(float* W, int64_t d_out, int64_t d_in, const float* Lt, int bits,
                                     int group, int block, uint8_t* codes, float* scale, int32_t* zero,
                                     float* col_loss, float* pre_q, void* ws, size_t ws_bytes,
                                     kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!W || !Lt || !codes || !scale || !zero || d_out < 1 || d_in < 1 || bits < 1 || bits > 8) {
        set_error("kq_obs_quantize: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (block != BLK || (group != 0 && group != block)) {
        set_error("kq_obs_quantize: block must be %d and group 0 or equal to block", BLK);
        return KQ_ERR_UNSUPPORTED;
    }
    if (!ws || ws_bytes < kq_obs_quantize_workspace(d_out, d_in, block) ||
        (reinterpret_cast<uintptr_t>(ws) & 15u)) {
        set_error("kq_obs_quantize: workspace must be 16-byte aligned and hold %zu bytes",
                  kq_obs_quantize_workspace(d_out, d_in, block));
        return KQ_ERR_WORKSPACE;
    }
    static bool attr = false;
    if (!attr) {
        KQ_CUDA(cudaFuncSetAttribute(obs_block_kernel<kRowsPerLane>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     BLK * RTLD * 4));
        KQ_CUDA(cudaFuncSetAttribute(trailing_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(G_SMEM)));
        KQ_CUDA(cudaFuncSetAttribute(trailing_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(G_SMEM)));
        attr = true;
    }
    ObsWs o = carve(ws, d_out, d_in);
    if (group == 0) {
        rowgrid_kernel<<<static_cast<unsigned>(cdiv(d_out, 8)), 256, 0, stream>>>(W, d_out, d_in, bits, scale,
                                                                                zero, o.gscale, o.gzero);
        KQ_LAUNCH_CHECK("rowgrid_kernel");
    }
    const bool vec = (d_in % 4 == 0) && (reinterpret_cast<uintptr_t>(Lt) % 16 == 0);
    const int64_t rows_per_cta = 4 * (32 / LPR) * kRowsPerLane;   // 4 warps per CTA
    const int64_t row_ctas = std::min<int64_t>(cdiv(d_out, rows_per_cta), static_cast<int64_t>(num_sms()) * 3);
    for (int64_t i0 = 0; i0 < d_in; i0 += BLK) {
        const int kb = static_cast<int>(std::min<int64_t>(BLK, d_in - i0));
        obs_block_kernel<kRowsPerLane><<<static_cast<unsigned>(row_ctas), 128, BLK * RTLD * 4, stream>>>(
            W, d_out, d_in, Lt, i0, bits, group, o.gscale, o.gzero, codes, scale, zero, o.E, pre_q, vec);
        KQ_LAUNCH_CHECK("obs_block_kernel");
        const int64_t rest = d_in - (i0 + kb);
        if (rest > 0) {
            dim3 grid(static_cast<unsigned>(cdiv(rest, GT)), static_cast<unsigned>(cdiv(d_out, GT)));
            if (vec)
                trailing_kernel<true><<<grid, G_THREADS, G_SMEM, stream>>>(W, o.E, Lt, d_out, d_in, i0, kb);
            else
                trailing_kernel<false><<<grid, G_THREADS, G_SMEM, stream>>>(W, o.E, Lt, d_out, d_in, i0, kb);
            KQ_LAUNCH_CHECK("trailing_kernel");
        }
    }
    if (col_loss) {
        colloss_kernel<<<static_cast<unsigned>(cdiv(d_in, 32)), dim3(32, 8), 0, stream>>>(o.E, d_out, d_in, col_loss);
        KQ_LAUNCH_CHECK("colloss_kernel");
    }
    return KQ_OK;
}
