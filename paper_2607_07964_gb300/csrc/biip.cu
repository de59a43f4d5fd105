// Stage 2: bidirectional incoherence processing (BiIP) and the sensitivity traces.
//
// Paper: Sec. 3.2 Eq. (rescale) (S_X, S_G from Hessian diagonals and weight norms),
// Eq. (biip) (W <- U W V^T, H_X <- V H_X V^T, H_G <- U H_G U^T), Algorithm 1 (rescale,
// then rotate, then release H_G); Sec. 3.3 Eq. (sensitivity) (s = tr(H_G) tr(H_X),
// computed after BiIP).
//
// The rotations are randomized Hadamard transforms applied as fast transforms, never as
// dense matrices (the paper's dense products cost O(n^3); these cost O(n^2 log n) and are
// bound by HBM): a row transform (along the contiguous dimension, one row per CTA in
// shared memory) and a column transform (along the strided dimension) done as one pass
// per radix stage, each CTA holding R rows x CW columns. For n = 28 * 2^k the 2^k part is
// a Walsh-Hadamard butterfly and the 28-point factor a dense +-1 mix at stride 2^k.
#include <math.h>

#include <algorithm>

#include "kq_common.cuh"
#include "rht.cuh"
#include "sumsq.cuh"

namespace kq {
namespace {

// ------------------------------------------------------------------ row transform
// For each row of M [rows x n]: v <- pre (.) v; v <- (H_28 (x) H_P) v (or H_P); row <-
// post (.) v / sqrt(n). A CTA walks rows r = blockIdx.x, + gridDim.x, ... with two shared
// row buffers when they fit (DBL): the next row's cp.async copy is issued before the
// current row's butterflies, so loads overlap compute within the CTA. The power-of-two
// part runs as radix-8 passes (one barrier per pass); the last pass (or the 28-point mix)
// writes straight to global memory.
template <bool HAS28>
__global__ void __launch_bounds__(256, HAS28 ? 2 : 4) rht_rows_kernel(float* __restrict__ M, int64_t rows, int n, int lgP,
                                int pre_mode, int post_mode, const int8_t* __restrict__ sign,
                                const float* __restrict__ s, float inv_sqrt_n, int dbl) {
    extern __shared__ __align__(16) float smem_rows[];
    const int P = 1 << lgP;
    const bool async = (reinterpret_cast<uintptr_t>(M) & 15u) == 0 && (n & 3) == 0;
    auto issue = [&](int64_t r, float* dst) {
        const float* src = M + r * n;
        for (int q = threadIdx.x; q < (n >> 2); q += blockDim.x) cp_async16(dst + 4 * q, src + 4 * q, 16);
        cp_async_commit();
    };
    int it = 0;
    if (async && dbl && blockIdx.x < rows) issue(blockIdx.x, smem_rows);
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x, ++it) {
        float* row = M + r * n;
        float* v = smem_rows + ((async && dbl) ? (it & 1) * n : 0);
        if (async && dbl) {
            const int64_t nxt = r + gridDim.x;
            if (nxt < rows) {
                issue(nxt, smem_rows + ((it + 1) & 1) * n);
                cp_async_wait<1>();
            } else {
                cp_async_wait<0>();
            }
            __syncthreads();
        } else {
            stage_row(v, row, n);
        }
        bool first = true;
        if (!HAS28 && lgP == 0) {   // n == 1
            for (int j = threadIdx.x; j < n; j += blockDim.x)
                row[j] = v[j] * factor(pre_mode, sign, s, j) * (factor(post_mode, sign, s, j) * inv_sqrt_n);
        }
        for (int lgh = 0; lgh < lgP;) {   // I_28 (x) H_P: passes stay inside P-aligned chunks
            const int lgr = min(3, lgP - lgh);
            const bool last = !HAS28 && lgh + lgr == lgP;
            if (first && last) fwht_pass<true, true>(v, n, lgh, lgr, pre_mode, post_mode, sign, s, inv_sqrt_n, row);
            else if (first) fwht_pass<true, false>(v, n, lgh, lgr, pre_mode, post_mode, sign, s, inv_sqrt_n, row);
            else if (last) fwht_pass<false, true>(v, n, lgh, lgr, pre_mode, post_mode, sign, s, inv_sqrt_n, row);
            else fwht_pass<false, false>(v, n, lgh, lgr, pre_mode, post_mode, sign, s, inv_sqrt_n, row);
            first = false;
            __syncthreads();
            lgh += lgr;
        }
        if (HAS28) {   // H_28 (x) I_P, written straight to global memory
            for (int b = threadIdx.x; b < P; b += blockDim.x) {
                float x[28];
#pragma unroll
                for (int a = 0; a < 28; ++a) {
                    x[a] = v[a * P + b];
                    if (first) x[a] *= factor(pre_mode, sign, s, a * P + b);
                }
                mix28(x, [&](int a, float y) {
                    row[a * P + b] = y * (factor(post_mode, sign, s, a * P + b) * inv_sqrt_n);
                });
            }
            __syncthreads();
        }
    }
}

// ------------------------------------------------------- row transform in registers
// For n = 2^LG (LG in [9, 14]), the register transform of rht.cuh per row: phase 0 reads
// the thread's 16 contiguous elements from global memory with the pre-factor (a per-CTA
// table), the last phase writes straight to global memory (consecutive threads,
// consecutive elements) with the post-factor and 1/sqrt(n). Each CTA walks rows
// r = blockIdx.x, + gridDim.x, ..., loading the next row into registers first.
template <int LG, bool POST>
__global__ void __launch_bounds__((1 << LG) / 16) rht_rows_reg_kernel(float* __restrict__ M, int64_t rows,
                                                                      int pre_mode, int post_mode,
                                                                      const int8_t* __restrict__ sign,
                                                                      const float* __restrict__ s, float inv_sqrt_n) {
    constexpr int N = 1 << LG, T = N / 16, NPH = rr_phases(LG);
    constexpr uint32_t ML = rr_mask(LG, NPH - 1);
    static_assert(rr_mask(LG, 0) == 0xFu, "phase 0 is the thread's 16 contiguous elements");
    static_assert(ML >> (LG - 4) == 0xFu, "the last phase covers the top four bits");
    extern __shared__ __align__(16) float sm_rr[];
    float* fpre = sm_rr;            // [N]
    float* fpost = sm_rr + N;       // [N], times 1/sqrt(n)
    float* buf = sm_rr + 2 * N;     // [N + N / 32]
    const int t = threadIdx.x;
    for (int j = t; j < N; j += T) {
        fpre[j] = factor(pre_mode, sign, s, j);
        fpost[j] = factor(post_mode, sign, s, j) * inv_sqrt_n;
    }
    auto load = [&](int64_t row, float (&v)[16]) {
        const float4* src = reinterpret_cast<const float4*>(M + row * N + 16 * t);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float4 a = src[q];
            v[4 * q] = a.x;
            v[4 * q + 1] = a.y;
            v[4 * q + 2] = a.z;
            v[4 * q + 3] = a.w;
        }
    };
    float x[16], nx[16];
    int64_t r = blockIdx.x;
    if (r < rows) load(r, x);
    __syncthreads();   // factors ready
    const int tl = deposit_bits<((1u << LG) - 1u) & ~ML>(t);
    for (; r < rows; r += gridDim.x) {
        if (r + gridDim.x < rows) load(r + gridDim.x, nx);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float4 f = reinterpret_cast<const float4*>(fpre + 16 * t)[q];
            x[4 * q] *= f.x;
            x[4 * q + 1] *= f.y;
            x[4 * q + 2] *= f.z;
            x[4 * q + 3] *= f.w;
        }
        fwht_kbits<0xFu>(x);
        rr_transpose<LG, 1>(x, buf, t);
        if constexpr (NPH > 2) rr_transpose<LG, 2>(x, buf, t);
        if constexpr (NPH > 3) rr_transpose<LG, 3>(x, buf, t);
        float* dst = M + r * N;
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const int j = tl | deposit_bits<ML>(k);
            if (KQ_IN_RANGE(r * N + j, rows * N)) dst[j] = POST ? x[k] * fpost[j] : x[k] * inv_sqrt_n;
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) x[k] = nx[k];
    }
}

// ------------------------------------------- row transform in registers, n = 28 * 2^LG
// For n = 28 P (P = 2^LG, LG in [9, 10]: 14336 and 28672) with index j = a P + b (b
// fastest): every chunk a of P contiguous elements takes the Walsh-Hadamard transform H_P,
// then every column b takes the 28-point mix across the chunks. Fourteen groups of P / 16
// threads; group g transforms chunks g and g + 14 one after the other with the four-bit
// register phases of rht.cuh (each group with its own exchange buffer) and leaves them in
// a shared-memory copy of the row; then each thread mixes whole columns b (mix28_paley)
// and writes the 28 results straight to global memory, consecutive threads at consecutive
// b. At n = 28672 the 112 KB row copy leaves one CTA (28 warps) per SM, at 14336 two (the
// launch bound holds the registers to what two CTAs of 14 warps can share: down_8b's
// rotation stage 2.89 -> 2.42 ms against one CTA per SM); the
// warps of the other groups keep loads in flight while one group waits on its chunk.
// (Seven groups of four chunks each, with the next row prefetched into registers,
// measured 14.6-14.8 against 13.3 ms for the rotation stage of the 70B down_proj layer.)
template <int LG, bool POST>
__global__ void __launch_bounds__(14 * (1 << LG) / 16, LG == 9 ? 2 : 1) rht_rows28_reg_kernel(float* __restrict__ M, int64_t rows,
                                                                              int pre_mode, int post_mode,
                                                                              const int8_t* __restrict__ sign,
                                                                              const float* __restrict__ s,
                                                                              float inv_sqrt_n) {
    constexpr int G = 14, P = 1 << LG, N = 28 * P, TG = P / 16, T = G * TG, NPH = rr_phases(LG), CPG = 28 / G;
    constexpr uint32_t ML = rr_mask(LG, NPH - 1);
    static_assert(NPH == 3, "three register phases for P = 512 and 1024");
    extern __shared__ __align__(16) float sm28[];
    float* v = sm28;                                         // [N]
    const int t = threadIdx.x, g = t / TG, tl = t - g * TG;
    float* buf = sm28 + N + g * P;                           // this group's exchange buffer
    const int tw = deposit_bits<(P - 1) & ~ML>(tl);
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
#pragma unroll
        for (int c = 0; c < CPG; ++c) {
            const int a = g + G * c;
            float x[16];
            const float4* src = reinterpret_cast<const float4*>(M + r * N + a * P + 16 * tl);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float4 w4 = src[q];
                x[4 * q] = w4.x;
                x[4 * q + 1] = w4.y;
                x[4 * q + 2] = w4.z;
                x[4 * q + 3] = w4.w;
            }
            float f[16];
            factors16(pre_mode, sign, s, a * P + 16 * tl, f);
#pragma unroll
            for (int k = 0; k < 16; ++k) x[k] *= f[k];
            fwht_kbits<0xFu>(x);
            rr_transpose<LG, 1, true>(x, buf, tl);
            rr_transpose<LG, 2, true>(x, buf, tl);
#pragma unroll
            for (int k = 0; k < 16; ++k)
                if (KQ_IN_RANGE(a * P + (tw | deposit_bits<ML>(k)), N)) v[a * P + (tw | deposit_bits<ML>(k))] = x[k];
        }
        __syncthreads();
        float* dst = M + r * N;
        for (int b = t; b < P; b += T) {
            float y[28];
#pragma unroll
            for (int a = 0; a < 28; ++a) y[a] = v[a * P + b];
            mix28_paley(y, [&](int a, float val) {
                const int j = a * P + b;
                if (KQ_IN_RANGE(r * N + j, rows * N))
                    dst[j] = POST ? val * (factor(post_mode, sign, s, j) * inv_sqrt_n) : val * inv_sqrt_n;
            });
        }
        __syncthreads();   // v is rewritten by the next row
    }
}

// M [n x n] <- M^T in place: the CTA at (bj, bi) of an nt x nt grid of 64 x 64 tiles swaps
// tiles (bi, bj) and (bj, bi) through shared memory when bi <= bj (a diagonal tile is
// transposed alone); the CTAs below the diagonal have nothing to do. Each of the 256
// threads has 16 loads of each tile in flight before the barrier.
constexpr int TT = 64;
__global__ void __launch_bounds__(256) transpose_sq_kernel(float* __restrict__ M, int64_t n) {
    __shared__ float a[TT][TT + 1], b[TT][TT + 1];
    const int64_t bi = blockIdx.y, bj = blockIdx.x;
    if (bi > bj) return;
    const int tx = threadIdx.x & 63, ty = threadIdx.x >> 6;   // 64 x 4
    float ra[TT / 4], rb[TT / 4];   // all loads in flight before the shared-memory stores
#pragma unroll
    for (int q = 0; q < TT / 4; ++q) {
        const int yy = ty + 4 * q;
        const int64_t r1 = bi * TT + yy, c1 = bj * TT + tx;
        ra[q] = (r1 < n && c1 < n) ? M[r1 * n + c1] : 0.0f;
        const int64_t r2 = bj * TT + yy, c2 = bi * TT + tx;
        rb[q] = (bi != bj && r2 < n && c2 < n) ? M[r2 * n + c2] : 0.0f;
    }
#pragma unroll
    for (int q = 0; q < TT / 4; ++q) {
        a[ty + 4 * q][tx] = ra[q];
        b[ty + 4 * q][tx] = rb[q];
    }
    __syncthreads();
    for (int yy = ty; yy < TT; yy += 4) {
        const int64_t r1 = bj * TT + yy, c1 = bi * TT + tx;   // tile (bj, bi) <- a^T
        if (r1 < n && c1 < n && KQ_IN_RANGE(r1 * n + c1, n * n)) M[r1 * n + c1] = a[tx][yy];
        const int64_t r2 = bi * TT + yy, c2 = bj * TT + tx;   // tile (bi, bj) <- b^T
        if (bi != bj && r2 < n && c2 < n && KQ_IN_RANGE(r2 * n + c2, n * n)) M[r2 * n + c2] = b[tx][yy];
    }
}

// ------------------------------------------------- column transform in registers
// One radix stage along the row index of M [n x ncols] with the whole radix in registers:
// a work item is a group of R rows (base + i S, i < R) and a strip of columns; the TPC =
// max(1, R / 32) consecutive lanes of a column each hold V = R / TPC of its values (lane u:
// rows u V .. u V + V - 1), transform them (butterflies for R = 2^k, the cross-lane stages
// by shuffles; the 28-point mix for R = 28) and store them back. Consecutive columns sit in
// consecutive lane groups, so every row load of a warp is 32 / TPC contiguous floats. The
// group's pre- and post-factors are staged once in shared memory. No shared-memory round
// trips between radix-2 stages (a tiled shared-memory version with radix-8 sub-stages moved
// each element through shared memory several times per pass: 2.35 against ~4 TB/s).
template <int V>
__device__ __forceinline__ void fwht_regs(float (&x)[V]) {
#pragma unroll
    for (int h = 1; h < V; h <<= 1)
#pragma unroll
        for (int i = 0; i < V; i += 2 * h)
#pragma unroll
            for (int j = i; j < i + h; ++j) {
                const float a = x[j], b = x[j + h];
                x[j] = a + b;
                x[j + h] = a - b;
            }
}

template <int R>
__global__ void __launch_bounds__(128) rht_cols_reg_kernel(float* __restrict__ M, int n, int64_t ncols, int S,
                                                           int pre_mode, int post_mode,
                                                           const int8_t* __restrict__ sign,
                                                           const float* __restrict__ s, float post_scale) {
    constexpr int TPC = R > 32 ? R / 32 : 1, V = R / TPC, CPB = 128 / TPC;   // columns per CTA
    __shared__ float pf[R], qf[R];
    const int u = threadIdx.x % TPC, cl = threadIdx.x / TPC;
    const int64_t ngroups = n / R;
    const int64_t nstrips = (ncols + CPB - 1) / CPB;
    for (int64_t w = blockIdx.x; w < ngroups * nstrips; w += gridDim.x) {
        const int64_t g = w / nstrips, c0 = (w - g * nstrips) * CPB;
        const int64_t base = (g / S) * static_cast<int64_t>(R) * S + (g % S);
        __syncthreads();   // the previous item's factors are no longer read
        for (int i = threadIdx.x; i < R; i += blockDim.x) {
            const int64_t r = base + static_cast<int64_t>(i) * S;
            pf[i] = factor(pre_mode, sign, s, r);
            qf[i] = factor(post_mode, sign, s, r) * post_scale;
        }
        __syncthreads();
        const int64_t c = c0 + cl;
        const bool act = c < ncols;   // whole lane groups agree (a column's lanes share c)
        const int64_t step = static_cast<int64_t>(S) * ncols;
        float* col = M + (base + static_cast<int64_t>(u) * V * S) * ncols + (act ? c : 0);
        float x[V];
#pragma unroll
        for (int i = 0; i < V; ++i) x[i] = act ? col[i * step] * pf[u * V + i] : 0.0f;
        if constexpr (R == 28) {
            float y[28];
            mix28_paley(x, [&](int a, float v) { y[a] = v; });
#pragma unroll
            for (int i = 0; i < 28; ++i) x[i] = y[i];
        } else {
            fwht_regs<V>(x);
#pragma unroll
            for (int m = 1; m < TPC; m <<= 1) {   // the stages across the column's lanes
                const bool hi = (u & m) != 0;
#pragma unroll
                for (int i = 0; i < V; ++i) {
                    const float o = __shfl_xor_sync(0xffffffffu, x[i], m);
                    x[i] = hi ? o - x[i] : x[i] + o;
                }
            }
        }
        if (act) {
#pragma unroll
            for (int i = 0; i < V; ++i)
                if (KQ_IN_RANGE((col - M) + i * step, static_cast<int64_t>(n) * ncols))
                    col[i * step] = x[i] * qf[u * V + i];
        }
    }
}

template <int R>
kq_status launch_cols_reg(float* M, int64_t n, int64_t ncols, int S, int pm, int qm, const int8_t* sign,
                          const float* s, float ps, cudaStream_t stream) {
    const int64_t items = (n / R) * cdiv(ncols, 128 / (R > 32 ? R / 32 : 1));
    const int64_t grid = std::min<int64_t>(items, static_cast<int64_t>(num_sms()) * 16);
    rht_cols_reg_kernel<R><<<static_cast<unsigned>(grid), 128, 0, stream>>>(M, static_cast<int>(n), ncols, S, pm, qm,
                                                                         sign, s, ps);
    KQ_LAUNCH_CHECK("rht_cols_reg_kernel");
    return KQ_OK;
}


// ------------------------------------------------------------------------ scales
__device__ __forceinline__ float quarter_root_ratio(float h, double a) {
    if (!(h > 0.0f) || !(a > 0.0)) return 1.0f;   // dead channel (or NaN): scale 1
    return static_cast<float>(sqrt(sqrt(static_cast<double>(h) / a)));
}

// (h / a)^e; e == 1/4 takes the same sqrt(sqrt()) as Eq. (rescale)'s scales.
__device__ __forceinline__ float ratio_pow(float h, double a, float e) {
    if (e == 0.25f) return quarter_root_ratio(h, a);
    if (!(h > 0.0f) || !(a > 0.0)) return 1.0f;
    return static_cast<float>(pow(static_cast<double>(h) / a, static_cast<double>(e)));
}

// a_j = ||W[:, j]||^2 and s_x[j] = (H_X[j][j] / a_j)^e (e = 1/4: Eq. rescale). Block (CS_X, CS_Y).
__global__ void colscale_kernel(const float* __restrict__ W, int64_t d_out, int64_t d_in,
                                const float* __restrict__ HX, int64_t hstride, float* __restrict__ s_x, float e) {
    const int64_t j = static_cast<int64_t>(blockIdx.x) * CS_X + threadIdx.x;
    const double a = col_sumsq(W, d_out, d_in, j);
    if (threadIdx.y == 0 && j < d_in) s_x[j] = ratio_pow(HX[j * hstride], a, e);
}

// r_i = ||W[i, :]||^2 and s_g[i] = (H_G[i][i] / r_i)^e (1 when H_G is NULL). Warp per row.
__global__ void rowscale_kernel(const float* __restrict__ W, int64_t d_out, int64_t d_in,
                                const float* __restrict__ HG, int64_t hstride, float* __restrict__ s_g, float e) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * (blockDim.x / 32) + threadIdx.x / 32;
    if (i >= d_out) return;
    const double acc = row_sumsq(W + i * d_in, d_in);
    if ((threadIdx.x & 31) == 0) s_g[i] = HG ? ratio_pow(HG[i * hstride], acc, e) : 1.0f;
}

// Squared column norms (a) and squared row norms (r) of W in fp64, for the BiIP statistics.
__global__ void colnorm2_kernel(const float* __restrict__ W, int64_t d_out, int64_t d_in, double* __restrict__ a) {
    const int64_t j = static_cast<int64_t>(blockIdx.x) * CS_X + threadIdx.x;
    const double v = col_sumsq(W, d_out, d_in, j);
    if (threadIdx.y == 0 && j < d_in) a[j] = v;
}
__global__ void rownorm2_kernel(const float* __restrict__ W, int64_t d_out, int64_t d_in, double* __restrict__ r) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * (blockDim.x / 32) + threadIdx.x / 32;
    if (i >= d_out) return;
    const double v = row_sumsq(W + i * d_in, d_in);
    if ((threadIdx.x & 31) == 0) r[i] = v;
}

// out = [CV_in, CV_out, rho_in, rho_out]: coefficient of variation (population standard
// deviation over mean) of the column and row norms sqrt(a), sqrt(r), and
// rho = (sum sqrt(h a))^2 / (sum h sum a) with h the factor's diagonal (entries 2 and 3 are
// left as they are when the factor is NULL). One CTA, fp64, fixed order.
__global__ void biip_stats_kernel(const double* __restrict__ a, int64_t d_in, const double* __restrict__ r,
                                  int64_t d_out, const float* __restrict__ HX, int64_t xs,
                                  const float* __restrict__ HG, int64_t gs, double* __restrict__ out) {
    __shared__ double part[6][32];
    double v[6];
    for (int side = 0; side < 2; ++side) {
        const double* n2 = side == 0 ? a : r;
        const int64_t n = side == 0 ? d_in : d_out;
        const float* H = side == 0 ? HX : HG;
        const int64_t hs = side == 0 ? xs : gs;
        for (int k = 0; k < 6; ++k) v[k] = 0.0;
        for (int64_t j = threadIdx.x; j < n; j += blockDim.x) {
            const double nn = sqrt(n2[j]);
            v[0] += nn;                       // sum of norms
            v[1] += n2[j];                    // sum of squared norms
            if (H) {
                const double h = static_cast<double>(H[j * hs]);
                v[2] += sqrt(h * n2[j]);
                v[3] += h;
            }
        }
        for (int k = 0; k < 4; ++k) {
            for (int o = 16; o > 0; o >>= 1) v[k] += __shfl_xor_sync(0xffffffffu, v[k], o);
            if ((threadIdx.x & 31) == 0) part[k][threadIdx.x >> 5] = v[k];
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            double t[4] = {0.0, 0.0, 0.0, 0.0};
            for (int w = 0; w < static_cast<int>(blockDim.x / 32); ++w)
                for (int k = 0; k < 4; ++k) t[k] += part[k][w];
            const double mean = t[0] / static_cast<double>(n);
            const double var = fmax(t[1] / static_cast<double>(n) - mean * mean, 0.0);
            out[side] = sqrt(var) / mean;
            if (H) out[2 + side] = t[2] * t[2] / (t[3] * t[1]);
        }
        __syncthreads();
    }
}

// out = [tr H_X, tr H_G, product, tr H_X', tr H_G', product'] with tr H' = sum h_j / s_j^2.
// A NULL factor leaves its entries of out as they are; the products use whatever out then
// holds for the other side (so the two sides may be filled by two calls, X side first).
__global__ void traces_kernel(const float* __restrict__ HX, int64_t xstride, const float* __restrict__ s_x,
                              int64_t d_in, const float* __restrict__ HG, int64_t gstride,
                              const float* __restrict__ s_g, int64_t d_out, double* out) {
    __shared__ double part[4][32];
    double v[4] = {0.0, 0.0, 0.0, 0.0};
    if (HX)
        for (int64_t j = threadIdx.x; j < d_in; j += blockDim.x) {
            const double h = HX[j * xstride];
            const double sc = s_x ? static_cast<double>(s_x[j]) : 1.0;
            v[0] += h;
            v[2] += h / (sc * sc);
        }
    if (HG)
        for (int64_t i = threadIdx.x; i < d_out; i += blockDim.x) {
            const double h = HG[i * gstride];
            const double sc = s_g ? static_cast<double>(s_g[i]) : 1.0;
            v[1] += h;
            v[3] += h / (sc * sc);
        }
    for (int k = 0; k < 4; ++k) {
        for (int o = 16; o > 0; o >>= 1) v[k] += __shfl_xor_sync(0xffffffffu, v[k], o);
        if ((threadIdx.x & 31) == 0) part[k][threadIdx.x >> 5] = v[k];
    }
    __syncthreads();
    if (threadIdx.x < 32) {
        for (int k = 0; k < 4; ++k) {
            double x = threadIdx.x < blockDim.x / 32 ? part[k][threadIdx.x] : 0.0;
            for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
            v[k] = x;
        }
        if (threadIdx.x == 0) {
            if (HX) {
                out[0] = v[0];
                out[3] = v[2];
            }
            if (HG) {
                out[1] = v[1];
                out[4] = v[3];
            }
            out[2] = out[0] * out[1];
            out[5] = out[3] * out[4];
        }
    }
}

// diag(A^T A): per (row split, 128-column strip) CTA, fp32 partial sums of squares over
// 32 rows at a time added into fp64; partial[split][j] in the workspace.
constexpr int DG_COLS = 128;
constexpr int DG_ROWS = 8;   // row groups per CTA (256 threads = 8 x 32, 4 columns per thread)

__global__ void __launch_bounds__(256) factor_diag_partial_kernel(const uint16_t* __restrict__ A, int64_t T, int64_t d,
                                                                  int64_t lda, int64_t rows_per_split,
                                                                  double* __restrict__ partial) {
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int64_t c0 = static_cast<int64_t>(blockIdx.x) * DG_COLS + 4 * tx;
    const int64_t r_begin = static_cast<int64_t>(blockIdx.y) * rows_per_split;
    const int64_t r_end = min(T, r_begin + rows_per_split);
    const bool vec = c0 + 4 <= d && (lda & 3) == 0 && (reinterpret_cast<uintptr_t>(A) & 7u) == 0;
    double acc[4] = {0.0, 0.0, 0.0, 0.0};
    float p[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    int cnt = 0;
    // products of bf16 values are exact in fp32; 32-row fp32 partials are added in fp64
#pragma unroll 4
    for (int64_t r = r_begin + ty; r < r_end; r += DG_ROWS) {
        const uint16_t* row = A + r * lda + c0;
        uint32_t b[4] = {0u, 0u, 0u, 0u};
        if (vec) {
            const uint2 v = *reinterpret_cast<const uint2*>(row);
            b[0] = v.x & 0xFFFFu;
            b[1] = v.x >> 16;
            b[2] = v.y & 0xFFFFu;
            b[3] = v.y >> 16;
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) b[u] = (c0 + u < d) ? row[u] : 0u;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const float x = __uint_as_float(b[u] << 16);
            p[u] = fmaf(x, x, p[u]);
        }
        if (++cnt == 32) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                acc[u] += p[u];
                p[u] = 0.0f;
            }
            cnt = 0;
        }
    }
    __shared__ double part[DG_ROWS][DG_COLS];
#pragma unroll
    for (int u = 0; u < 4; ++u) part[ty][4 * tx + u] = acc[u] + p[u];
    __syncthreads();
    if (ty == 0) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            double sum = 0.0;
            for (int y = 0; y < DG_ROWS; ++y) sum += part[y][4 * tx + u];
            if (c0 + u < d) partial[static_cast<int64_t>(blockIdx.y) * d + c0 + u] = sum;
        }
    }
}

// diag[j] = sum over splits (fixed order), trace = sum_j (one CTA, fixed order per thread).
__global__ void factor_diag_reduce_kernel(const double* __restrict__ partial, int nsplit, int64_t d,
                                          float* __restrict__ diag, double* trace) {
    __shared__ double red[32];
    double t = 0.0;
    for (int64_t j = threadIdx.x; j < d; j += blockDim.x) {
        double s = 0.0;
        for (int q = 0; q < nsplit; ++q) s += partial[static_cast<int64_t>(q) * d + j];
        diag[j] = static_cast<float>(s);
        t += s;
    }
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = t;
    __syncthreads();
    if (threadIdx.x < 32) {
        t = threadIdx.x < blockDim.x / 32 ? red[threadIdx.x] : 0.0;
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (threadIdx.x == 0 && trace) *trace = t;
    }
}

int diag_splits(int64_t T, int64_t d) {
    const int64_t strips = cdiv(d, DG_COLS);
    int64_t s = cdiv(4 * static_cast<int64_t>(num_sms()), strips);
    s = std::max<int64_t>(1, std::min<int64_t>(s, cdiv(T, 256)));
    return static_cast<int>(std::min<int64_t>(s, 64));
}

// ------------------------------------------------------------------ host helpers
struct HadamardPlan {
    int P = 0;       // power-of-two factor
    int has28 = 0;   // n = 28 * P
};

bool plan_of(int64_t n, HadamardPlan* p) {
    if (n < 1 || n > 32768) return false;
    if ((n & (n - 1)) == 0) {
        p->P = static_cast<int>(n);
        p->has28 = 0;
        return true;
    }
    if (n % 28 == 0) {
        const int64_t q = n / 28;
        if ((q & (q - 1)) == 0 && q <= 1024) {
            p->P = static_cast<int>(q);
            p->has28 = 1;
            return true;
        }
    }
    return false;
}

int log2i(int64_t x) {
    int k = 0;
    while ((1ll << k) < x) ++k;
    return k;
}

template <int LG>
kq_status launch_rows_reg(float* M, int64_t rows, int pre, int post, const int8_t* sign, const float* s,
                          cudaStream_t stream) {
    constexpr int N = 1 << LG, T = N / 16;
    constexpr size_t smem = (3 * static_cast<size_t>(N) + N / 32) * sizeof(float);
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(rht_rows_reg_kernel<LG, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(smem)));
        KQ_CUDA(cudaFuncSetAttribute(rht_rows_reg_kernel<LG, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(smem)));
        return KQ_OK;
    }));
    // as many CTAs as fit on an SM by shared memory and threads, each walking rows
    const int64_t per_sm = std::max<int64_t>(1, std::min<int64_t>(static_cast<int64_t>((227 * 1024) / smem), 2048 / T));
    const int64_t grid = std::min<int64_t>(rows, static_cast<int64_t>(num_sms()) * per_sm);
    const float isn = static_cast<float>(1.0 / sqrt(static_cast<double>(N)));
    if (post == F_NONE)
        rht_rows_reg_kernel<LG, false><<<static_cast<unsigned>(grid), T, smem, stream>>>(M, rows, pre, post, sign, s, isn);
    else
        rht_rows_reg_kernel<LG, true><<<static_cast<unsigned>(grid), T, smem, stream>>>(M, rows, pre, post, sign, s, isn);
    KQ_LAUNCH_CHECK("rht_rows_reg_kernel");
    return KQ_OK;
}

template <int LG>
kq_status launch_rows28_reg(float* M, int64_t rows, int pre, int post, const int8_t* sign, const float* s,
                            cudaStream_t stream) {
    constexpr int P = 1 << LG, T = 14 * P / 16;
    constexpr size_t smem = (28 * static_cast<size_t>(P) + 14 * static_cast<size_t>(P)) * sizeof(float);
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(rht_rows28_reg_kernel<LG, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(smem)));
        KQ_CUDA(cudaFuncSetAttribute(rht_rows28_reg_kernel<LG, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(smem)));
        return KQ_OK;
    }));
    const int64_t per_sm = std::max<int64_t>(1, std::min<int64_t>(static_cast<int64_t>((227 * 1024) / smem), 2048 / T));
    const int64_t grid = std::min<int64_t>(rows, static_cast<int64_t>(num_sms()) * per_sm);
    const float isn = static_cast<float>(1.0 / sqrt(static_cast<double>(28 * P)));
    if (post == F_NONE)
        rht_rows28_reg_kernel<LG, false><<<static_cast<unsigned>(grid), T, smem, stream>>>(M, rows, pre, post, sign, s, isn);
    else
        rht_rows28_reg_kernel<LG, true><<<static_cast<unsigned>(grid), T, smem, stream>>>(M, rows, pre, post, sign, s, isn);
    KQ_LAUNCH_CHECK("rht_rows28_reg_kernel");
    return KQ_OK;
}

// M 16-byte aligned and n a power of two from 512 to 16384, or 28 * 512 / 28 * 1024: a
// register row transform.
bool rows_reg_ok(const float* M, int64_t n) {
    if ((reinterpret_cast<uintptr_t>(M) & 15u) != 0) return false;
    if (n == 28 * 512 || n == 28 * 1024) return true;
    return n >= 512 && n <= 16384 && (n & (n - 1)) == 0;
}

kq_status rows_transform(float* M, int64_t rows, int64_t n, int pre, int post, const int8_t* sign,
                         const float* s, cudaStream_t stream) {
    HadamardPlan p;
    if (!plan_of(n, &p)) return KQ_ERR_UNSUPPORTED;
    if (rows > 0 && rows_reg_ok(M, n) && p.has28 && (reinterpret_cast<uintptr_t>(sign) & 15u) == 0 &&
        (reinterpret_cast<uintptr_t>(s) & 15u) == 0) {
        if (p.P == 512) return launch_rows28_reg<9>(M, rows, pre, post, sign, s, stream);
        return launch_rows28_reg<10>(M, rows, pre, post, sign, s, stream);
    }
    if (rows > 0 && rows_reg_ok(M, n)) {
        switch (log2i(n)) {
            case 9: return launch_rows_reg<9>(M, rows, pre, post, sign, s, stream);
            case 10: return launch_rows_reg<10>(M, rows, pre, post, sign, s, stream);
            case 11: return launch_rows_reg<11>(M, rows, pre, post, sign, s, stream);
            case 12: return launch_rows_reg<12>(M, rows, pre, post, sign, s, stream);
            case 13: return launch_rows_reg<13>(M, rows, pre, post, sign, s, stream);
            case 14: return launch_rows_reg<14>(M, rows, pre, post, sign, s, stream);
            default: break;
        }
    }
    constexpr size_t kMaxSmem = 227 * 1024;
    const size_t row_bytes = static_cast<size_t>(n) * sizeof(float);
    const int dbl = 2 * row_bytes <= kMaxSmem ? 1 : 0;
    const size_t smem = (dbl ? 2 : 1) * row_bytes;
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(rht_rows_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(kMaxSmem)));
        KQ_CUDA(cudaFuncSetAttribute(rht_rows_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(kMaxSmem)));
        return KQ_OK;
    }));
    const int threads = n >= 512 ? 256 : 128;
    // as many CTAs as fit on an SM by shared memory (at most 8), each walking rows
    const int64_t per_sm = std::max<int64_t>(1, std::min<int64_t>(8, static_cast<int64_t>(kMaxSmem / smem)));
    const int64_t grid = std::min<int64_t>(rows, static_cast<int64_t>(num_sms()) * per_sm);
    if (grid > 0) {
        const float isn = static_cast<float>(1.0 / sqrt(static_cast<double>(n)));
        if (p.has28)
            rht_rows_kernel<true><<<static_cast<unsigned>(grid), threads, smem, stream>>>(
                M, rows, static_cast<int>(n), log2i(p.P), pre, post, sign, s, isn, dbl);
        else
            rht_rows_kernel<false><<<static_cast<unsigned>(grid), threads, smem, stream>>>(
                M, rows, static_cast<int>(n), log2i(p.P), pre, post, sign, s, isn, dbl);
        KQ_LAUNCH_CHECK("rht_rows_kernel");
    }
    return KQ_OK;
}

kq_status cols_transform(float* M, int64_t n, int64_t ncols, int pre, int post, const int8_t* sign,
                         const float* s, cudaStream_t stream) {
    HadamardPlan p;
    if (!plan_of(n, &p)) return KQ_ERR_UNSUPPORTED;
    // Radix stages: (R, S) pairs applied in order; S = product of earlier radices. Radix at
    // most 128 (values of a column spread over up to four lanes), as even as possible: n =
    // 8192 in two passes (64 x 128), each reading and writing M once.
    int R[4], S[4], ns = 0;
    const int kp = log2i(p.P);
    const int nst = (kp + 6) / 7;
    for (int st = 0, done = 0; st < nst; ++st) {
        const int kb = (kp - done) / (nst - st);
        R[ns] = 1 << kb;
        S[ns] = 1 << done;
        ++ns;
        done += kb;
    }
    if (p.has28) { R[ns] = 28; S[ns] = p.P; ++ns; }
    if (ns == 0) {   // n == 1: only the factors apply
        R[0] = 1; S[0] = 1; ns = 1;
    }
    const float post_scale = static_cast<float>(1.0 / sqrt(static_cast<double>(n)));
    for (int st = 0; st < ns; ++st) {
        const int pm = st == 0 ? pre : F_NONE, qm = st == ns - 1 ? post : F_NONE;
        const float ps = st == ns - 1 ? post_scale : 1.0f;
        kq_status rs = KQ_ERR_UNSUPPORTED;
        switch (R[st]) {
            case 1: rs = launch_cols_reg<1>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            case 2: rs = launch_cols_reg<2>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            case 4: rs = launch_cols_reg<4>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            case 8: rs = launch_cols_reg<8>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            case 16: rs = launch_cols_reg<16>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            case 32: rs = launch_cols_reg<32>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            case 64: rs = launch_cols_reg<64>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            case 128: rs = launch_cols_reg<128>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            case 28: rs = launch_cols_reg<28>(M, n, ncols, S[st], pm, qm, sign, s, ps, stream); break;
            default: break;
        }
        if (rs != KQ_OK) return rs;
    }
    return KQ_OK;
}

// M <- R M R^T for M [n x n], R = H_n diag(pre) / sqrt(n) (pre from the factor mode). With
// the register row transform: B = M R^T (rows), B^T = R M^T, its rows give R M^T R^T, and a
// last transpose gives R M R^T -- four streaming passes instead of a row pass and two
// column passes; for a symmetric M (sym) R M^T R^T is already R M R^T up to rounding and the
// last transpose is left out. Otherwise the row and column transforms.
kq_status two_sided_transform(float* M, int64_t n, int pre, const int8_t* sign, const float* s, bool sym,
                              cudaStream_t stream) {
    kq_status st = rows_transform(M, n, n, pre, F_NONE, sign, s, stream);
    if (st != KQ_OK) return st;
    if (!rows_reg_ok(M, n)) return cols_transform(M, n, n, pre, F_NONE, sign, s, stream);
    const dim3 tg(static_cast<unsigned>(cdiv(n, TT)), static_cast<unsigned>(cdiv(n, TT)));
    transpose_sq_kernel<<<tg, 256, 0, stream>>>(M, n);
    KQ_LAUNCH_CHECK("transpose_sq_kernel");
    st = rows_transform(M, n, n, pre, F_NONE, sign, s, stream);
    if (st != KQ_OK || sym) return st;
    transpose_sq_kernel<<<tg, 256, 0, stream>>>(M, n);
    KQ_LAUNCH_CHECK("transpose_sq_kernel");
    return KQ_OK;
}

}  // namespace

KQ_DEBUG_UNIT(biip)
}  // namespace kq

using namespace kq;

namespace {
kq_status scales_impl(const float* W, int64_t d_out, int64_t d_in, const float* hx, int64_t xs, const float* hg,
                      int64_t gs, float* s_x, float* s_g, cudaStream_t stream, const char* who, float ex = 0.25f,
                      float eg = 0.25f) {
    if (!W || d_out < 1 || d_in < 1 || (!s_x && !s_g) || (s_x && !hx)) {
        set_error("%s: invalid arguments", who);
        return KQ_ERR_INVALID_ARG;
    }
    if (s_x) {
        colscale_kernel<<<static_cast<unsigned>(cdiv(d_in, CS_X)), dim3(CS_X, CS_Y), 0, stream>>>(W, d_out, d_in, hx, xs, s_x,
                                                                                               ex);
        KQ_LAUNCH_CHECK("colscale_kernel");
    }
    if (s_g) {
        rowscale_kernel<<<static_cast<unsigned>(cdiv(d_out, 8)), 256, 0, stream>>>(W, d_out, d_in, hg, gs, s_g, eg);
        KQ_LAUNCH_CHECK("rowscale_kernel");
    }
    return KQ_OK;
}

kq_status traces_impl(const float* hx, int64_t xs, const float* s_x, int64_t d_in, const float* hg, int64_t gs,
                      const float* s_g, int64_t d_out, double* out, cudaStream_t stream, const char* who) {
    if ((!hx && !hg) || !out || (hx && d_in < 1) || (hg && d_out < 1)) {
        set_error("%s: invalid arguments", who);
        return KQ_ERR_INVALID_ARG;
    }
    traces_kernel<<<1, 1024, 0, stream>>>(hx, xs, s_x, d_in, hg, gs, s_g, d_out, out);
    KQ_LAUNCH_CHECK("traces_kernel");
    return KQ_OK;
}
}  // namespace

extern "C" kq_status kq_compute_scales(const float* W, int64_t d_out, int64_t d_in, const float* H_X,
                                       const float* H_G, float* s_x, float* s_g, kq_stream_t stream_) {
    return scales_impl(W, d_out, d_in, H_X, d_in + 1, H_G, d_out + 1, s_x, s_g,
                       reinterpret_cast<cudaStream_t>(stream_), "kq_compute_scales");
}

extern "C" kq_status kq_compute_scales_diag(const float* W, int64_t d_out, int64_t d_in, const float* hx_diag,
                                            const float* hg_diag, float* s_x, float* s_g, kq_stream_t stream_) {
    return scales_impl(W, d_out, d_in, hx_diag, 1, hg_diag, 1, s_x, s_g, reinterpret_cast<cudaStream_t>(stream_),
                       "kq_compute_scales_diag");
}

extern "C" kq_status kq_compute_scales_exp(const float* W, int64_t d_out, int64_t d_in, const float* H_X,
                                           const float* H_G, float* s_x, float* s_g, float ex, float eg,
                                           kq_stream_t stream_) {
    if (!(ex >= 0.0f && ex <= 1.0f) || !(eg >= 0.0f && eg <= 1.0f)) {
        set_error("kq_compute_scales_exp: exponents must lie in [0, 1]");
        return KQ_ERR_INVALID_ARG;
    }
    return scales_impl(W, d_out, d_in, H_X, d_in + 1, H_G, d_out + 1, s_x, s_g, reinterpret_cast<cudaStream_t>(stream_),
                       "kq_compute_scales_exp", ex, eg);
}

extern "C" size_t kq_biip_stats_workspace(int64_t d_out, int64_t d_in) {
    if (d_out < 1 || d_in < 1) return 0;
    return static_cast<size_t>(d_out + d_in) * sizeof(double) + 256;
}

extern "C" kq_status kq_biip_stats(const float* W, int64_t d_out, int64_t d_in, const float* H_X, const float* H_G,
                                   double* out, void* ws, size_t ws_bytes, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!W || !out || d_out < 1 || d_in < 1) {
        set_error("kq_biip_stats: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (!ws || ws_bytes < kq_biip_stats_workspace(d_out, d_in) || (reinterpret_cast<uintptr_t>(ws) & 15u)) {
        set_error("kq_biip_stats: workspace must be 16-byte aligned and hold %zu bytes", kq_biip_stats_workspace(d_out, d_in));
        return KQ_ERR_WORKSPACE;
    }
    double* a = static_cast<double*>(ws);
    double* r = a + d_in;
    colnorm2_kernel<<<static_cast<unsigned>(cdiv(d_in, CS_X)), dim3(CS_X, CS_Y), 0, stream>>>(W, d_out, d_in, a);
    KQ_LAUNCH_CHECK("colnorm2_kernel");
    rownorm2_kernel<<<static_cast<unsigned>(cdiv(d_out, 8)), 256, 0, stream>>>(W, d_out, d_in, r);
    KQ_LAUNCH_CHECK("rownorm2_kernel");
    biip_stats_kernel<<<1, 1024, 0, stream>>>(a, d_in, r, d_out, H_X, d_in + 1, H_G, d_out + 1, out);
    KQ_LAUNCH_CHECK("biip_stats_kernel");
    return KQ_OK;
}

extern "C" kq_status kq_traces(const float* H_X, const float* s_x, int64_t d_in, const float* H_G,
                               const float* s_g, int64_t d_out, double* out, kq_stream_t stream_) {
    return traces_impl(H_X, d_in + 1, s_x, d_in, H_G, d_out + 1, s_g, d_out, out,
                       reinterpret_cast<cudaStream_t>(stream_), "kq_traces");
}

extern "C" kq_status kq_traces_diag(const float* hx_diag, const float* s_x, int64_t d_in, const float* hg_diag,
                                    const float* s_g, int64_t d_out, double* out, kq_stream_t stream_) {
    return traces_impl(hx_diag, 1, s_x, d_in, hg_diag, 1, s_g, d_out, out, reinterpret_cast<cudaStream_t>(stream_),
                       "kq_traces_diag");
}

extern "C" kq_status kq_rotate_in(float* W, int64_t d_out, int64_t d_in, float* H_X, const float* s_x,
                                  const int8_t* sign_v, int dir, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    HadamardPlan p;
    const bool sym = dir == KQ_FWD_SYM;
    if (sym) dir = KQ_FWD;
    if ((!W && !(H_X && dir == KQ_FWD)) || !sign_v || d_in < 1 || (W && d_out < 1) ||
        (dir != KQ_FWD && dir != KQ_INV)) {
        set_error("kq_rotate_in: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (!plan_of(d_in, &p)) {
        set_error("kq_rotate_in: d_in=%lld has no Hadamard construction", (long long)d_in);
        return KQ_ERR_UNSUPPORTED;
    }
    kq_status st;
    if (dir == KQ_FWD) {
        // W <- (W S_X) V^T: each row times sigma_j s_j, then H_n, then 1/sqrt(n).
        if (W) {
            st = rows_transform(W, d_out, d_in, s_x ? F_SMUL : F_SIGN, F_NONE, sign_v, s_x, stream);
            if (st != KQ_OK) return st;
        }
        if (H_X) {
            // H_X <- V S_X^-1 H_X S_X^-1 V^T: both sides scaled by sigma / s, then H_n twice.
            st = two_sided_transform(H_X, d_in, s_x ? F_SDIV : F_SIGN, sign_v, s_x, sym, stream);
            if (st != KQ_OK) return st;
        }
    } else {
        // W <- (W V) S_X^-1 = (W H_n) diag(sigma / s) / sqrt(n).
        st = rows_transform(W, d_out, d_in, F_NONE, s_x ? F_SDIV : F_SIGN, sign_v, s_x, stream);
        if (st != KQ_OK) return st;
    }
    return KQ_OK;
}

extern "C" kq_status kq_rotate_out(float* W, int64_t d_out, int64_t d_in, float* H_G, const float* s_g,
                                   const int8_t* sign_u, int dir, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    HadamardPlan p;
    const bool sym = dir == KQ_FWD_SYM;
    if (sym) dir = KQ_FWD;
    if ((!W && !(H_G && dir == KQ_FWD)) || !sign_u || d_out < 1 || (W && d_in < 1) ||
        (dir != KQ_FWD && dir != KQ_INV)) {
        set_error("kq_rotate_out: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (!plan_of(d_out, &p)) {
        set_error("kq_rotate_out: d_out=%lld has no Hadamard construction", (long long)d_out);
        return KQ_ERR_UNSUPPORTED;
    }
    kq_status st;
    if (dir == KQ_FWD) {
        // W <- U (S_G W): rows scaled by sigma_i s_i, then H_n along the row index.
        if (W) {
            st = cols_transform(W, d_out, d_in, s_g ? F_SMUL : F_SIGN, F_NONE, sign_u, s_g, stream);
            if (st != KQ_OK) return st;
        }
        if (H_G) {
            st = two_sided_transform(H_G, d_out, s_g ? F_SDIV : F_SIGN, sign_u, s_g, sym, stream);
            if (st != KQ_OK) return st;
        }
    } else {
        // W <- S_G^-1 U^T W = diag(sigma / s) H_n W / sqrt(n).
        st = cols_transform(W, d_out, d_in, F_NONE, s_g ? F_SDIV : F_SIGN, sign_u, s_g, stream);
        if (st != KQ_OK) return st;
    }
    return KQ_OK;
}

// Used by the check-only revert (check.cu).
namespace kq {
// Used by the inference call (infer.cu): rows <- V S^-1 rows (pre-factor sigma / s).
kq_status rotate_rows_pre_div(float* M, int64_t rows, int64_t n, const float* s, const int8_t* sign,
                              cudaStream_t stream) {
    return rows_transform(M, rows, n, s ? F_SDIV : F_SIGN, F_NONE, sign, s, stream);
}
kq_status rotate_rows_inv(float* M, int64_t rows, int64_t n, const float* s, const int8_t* sign,
                          cudaStream_t stream) {
    return rows_transform(M, rows, n, F_NONE, s ? F_SDIV : F_SIGN, sign, s, stream);
}
kq_status rotate_cols_inv(float* M, int64_t n, int64_t ncols, const float* s, const int8_t* sign,
                          cudaStream_t stream) {
    return cols_transform(M, n, ncols, F_NONE, s ? F_SDIV : F_SIGN, sign, s, stream);
}
}  // namespace kq

extern "C" size_t kq_factor_diag_workspace(int64_t T, int64_t d) {
    if (d < 1 || T < 0) return 0;
    return 64 * static_cast<size_t>(d) * sizeof(double) + 256;
}

extern "C" kq_status kq_factor_diag(const uint16_t* A, int64_t T, int64_t d, int64_t lda, float* diag, double* trace,
                                    void* ws, size_t ws_bytes, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!diag || d < 1 || T < 0 || (T > 0 && !A) || lda < d) {
        set_error("kq_factor_diag: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (!ws || ws_bytes < kq_factor_diag_workspace(T, d) || (reinterpret_cast<uintptr_t>(ws) & 15u)) {
        set_error("kq_factor_diag: workspace must be 16-byte aligned and hold %zu bytes", kq_factor_diag_workspace(T, d));
        return KQ_ERR_WORKSPACE;
    }
    const int nsplit = T > 0 ? diag_splits(T, d) : 1;
    double* partial = static_cast<double*>(ws);
    if (T > 0) {
        const int64_t rows_per_split = cdiv(T, nsplit);
        dim3 grid(static_cast<unsigned>(cdiv(d, DG_COLS)), static_cast<unsigned>(nsplit));
        factor_diag_partial_kernel<<<grid, 256, 0, stream>>>(A, T, d, lda, rows_per_split, partial);
        KQ_LAUNCH_CHECK("factor_diag_partial_kernel");
    } else {
        KQ_CUDA(cudaMemsetAsync(partial, 0, sizeof(double) * d, stream));
    }
    factor_diag_reduce_kernel<<<1, 1024, 0, stream>>>(partial, nsplit, d, diag, trace);
    KQ_LAUNCH_CHECK("factor_diag_reduce_kernel");
    return KQ_OK;
}
