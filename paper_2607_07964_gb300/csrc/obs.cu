// Stage 4: the column-wise OBS sweep with b-bit asymmetric grids.
//
// Paper: Sec. 2.1 Eq. (obs_update) (compensation -(w_p - q_p)/[H^-1]_pp [H^-1]_{p,p+1:}),
// Algorithm 2 (inner column loop over a block of B columns with error E, then the lazy
// trailing update W[:, i+B:] -= E R[i:i+B, i+B:]), Proposition 1 (H_G cancels, so only
// L = R^T enters). With the GPTAQ correction P (Proposition 1, Algorithm 2) each column j
// also adds w_j P[j, k] to the later columns k, w_j being column j's value just before it
// is quantized; the lazy update then subtracts [E | -Wpre] [R ; P]. GPTQ mode: no P.
//
// Every fp32 operation is written with an explicit round-to-nearest intrinsic so the
// compiler cannot contract or reorder it; the order is:
//   grid      scale = (xmax - xmin) / (2^b - 1), zero = rint(-xmin / scale)
//   column j  q = clamp(rint(w / scale) + zero, 0, 2^b - 1); what = scale * (q - zero)
//             E = (w - what) / R_jj;  w_k = fma(-E, R_jk, w_k) for k in (j, block end)
//             with P: w_k = fma(w_j, P_jk, fma(-E, R_jk, w_k))
//   trailing  acc = fma(E_k, R_kc, acc) over ascending k; with P continuing
//             acc = fma(-wpre_k, P_kc, acc) over ascending k; w_c = w_c - acc
// Kernels:
//   rowgrid_kernel   per-row grid (group = 0) from the whole row before the sweep
//   pack_r_kernel    the diagonal 128 x 128 blocks of R in the block kernel's layout
//   obs_block_kernel 8 lanes per row, 16 columns per lane; the block's R in shared memory
//   trailing_kernel  128 x 128 output tiles of the shared tile GEMM (tile_gemm.cuh)
//   colloss_kernel   col_loss[j] = sum over rows of E_j^2, fixed order (sumsq.cuh)
#include <math.h>

#include <cstdlib>
#include <type_traits>

#include "kq_common.cuh"
#include "tile_gemm.cuh"
#include "sumsq.cuh"
#include "trail_tc.cuh"

namespace kq {
namespace {

constexpr int BLK = 128;          // block size B (Algorithm 2); the only supported value
constexpr int SPB = 8;            // blocks per super-panel of the two-level lazy update

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
    if (lane == 0 && KQ_IN_RANGE(r, d_out)) {
        scale[r] = g.scale;
        zero[r] = static_cast<int32_t>(g.zero);
        gscale[r] = g.scale;
        gzero[r] = g.zero;
    }
}

// One block [i0, e) of the sweep for all rows. A group of LPR = 8 lanes handles one row;
// lane position lp holds the CPL = 16 consecutive columns i0 + CPL lp + t of it in
// registers. Column j = CPL o + jj is owned by lane o: for each o (rolled loop) the 16
// columns are an unrolled loop, so every register index is a compile-time constant. Per
// column the owner's w_j is broadcast in the group, every lane computes the (identical)
// quantization and error, and every lane updates all CPL of its registers with R_jk. The
// updates of columns k < j (lanes before the owner, or the owner's own earlier columns)
// read R_jk = 0 or hit values that are no longer read, so no update needs a predicate and
// the live columns k > j see exactly the operations of the definition.
#ifndef KQ_OBS_LANES_PER_ROW
#define KQ_OBS_LANES_PER_ROW 8
#endif
constexpr int LPR = KQ_OBS_LANES_PER_ROW;   // lanes per row (8 or 16)
constexpr int CPL = BLK / LPR;              // columns per lane
constexpr int NV = CPL / 4;                 // float4 slots per lane
static_assert(LPR == 8 || LPR == 16, "lanes per row must be 8 or 16");
// 32 rows per CTA (8 warps): with 64 KB of shared memory and at most 128 registers a
// thread, a CTA fits beside one CTA of the 3xTF32 far-column update (129 KB, 320 threads),
// so block b + 1 runs while block b's far columns are updated (one CTA per SM up to 4864
// rows, two beyond).
constexpr int OBS_ROWS = 32;                // rows per CTA
constexpr int OBS_THREADS = OBS_ROWS * LPR; // 256 or 512
// With P the CTA holds both diagonal blocks (R and P, 128 KB): one CTA per SM, alone.
constexpr int OBS_ROWS_P = 32;
// Dynamic shared memory of the block kernel with the tensor-core fused update: R's block
// and 32 rows of E_prev (padded), 80.5 KB -- still beside a 129 KB far-update CTA.
constexpr int OBS_SMEM_MMA = (BLK * BLK + 32 * (BLK + 4)) * 4;
constexpr int OBS_THREADS_P = OBS_ROWS_P * LPR;

// Packed layout of one diagonal block of R: row j holds R[i0 + j][i0 + c] at pos(c). The
// CPL columns of lane lp fill slots [lp NV, lp NV + NV) of 16 bytes, rotated by lane so
// that the NV float4 loads of 8 consecutive lanes hit 8 distinct bank groups.
__host__ __device__ constexpr int slot_of(int lp, int v) { return lp * NV + ((v + ((lp * NV) >> 3)) & (NV - 1)); }
__device__ __forceinline__ int pos_of(int c) { return 4 * slot_of(c / CPL, (c % CPL) >> 2) + (c & 3); }

// Rp[b][j][pos(c)] = R[i0 + j][i1 + c] = Lt[i1 + c][i0 + j] (0 outside the matrix),
// i0 = b BLK, i1 = i0 + coff BLK: the diagonal blocks (coff = 0) or the blocks right of them
// (coff = 1). Block (32, 8) transposes one 32 x 32 tile through shared memory.
__global__ void pack_r_kernel(const float* __restrict__ Lt, int64_t n, float* __restrict__ Rp, int coff) {
    __shared__ float t[32][33];
    const int64_t i0 = static_cast<int64_t>(blockIdx.z) * BLK;
    const int64_t i1 = i0 + static_cast<int64_t>(coff) * BLK;
    const int c0 = blockIdx.y * 32, j0 = blockIdx.x * 32;
    for (int r = threadIdx.y; r < 32; r += 8) {
        const int64_t c = i1 + c0 + r, j = i0 + j0 + threadIdx.x;
        t[r][threadIdx.x] = (c < n && j < n) ? Lt[c * n + j] : 0.0f;
    }
    __syncthreads();
    float* out = Rp + static_cast<int64_t>(blockIdx.z) * BLK * BLK;
    for (int r = threadIdx.y; r < 32; r += 8) {
        const int j = j0 + r, c = c0 + threadIdx.x;
        if (KQ_IN_RANGE(j * BLK + pos_of(c), BLK * BLK)) out[j * BLK + pos_of(c)] = t[threadIdx.x][r];
    }
}

// Rq[b][c][k ^ (4 (c & 7))] = R[i0 + k][i1 + c] = Lt[i1 + c][i0 + k] (0 outside the matrix),
// i0 = b BLK, i1 = i0 + BLK: the block of R right of diagonal block b, column-major with
// the k index swizzled within 32-float groups, for the tensor-core form of the fused update
// (its fragment loads then hit 32 banks). Block (32, 8), one 32 x 32 tile per CTA; Lt rows
// are contiguous in k, so no transpose.
__global__ void pack_rq_mma_kernel(const float* __restrict__ Lt, int64_t n, float* __restrict__ Rq) {
    const int64_t i0 = static_cast<int64_t>(blockIdx.z) * BLK, i1 = i0 + BLK;
    const int k0 = blockIdx.x * 32, c0 = blockIdx.y * 32;
    float* out = Rq + static_cast<int64_t>(blockIdx.z) * BLK * BLK;
    for (int r = threadIdx.y; r < 32; r += 8) {
        const int c = c0 + r, k = k0 + threadIdx.x;
        const int64_t lr = i1 + c, lc = i0 + k;
        if (KQ_IN_RANGE(c * BLK + (k ^ (4 * (c & 7))), BLK * BLK))
            out[c * BLK + (k ^ (4 * (c & 7)))] = (lr < n && lc < n) ? Lt[lr * n + lc] : 0.0f;
    }
}

// The previous block's lazy update of this block column for the CTA's 32 rows on the tensor
// cores (mma.sync m16n8k8 tf32, 3xTF32 split): C = E_prev R_prev,this with E_prev staged in
// Es ([32][BLK + 4]) and R_prev,this in Rs (pack_rq_mma_kernel's layout); 8 warps of 16 x 32.
// C is left in Es (same layout) after a barrier.
__device__ __forceinline__ void prev_block_update_mma(float* Es, const float* Rs) {
    constexpr int ESLD = BLK + 4;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, g = lane >> 2, t4 = lane & 3;
    const int wr = wid >> 2, wc = wid & 3;
    float c[4][4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) c[nt][e] = 0.0f;
    const float* a0p = Es + (16 * wr + g) * ESLD;
    const float* a1p = a0p + 8 * ESLD;
#pragma unroll 2
    for (int ks = 0; ks < BLK; ks += 8) {
        const float a[4] = {a0p[ks + t4], a1p[ks + t4], a0p[ks + t4 + 4], a1p[ks + t4 + 4]};
        uint32_t ah[4], al[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float hi = tf32_hi(a[e]);
            ah[e] = __float_as_uint(hi);
            al[e] = __float_as_uint(a[e] - hi);
        }
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
            const int col = 32 * wc + 8 * nt + g;   // col & 7 == g
            const float b0 = Rs[col * BLK + ((ks + t4) ^ (4 * g))];
            const float b1 = Rs[col * BLK + ((ks + t4 + 4) ^ (4 * g))];
            const float bh0 = tf32_hi(b0), bh1 = tf32_hi(b1);
            const uint32_t bh[2] = {__float_as_uint(bh0), __float_as_uint(bh1)};
            const uint32_t bl[2] = {__float_as_uint(b0 - bh0), __float_as_uint(b1 - bh1)};
            mma_tf32(c[nt], al, bh);
            mma_tf32(c[nt], ah, bl);
            mma_tf32(c[nt], ah, bh);
        }
    }
    __syncthreads();   // every warp is done with Es
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
        const int r = 16 * wr + g, col = 32 * wc + 8 * nt + 2 * t4;
        Es[r * ESLD + col] = c[nt][0];
        Es[r * ESLD + col + 1] = c[nt][1];
        Es[(r + 8) * ESLD + col] = c[nt][2];
        Es[(r + 8) * ESLD + col + 1] = c[nt][3];
    }
    __syncthreads();
}

__device__ __forceinline__ float group_min(float v) {
    for (int o = LPR / 2; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float group_max(float v) {
    for (int o = LPR / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// A lane's CPL columns [cb, cb + CPL) of row r of the block starting at column i0 (0 past
// the block end nb or past the last row).
// NC: through the read-only path (data this kernel does not write); else plain loads.
template <bool VEC, bool NC = true>
__device__ __forceinline__ void load_cols(const float* __restrict__ W, int64_t r, int64_t d_out, int64_t d_in,
                                          int64_t i0, int cb, int nb, float (&w)[CPL]) {
    const bool live = r < d_out;
    const float* src = W + r * d_in + i0 + cb;
    if (VEC && cb + CPL <= nb) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const float4* p = reinterpret_cast<const float4*>(src) + v;
            const float4 x = live ? (NC ? __ldg(p) : *p) : make_float4(0.f, 0.f, 0.f, 0.f);
            w[4 * v] = x.x;
            w[4 * v + 1] = x.y;
            w[4 * v + 2] = x.z;
            w[4 * v + 3] = x.w;
        }
    } else {
#pragma unroll
        for (int t = 0; t < CPL; ++t) w[t] = (live && cb + t < nb) ? src[t] : 0.0f;
    }
}

template <bool VEC>
__device__ __forceinline__ void store_cols(float* W, int64_t r, int64_t d_out, int64_t d_in, int64_t i0, int cb,
                                           int nb, const float (&w)[CPL]) {
    if (r >= d_out || !KQ_IN_RANGE(r * d_in + i0 + cb + min(CPL, nb - cb) - 1, d_out * d_in)) return;
    float* dst = W + r * d_in + i0 + cb;
    if (VEC && cb + CPL <= nb) {
#pragma unroll
        for (int v = 0; v < NV; ++v)
            reinterpret_cast<float4*>(dst)[v] = make_float4(w[4 * v], w[4 * v + 1], w[4 * v + 2], w[4 * v + 3]);
    } else {
#pragma unroll
        for (int t = 0; t < CPL; ++t)
            if (cb + t < nb) dst[t] = w[t];
    }
}

// w -= E_prev R_prev,this for one row: the previous block's lazy update of this block
// column, in the order of the trailing update (acc = fma(E_k, R_kc, acc) over ascending k,
// then w - acc). Rq: the block of R (rows = the previous block's columns) packed like the
// diagonal blocks, in shared memory; ep: this lane's CPL entries of the row of E_prev.
__device__ __forceinline__ void prev_block_update(const float* Rq, const float (&ep)[CPL], int lp, int gbase,
                                                  float (&w)[CPL]) {
    float acc[CPL];
#pragma unroll
    for (int t = 0; t < CPL; ++t) acc[t] = 0.0f;
#pragma unroll 1
    for (int o = 0; o < LPR; ++o) {
#pragma unroll
        for (int jj = 0; jj < CPL; ++jj) {
            const float ek = __shfl_sync(0xffffffffu, ep[jj], gbase | o);
            const float* rr = Rq + (CPL * o + jj) * BLK;
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const float4 x = *reinterpret_cast<const float4*>(rr + 4 * slot_of(lp, v));
                acc[4 * v] = __fmaf_rn(ek, x.x, acc[4 * v]);
                acc[4 * v + 1] = __fmaf_rn(ek, x.y, acc[4 * v + 1]);
                acc[4 * v + 2] = __fmaf_rn(ek, x.z, acc[4 * v + 2]);
                acc[4 * v + 3] = __fmaf_rn(ek, x.w, acc[4 * v + 3]);
            }
        }
    }
#pragma unroll
    for (int t = 0; t < CPL; ++t) w[t] = __fsub_rn(w[t], acc[t]);
}

// VEC: d_in % 16 == 0 and W, codes (and pre_q) 16-byte aligned, so a lane's CPL columns
// of W, E and codes move as 16-byte vectors. HASP: with the GPTAQ correction; Pp is P's
// diagonal block packed like R's, and the block's -Wpre goes to Q (fp32 trailing update)
// or to Qh + Ql (tensor-core trailing update).
template <bool VEC, bool HASP>
__global__ void __launch_bounds__(HASP ? OBS_THREADS_P : OBS_THREADS, HASP ? 1 : 2) obs_block_kernel(
    float* __restrict__ W, int64_t d_out, int64_t d_in, const float* __restrict__ Rp, int64_t i0,
    int bits, int group, const float* __restrict__ gscale, const float* __restrict__ gzero,
    uint8_t* __restrict__ codes, float* __restrict__ scale, int32_t* __restrict__ zero,
    float* __restrict__ E, float* __restrict__ pre_q, float* __restrict__ Eh, float* __restrict__ El,
    const float* __restrict__ Pp, float* __restrict__ Q, float* __restrict__ Qh, float* __restrict__ Ql,
    const float* __restrict__ Rq, int fused_mma, int* info) {
    extern __shared__ __align__(16) float Rs[];   // [BLK][BLK], packed (pack_r_kernel); then P's
    float* Ps = Rs + BLK * BLK;
    const bool fused = !HASP && Rq != nullptr;
    // With Rq, the buffer first holds the previous block's R_prev,this for the fused update.
    for (int e = threadIdx.x; e < BLK * BLK / 4; e += blockDim.x) cp_async16(Rs + 4 * e, (fused ? Rq : Rp) + 4 * e, 16);
    if (HASP)
        for (int e = threadIdx.x; e < BLK * BLK / 4; e += blockDim.x) cp_async16(Ps + 4 * e, Pp + 4 * e, 16);
    cp_async_commit();
    const int nb = static_cast<int>(min(static_cast<int64_t>(BLK), d_in - i0));
    const float maxq = static_cast<float>((1 << bits) - 1);
    const int lane = threadIdx.x & 31;
    const int lp = lane & (LPR - 1);
    const int gbase = lane & ~(LPR - 1);
    const int cb = CPL * lp;                       // first column of this lane in the block
    const int64_t ngroups = group ? (d_in + group - 1) / group : 1;
    const int warps = blockDim.x / 32;
    constexpr int RPW = 32 / LPR;                  // rows per warp
    const int64_t rstride = static_cast<int64_t>(gridDim.x) * warps * RPW;
    const int64_t rw0 = (static_cast<int64_t>(blockIdx.x) * warps + threadIdx.x / 32) * RPW;
    float w[CPL];
    if (fused) {
        // Each row of this CTA goes back to W updated, and the sweep below reads it with
        // plain loads; then the diagonal block replaces R_prev,this in shared memory.
        cp_async_wait<0>();
        __syncthreads();
        if (VEC && fused_mma && rstride >= d_out) {
            // tensor-core form (one row group per CTA: its 32 rows from blockIdx.x * 32)
            constexpr int ESLD = BLK + 4;
            float* Es = Rs + BLK * BLK;
            const int64_t row0 = static_cast<int64_t>(blockIdx.x) * warps * RPW;
            for (int q = threadIdx.x; q < 32 * (BLK / 4); q += blockDim.x) {
                const int rr = q / (BLK / 4), c4 = q % (BLK / 4);
                const bool lv = row0 + rr < d_out;
                cp_async16(Es + rr * ESLD + 4 * c4, lv ? E + (row0 + rr) * d_in + (i0 - BLK) + 4 * c4 : E, lv ? 16 : 0);
            }
            cp_async_commit();
            cp_async_wait<0>();
            __syncthreads();
            prev_block_update_mma(Es, Rs);
            const int64_t r = rw0 + lane / LPR;
            const float* cu = Es + (r - row0) * ESLD + cb;
            load_cols<VEC>(W, r, d_out, d_in, i0, cb, nb, w);
#pragma unroll
            for (int t = 0; t < CPL; ++t) w[t] = __fsub_rn(w[t], cu[t]);
            store_cols<VEC>(W, r, d_out, d_in, i0, cb, nb, w);
        } else {
            for (int64_t rw = rw0; rw < d_out; rw += rstride) {
                const int64_t r = rw + lane / LPR;
                float ep[CPL];
                load_cols<VEC>(E, r, d_out, d_in, i0 - BLK, cb, BLK, ep);
                load_cols<VEC>(W, r, d_out, d_in, i0, cb, nb, w);
                prev_block_update(Rs, ep, lp, gbase, w);
                store_cols<VEC>(W, r, d_out, d_in, i0, cb, nb, w);
            }
        }
        __syncthreads();
        for (int e = threadIdx.x; e < BLK * BLK / 4; e += blockDim.x) cp_async16(Rs + 4 * e, Rp + 4 * e, 16);
        cp_async_commit();
        load_cols<VEC, false>(W, rw0 + lane / LPR, d_out, d_in, i0, cb, nb, w);
    } else {
        // The first row's weights load while R is staged.
        load_cols<VEC>(W, rw0 + lane / LPR, d_out, d_in, i0, cb, nb, w);
    }
    cp_async_wait<0>();
    __syncthreads();   // every thread reaches it
    // Reciprocals of the block's diagonal R_jj for the column steps' divisions.
    __shared__ float rds[BLK];
    for (int j = threadIdx.x; j < BLK; j += blockDim.x) rds[j] = j < nb ? div_recip(Rs[j * BLK + pos_of(j)]) : 0.0f;
    __syncthreads();
    for (int64_t rw = rw0; rw < d_out; rw += rstride) {
        const int64_t r = rw + lane / LPR;
        const bool live = r < d_out;
        if (rw != rw0) {
            if (fused)
                load_cols<VEC, false>(W, r, d_out, d_in, i0, cb, nb, w);
            else
                load_cols<VEC>(W, r, d_out, d_in, i0, cb, nb, w);
        }
        Grid g;
        if (group) {
            float mn = 0.0f, mx = 0.0f;
#pragma unroll
            for (int t = 0; t < CPL; ++t)
                if (cb + t < nb) {
                    mn = fminf(mn, w[t]);
                    mx = fmaxf(mx, w[t]);
                }
            g = make_grid(group_min(mn), group_max(mx), maxq);
            if (live && lp == 0 && KQ_IN_RANGE(r * ngroups + i0 / group, d_out * ngroups)) {
                const int64_t gi = r * ngroups + i0 / group;
                scale[gi] = g.scale;
                zero[gi] = static_cast<int32_t>(g.zero);
            }
        } else {
            g.scale = live ? gscale[r] : 1.0f;
            g.zero = live ? gzero[r] : 0.0f;
        }
        const float ys = div_recip(g.scale);
        bool finite = true;   // every value quantized in this row group was finite
        // The column steps of this row group; EXACT: IEEE divisions, else div_rn_fast, with
        // the return value telling whether every operand was inside its exact range.
        auto sweep = [&](auto exact_tag) -> bool {
        constexpr bool EXACT = decltype(exact_tag)::value;
        bool ok = true;
#pragma unroll 1
        for (int o = 0; o < LPR; ++o) {
            if (CPL * o >= nb) break;   // uniform across the CTA
            float e[CPL];
            float wq[HASP ? CPL : 1];   // the values before quantization (with P only)
            (void)wq;
            uint32_t cq[NV];
#pragma unroll
            for (int v = 0; v < NV; ++v) cq[v] = 0u;
#pragma unroll
            for (int jj = 0; jj < CPL; ++jj) {
                const int j = CPL * o + jj;
                e[jj] = 0.0f;
                if (j < nb) {   // uniform across the CTA
                    const float* rr = Rs + j * BLK;
                    const float dj = rr[4 * slot_of(o, jj >> 2) + (jj & 3)];
                    const float yd = rds[j];
                    float4 rv[NV];
#pragma unroll
                    for (int v = 0; v < NV; ++v) rv[v] = *reinterpret_cast<const float4*>(rr + 4 * slot_of(lp, v));
                    const float wj = __shfl_sync(0xffffffffu, w[jj], gbase | o);
                    finite = finite & (fabsf(wj) <= 3.402823466e38f);
                    float q0;
                    if constexpr (EXACT) {
                        q0 = __fdiv_rn(wj, g.scale);
                    } else {
                        q0 = div_rn_fast(wj, g.scale, ys);
                        ok = ok & div_rn_fast_ok(wj, ys);
                    }
                    float qq = __fadd_rn(rintf(q0), g.zero);
                    qq = fminf(fmaxf(qq, 0.0f), maxq);
                    const float what = __fmul_rn(g.scale, __fsub_rn(qq, g.zero));
                    const float dif = __fsub_rn(wj, what);
                    float err;
                    if constexpr (EXACT) {
                        err = __fdiv_rn(dif, dj);
                    } else {
                        err = div_rn_fast(dif, dj, yd);
                        ok = ok & div_rn_fast_ok(dif, yd);
                    }
                    e[jj] = err;
                    cq[jj >> 2] |= static_cast<uint32_t>(qq) << (8 * (jj & 3));
                    if (pre_q && live && lp == o && KQ_IN_RANGE(r * d_in + i0 + j, d_out * d_in))
                        pre_q[r * d_in + i0 + j] = wj;
                    if constexpr (HASP) {
                        wq[jj] = wj;
                        const float* pr = Ps + j * BLK;
                        float4 pv[NV];
#pragma unroll
                        for (int v = 0; v < NV; ++v) pv[v] = *reinterpret_cast<const float4*>(pr + 4 * slot_of(lp, v));
#pragma unroll
                        for (int v = 0; v < NV; ++v) {
                            w[4 * v] = __fmaf_rn(wj, pv[v].x, __fmaf_rn(-err, rv[v].x, w[4 * v]));
                            w[4 * v + 1] = __fmaf_rn(wj, pv[v].y, __fmaf_rn(-err, rv[v].y, w[4 * v + 1]));
                            w[4 * v + 2] = __fmaf_rn(wj, pv[v].z, __fmaf_rn(-err, rv[v].z, w[4 * v + 2]));
                            w[4 * v + 3] = __fmaf_rn(wj, pv[v].w, __fmaf_rn(-err, rv[v].w, w[4 * v + 3]));
                        }
                    } else {
#pragma unroll
                        for (int v = 0; v < NV; ++v) {
                            w[4 * v] = __fmaf_rn(-err, rv[v].x, w[4 * v]);
                            w[4 * v + 1] = __fmaf_rn(-err, rv[v].y, w[4 * v + 1]);
                            w[4 * v + 2] = __fmaf_rn(-err, rv[v].z, w[4 * v + 2]);
                            w[4 * v + 3] = __fmaf_rn(-err, rv[v].w, w[4 * v + 3]);
                        }
                    }
                } else if constexpr (HASP) {
                    wq[jj] = 0.0f;
                }
            }
            if (live && lp == o && KQ_IN_RANGE(r * d_in + i0 + min(CPL * o + CPL, nb) - 1, d_out * d_in)) {
                const int64_t ob = r * d_in + i0 + CPL * o;
                if (VEC && CPL * o + CPL <= nb) {
#pragma unroll
                    for (int v = 0; v < NV; ++v)
                        reinterpret_cast<float4*>(E + ob)[v] = make_float4(e[4 * v], e[4 * v + 1], e[4 * v + 2], e[4 * v + 3]);
                    if constexpr (NV == 4) {
                        *reinterpret_cast<uint4*>(codes + ob) = make_uint4(cq[0], cq[1], cq[2], cq[3]);
                    } else {
                        *reinterpret_cast<uint2*>(codes + ob) = make_uint2(cq[0], cq[1]);
                    }
                    if (Eh) {   // tensor-core trailing update: E = E_hi + E_lo
#pragma unroll
                        for (int v = 0; v < NV; ++v) {
                            float h[4], l[4];
#pragma unroll
                            for (int t = 0; t < 4; ++t) {
                                h[t] = tf32_hi(e[4 * v + t]);
                                l[t] = e[4 * v + t] - h[t];
                            }
                            reinterpret_cast<float4*>(Eh + ob)[v] = make_float4(h[0], h[1], h[2], h[3]);
                            reinterpret_cast<float4*>(El + ob)[v] = make_float4(l[0], l[1], l[2], l[3]);
                        }
                    }
                    if constexpr (HASP) {   // -Wpre of the block, for the trailing update
                        if (Qh) {
#pragma unroll
                            for (int v = 0; v < NV; ++v) {
                                float h[4], l[4];
#pragma unroll
                                for (int t = 0; t < 4; ++t) {
                                    h[t] = tf32_hi(-wq[4 * v + t]);
                                    l[t] = -wq[4 * v + t] - h[t];
                                }
                                reinterpret_cast<float4*>(Qh + ob)[v] = make_float4(h[0], h[1], h[2], h[3]);
                                reinterpret_cast<float4*>(Ql + ob)[v] = make_float4(l[0], l[1], l[2], l[3]);
                            }
                        } else {
#pragma unroll
                            for (int v = 0; v < NV; ++v)
                                reinterpret_cast<float4*>(Q + ob)[v] =
                                    make_float4(-wq[4 * v], -wq[4 * v + 1], -wq[4 * v + 2], -wq[4 * v + 3]);
                        }
                    }
                } else {
#pragma unroll
                    for (int t = 0; t < CPL; ++t)
                        if (CPL * o + t < nb) {
                            E[ob + t] = e[t];
                            codes[ob + t] = static_cast<uint8_t>(cq[t >> 2] >> (8 * (t & 3)));
                            if (Eh) {
                                const float h = tf32_hi(e[t]);
                                Eh[ob + t] = h;
                                El[ob + t] = e[t] - h;
                            }
                            if constexpr (HASP) {
                                if (Qh) {
                                    const float h = tf32_hi(-wq[t]);
                                    Qh[ob + t] = h;
                                    Ql[ob + t] = -wq[t] - h;
                                } else {
                                    Q[ob + t] = -wq[t];
                                }
                            }
                        }
                }
            }
        }
        return ok;
        };
        if (!__all_sync(0xffffffffu, sweep(std::false_type{}))) {
            // an operand outside the fast division's range in this warp's rows: the row
            // group again from its start, with IEEE divisions (same outputs overwritten)
            if (fused)
                load_cols<VEC, false>(W, r, d_out, d_in, i0, cb, nb, w);
            else
                load_cols<VEC>(W, r, d_out, d_in, i0, cb, nb, w);
            sweep(std::true_type{});
        }
        if (!__all_sync(0xffffffffu, finite) && lane == 0) record_error(info, -KQ_ERR_NONFINITE);
    }
}

// W[:, cb:ce] -= E[:, i0:i0+kb] R[i0:i0+kb, cb:ce] with R[k][c] = Lt[c][k]: 128 x 128 output
// tiles of the shared tile GEMM (acc = fma(E_k, R_kc, acc) over ascending k), then w = w - acc.
// With P (Q = -Wpre, P[k][c] = Pt[c][k]) the sum continues with acc = fma(Q_k, P_kc, acc).
template <bool VEC>
__global__ void __launch_bounds__(G_THREADS, 2) trailing_kernel(float* __restrict__ W, const float* __restrict__ E,
                                                                const float* __restrict__ Lt, int64_t d_out,
                                                                int64_t d_in, int64_t i0, int kb, int64_t cb,
                                                                int64_t ce, const float* __restrict__ Q,
                                                                const float* __restrict__ Pt) {
    extern __shared__ __align__(16) float sm[];
    const int64_t r0 = static_cast<int64_t>(blockIdx.y) * GT;
    const int64_t c0 = cb + static_cast<int64_t>(blockIdx.x) * GT;
    const int arows = static_cast<int>(min(static_cast<int64_t>(GT), d_out - r0));
    const int bcols = static_cast<int>(min(static_cast<int64_t>(GT), ce - c0));
    float acc[8][8];
    gemm_tile<false, VEC>(E + r0 * d_in + i0, d_in, arows, Lt + c0 * d_in + i0, d_in, bcols, kb, acc, sm);
    if (Pt) gemm_tile<false, VEC, false>(Q + r0 * d_in + i0, d_in, arows, Pt + c0 * d_in + i0, d_in, bcols, kb, acc, sm);
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
                if (rr < arows && cc < bcols && KQ_IN_RANGE((r0 + rr) * d_in + c0 + cc, d_out * d_in))
                    W[(r0 + rr) * d_in + c0 + cc] = __fsub_rn(wv[i][j], acc[4 * h + i][j]);
            }
    }
}

// col_loss[j] = sum over rows of E[r][j]^2 in a fixed order (fp32 runs, fp64 across them).
// Block (CS_X, CS_Y).
__global__ void colloss_kernel(const float* __restrict__ E, int64_t d_out, int64_t d_in,
                               float* __restrict__ col_loss) {
    const int64_t j = static_cast<int64_t>(blockIdx.x) * CS_X + threadIdx.x;
    const double a = col_sumsq(E, d_out, d_in, j);
    if (threadIdx.y == 0 && j < d_in && KQ_IN_RANGE(j, d_in)) col_loss[j] = static_cast<float>(a);
}

struct ObsWs {
    float* Rp;      // packed diagonal blocks of R, nblk x BLK x BLK
    float* Rq;      // packed blocks of R right of them (block b: rows of b, columns of b + 1)
    float* E;       // d_out x d_in
    float* gscale;  // d_out
    float* gzero;   // d_out
    float* Eh;      // tensor-core mode: E_hi, E_lo [d_out x d_in], Lt_hi, Lt_lo [d_in x d_in]
    float* El;
    float* Lh;
    float* Ll;
    float* Pp;      // with P: packed diagonal blocks of P; -Wpre [d_out x d_in] (fp32 mode)
    float* Q;
    float* Qh;      // with P, tensor-core mode: (-Wpre)_hi, _lo [d_out x d_in], Pt_hi, Pt_lo
    float* Ql;
    float* Ph;
    float* Pl;
};

inline size_t align256(size_t b) { return (b + 255) & ~static_cast<size_t>(255); }

size_t ws_base_bytes(int64_t d_out, int64_t d_in) {
    return align256((2 * static_cast<size_t>(cdiv(d_in, BLK)) * BLK * BLK + static_cast<size_t>(d_out) * d_in +
                     2 * static_cast<size_t>(d_out)) * sizeof(float));
}

// Byte sizes of the parts in carve order.
struct WsParts {
    size_t base, blk, wide, sq;
};
WsParts parts_of(int64_t d_out, int64_t d_in) {
    WsParts p;
    p.base = ws_base_bytes(d_out, d_in);
    p.blk = align256(static_cast<size_t>(cdiv(d_in, BLK)) * BLK * BLK * sizeof(float));
    p.wide = align256(static_cast<size_t>(d_out) * d_in * sizeof(float));
    p.sq = align256(static_cast<size_t>(d_in) * d_in * sizeof(float));
    return p;
}

size_t ws_bytes_of(int64_t d_out, int64_t d_in, int mode, bool with_p) {
    const WsParts p = parts_of(d_out, d_in);
    const bool tc = mode == KQ_TRAIL_3XTF32;
    size_t b = p.base;
    if (tc) b += 2 * p.wide + 2 * p.sq;
    if (with_p) b += p.blk + (tc ? 2 * p.wide + 2 * p.sq : p.wide);
    return b + 256;
}

ObsWs carve(void* ws, int64_t d_out, int64_t d_in, int mode, bool with_p) {
    const WsParts sz = parts_of(d_out, d_in);
    const bool tc = mode == KQ_TRAIL_3XTF32;
    ObsWs o;
    o.Rp = static_cast<float*>(ws);
    o.Rq = o.Rp + cdiv(d_in, BLK) * BLK * BLK;
    o.E = o.Rq + cdiv(d_in, BLK) * BLK * BLK;
    o.gscale = o.E + d_out * d_in;
    o.gzero = o.gscale + d_out;
    o.Eh = o.El = o.Lh = o.Ll = o.Pp = o.Q = o.Qh = o.Ql = o.Ph = o.Pl = nullptr;
    uint8_t* p = static_cast<uint8_t*>(ws) + sz.base;
    auto take = [&](size_t bytes) {
        float* f = reinterpret_cast<float*>(p);
        p += bytes;
        return f;
    };
    if (tc) {
        o.Eh = take(sz.wide);
        o.El = take(sz.wide);
        o.Lh = take(sz.sq);
        o.Ll = take(sz.sq);
    }
    if (with_p) {
        o.Pp = take(sz.blk);
        if (tc) {
            o.Qh = take(sz.wide);
            o.Ql = take(sz.wide);
            o.Ph = take(sz.sq);
            o.Pl = take(sz.sq);
        } else {
            o.Q = take(sz.wide);
        }
    }
    return o;
}

}  // namespace

KQ_DEBUG_UNIT(obs)
}  // namespace kq

using namespace kq;

extern "C" size_t kq_obs_quantize_workspace(int64_t d_out, int64_t d_in, int block, int mode, int with_p) {
    (void)block;
    if (d_out < 1 || d_in < 1 || (mode != KQ_TRAIL_FP32 && mode != KQ_TRAIL_3XTF32)) return 0;
    return ws_bytes_of(d_out, d_in, mode, with_p != 0);
}

extern "C" kq_status kq_obs_quantize(float* W, int64_t d_out, int64_t d_in, const float* Lt, const float* Pt,
                                     int bits, int group, int block, int mode, uint8_t* codes, float* scale,
                                     int32_t* zero, float* col_loss, float* pre_q, int* info, void* ws,
                                     size_t ws_bytes, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!W || !Lt || !codes || !scale || !zero || d_out < 1 || d_in < 1 || bits < 1 || bits > 8) {
        set_error("kq_obs_quantize: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (block != BLK || (group != 0 && group != block)) {
        set_error("kq_obs_quantize: block must be %d and group 0 or equal to block", BLK);
        return KQ_ERR_UNSUPPORTED;
    }
    if (mode != KQ_TRAIL_FP32 && mode != KQ_TRAIL_3XTF32) {
        set_error("kq_obs_quantize: unknown trailing-update mode %d", mode);
        return KQ_ERR_INVALID_ARG;
    }
    const bool tc = mode == KQ_TRAIL_3XTF32;
    const bool hp = Pt != nullptr;
    if (tc && ((d_in % 4) != 0 || (reinterpret_cast<uintptr_t>(W) & 15u) != 0)) {
        set_error("kq_obs_quantize: the tensor-core trailing update needs d_in %% 4 == 0 and a 16-byte aligned W");
        return KQ_ERR_UNSUPPORTED;
    }
    if (hp && ((d_in % 16) != 0 || (reinterpret_cast<uintptr_t>(W) & 15u) || (reinterpret_cast<uintptr_t>(codes) & 15u) ||
               (reinterpret_cast<uintptr_t>(Pt) & 15u))) {
        set_error("kq_obs_quantize: the drift correction needs d_in %% 16 == 0 and 16-byte aligned W, codes, Pt");
        return KQ_ERR_UNSUPPORTED;
    }
    if (!ws || ws_bytes < ws_bytes_of(d_out, d_in, mode, hp) || (reinterpret_cast<uintptr_t>(ws) & 255u)) {
        set_error("kq_obs_quantize: workspace must be 256-byte aligned and hold %zu bytes",
                  ws_bytes_of(d_out, d_in, mode, hp));
        return KQ_ERR_WORKSPACE;
    }
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(obs_block_kernel<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     OBS_SMEM_MMA));
        KQ_CUDA(cudaFuncSetAttribute(obs_block_kernel<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     BLK * BLK * 4));
        // Whole shared memory on the SM, so that a CTA fits beside a far-update CTA.
        KQ_CUDA(cudaFuncSetAttribute(obs_block_kernel<true, false>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                     cudaSharedmemCarveoutMaxShared));
        KQ_CUDA(cudaFuncSetAttribute(obs_block_kernel<false, false>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                     cudaSharedmemCarveoutMaxShared));
        KQ_CUDA(cudaFuncSetAttribute(obs_block_kernel<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     2 * BLK * BLK * 4));
        KQ_CUDA(cudaFuncSetAttribute(trailing_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(G_SMEM)));
        KQ_CUDA(cudaFuncSetAttribute(trailing_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(G_SMEM)));
        return KQ_OK;
    }));
    ObsWs o = carve(ws, d_out, d_in, mode, hp);
    TrailMaps maps;
    if (tc) {
        kq_status st0 = split_tf32(Lt, d_in * d_in, o.Lh, o.Ll, stream);
        if (st0 != KQ_OK) return st0;
        if ((st0 = maps.init(o.Eh, o.El, o.Lh, o.Ll, d_out, d_in)) != KQ_OK) return st0;
        if ((st0 = maps.set_w(W, d_out, d_in)) != KQ_OK) return st0;
        if (hp) {
            if ((st0 = split_tf32(Pt, d_in * d_in, o.Ph, o.Pl, stream)) != KQ_OK) return st0;
            if ((st0 = maps.init_p(o.Qh, o.Ql, o.Ph, o.Pl, d_out, d_in)) != KQ_OK) return st0;
        }
    }
    if (group == 0) {
        rowgrid_kernel<<<static_cast<unsigned>(cdiv(d_out, 8)), 256, 0, stream>>>(W, d_out, d_in, bits, scale,
                                                                                zero, o.gscale, o.gzero);
        KQ_LAUNCH_CHECK("rowgrid_kernel");
    }
    const bool vec = (d_in % 4 == 0) && (reinterpret_cast<uintptr_t>(Lt) % 16 == 0);
    const bool bvec = (d_in % 16 == 0) && (reinterpret_cast<uintptr_t>(W) % 16 == 0) &&
                      (reinterpret_cast<uintptr_t>(codes) % 16 == 0);
    const int64_t nblk = cdiv(d_in, BLK);
    const int64_t row_ctas = hp ? std::min<int64_t>(cdiv(d_out, OBS_ROWS_P), static_cast<int64_t>(num_sms()))
                                : std::min<int64_t>(cdiv(d_out, OBS_ROWS), 2 * static_cast<int64_t>(num_sms()));
    pack_r_kernel<<<dim3(BLK / 32, BLK / 32, static_cast<unsigned>(nblk)), dim3(32, 8), 0, stream>>>(Lt, d_in, o.Rp, 0);
    KQ_LAUNCH_CHECK("pack_r_kernel");
    // the blocks of R right of the diagonal ones, for the fused update: the tensor-core
    // form's layout in the 3xTF32 mode, the block kernel's own otherwise
    const bool fuse_ok = !hp && nblk > 1 && row_ctas <= static_cast<int64_t>(num_sms()) &&
                         d_out * d_in <= (int64_t{24} << 20);
    const bool mma_fused = fuse_ok && tc && bvec;
    if (fuse_ok && mma_fused) {
        pack_rq_mma_kernel<<<dim3(BLK / 32, BLK / 32, static_cast<unsigned>(nblk - 1)), dim3(32, 8), 0, stream>>>(
            Lt, d_in, o.Rq);
        KQ_LAUNCH_CHECK("pack_rq_mma_kernel");
    } else if (fuse_ok) {
        pack_r_kernel<<<dim3(BLK / 32, BLK / 32, static_cast<unsigned>(nblk - 1)), dim3(32, 8), 0, stream>>>(Lt, d_in,
                                                                                                          o.Rq, 1);
        KQ_LAUNCH_CHECK("pack_r_kernel");
    }
    if (hp) {   // P[i0 + j][i0 + c] = Pt[i0 + c][i0 + j]: the same packing as R from Lt
        pack_r_kernel<<<dim3(BLK / 32, BLK / 32, static_cast<unsigned>(nblk)), dim3(32, 8), 0, stream>>>(Pt, d_in, o.Pp, 0);
        KQ_LAUNCH_CHECK("pack_r_kernel");
    }
    // GPTQ mode: block b's kernel first applies the previous block's update of its own
    // columns (E_{b-1} R_{b-1,b}, fused), and the update of the columns beyond block b + 1
    // runs on a library side stream beside block b + 1, whose CTAs share the SMs with it.
    // Block b waits only for the far update of block b - 2 (the last one that writes its
    // columns); the two far-update events alternate. With P: after block b the update of
    // block column b + 1 runs on the caller's stream (the next block kernel waits for it),
    // the columns beyond on the side stream beside block b + 1.
    // Every column receives the block updates in block order either way. The fused update
    // is fp32 in the trailing update's order in the fp32 mode, and on the tensor cores
    // (mma.sync, 3xTF32) in the 3xTF32 mode, like the far updates there.
    SideStream* side = nblk > 2 ? side_stream(stream) : nullptr;
    bool forked = false;
    bool far_pending[2] = {false, false};
    // 128 x 64 far-update tiles (a CTA fits beside a block-kernel CTA) while the block kernel
    // runs one CTA per SM and the far updates take about as long as the block kernels
    // (their mean, ~d_out d_in / 2 multiply-adds per block, against ~35 us a block: up to
    // d_out d_in ~ 24M). Otherwise nothing fits beside the block kernel, or the sweep waits
    // on the far updates, and 128 x 128 tiles are faster.
    const bool narrow = !hp && row_ctas <= static_cast<int64_t>(num_sms()) && d_out * d_in <= (int64_t{24} << 20);
    // The previous block's update fused into the block kernel: only then, so that nothing
    // but the far update shares the SMs with the block kernel.
    const bool fuse = narrow;
    auto trailing = [&](int64_t i0, int kb, int64_t cb, int64_t ce, cudaStream_t st) -> kq_status {
        if (tc) return trail_tc(maps, W, d_out, d_in, i0, cb, ce, hp, narrow, kb, info, st);
        dim3 grid(static_cast<unsigned>(cdiv(ce - cb, GT)), static_cast<unsigned>(cdiv(d_out, GT)));
        if (vec)
            trailing_kernel<true><<<grid, G_THREADS, G_SMEM, st>>>(W, o.E, Lt, d_out, d_in, i0, kb, cb, ce, o.Q, Pt);
        else
            trailing_kernel<false><<<grid, G_THREADS, G_SMEM, st>>>(W, o.E, Lt, d_out, d_in, i0, kb, cb, ce, o.Q, Pt);
        KQ_LAUNCH_CHECK("trailing_kernel");
        return KQ_OK;
    };
    auto block_launch = [&](int64_t b, const float* rq) {
        const int64_t i0 = b * BLK;
        const float* rp = o.Rp + b * BLK * BLK;
        if (hp)
            obs_block_kernel<true, true><<<static_cast<unsigned>(row_ctas), OBS_THREADS_P, 2 * BLK * BLK * 4, stream>>>(
                W, d_out, d_in, rp, i0, bits, group, o.gscale, o.gzero, codes, scale, zero, o.E, pre_q, o.Eh, o.El,
                o.Pp + b * BLK * BLK, o.Q, o.Qh, o.Ql, nullptr, 0, info);
        else if (bvec)
            obs_block_kernel<true, false><<<static_cast<unsigned>(row_ctas), OBS_THREADS, mma_fused ? OBS_SMEM_MMA : BLK * BLK * 4,
                                             stream>>>(
                W, d_out, d_in, rp, i0, bits, group, o.gscale, o.gzero, codes, scale, zero, o.E, pre_q, o.Eh, o.El,
                nullptr, nullptr, nullptr, nullptr, rq, mma_fused ? 1 : 0, info);
        else
            obs_block_kernel<false, false><<<static_cast<unsigned>(row_ctas), OBS_THREADS, BLK * BLK * 4, stream>>>(
                W, d_out, d_in, rp, i0, bits, group, o.gscale, o.gzero, codes, scale, zero, o.E, pre_q, o.Eh, o.El,
                nullptr, nullptr, nullptr, nullptr, rq, 0, info);
    };
    // Two levels for the large layers on the tensor cores (super-panels of SPB blocks, the
    // GPTQ lazy update grouped once more): inside a super-panel each block updates the next
    // block column on the caller's stream and the rest of the super-panel's columns on the
    // side stream (K = 128); after a super-panel's last block one update with the whole
    // super-panel's K covers every column beyond it -- the next super-panel's columns on the
    // caller's stream, the rest on the second side stream beside the next super-panel's
    // blocks -- so each W tile beyond is read and written once per super-panel instead of
    // once per block. Every column still receives the block updates in block order (the
    // long update drains its accumulator into W one block's K at a time).
    const bool two_level = tc && !hp && !fuse && nblk > SPB;
    if (two_level) {
        constexpr int64_t SPW = static_cast<int64_t>(SPB) * BLK;
        bool in_pending = false;    // the in-panel update of the previous block (side stream)
        bool far_pending = false;   // the far update of the previous super-panel (second side stream)
        cudaStream_t s_in = side ? side->s : stream;
        cudaStream_t s_far = side ? side->s2 : stream;
        for (int64_t b = 0; b < nblk; ++b) {
            const int64_t i0 = b * BLK;
            block_launch(b, nullptr);
            KQ_LAUNCH_CHECK("obs_block_kernel");
            const int64_t nb0 = i0 + BLK;                               // next block column
            if (nb0 >= d_in) break;
            const int64_t sp0 = (b / SPB) * SPW;                         // this super-panel
            const int64_t spe = std::min(d_in, sp0 + SPW);
            if (side) KQ_CUDA(cudaEventRecord(side->ev[0], stream));     // E of this block ready
            kq_status st;
            if (nb0 < spe) {
                if (in_pending) {   // it wrote the next block column too
                    KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));
                    in_pending = false;
                }
                const int64_t nb1 = std::min(spe, nb0 + BLK);
                st = trailing(i0, BLK, nb0, nb1, stream);
                if (st != KQ_OK) return st;
                if (nb1 < spe) {
                    if (side) KQ_CUDA(cudaStreamWaitEvent(s_in, side->ev[0], 0));
                    st = trailing(i0, BLK, nb1, spe, s_in);
                    if (st != KQ_OK) return st;
                    if (side) {
                        KQ_CUDA(cudaEventRecord(side->ev[1], s_in));
                        in_pending = true;
                    }
                }
            } else {
                const int64_t sp1 = std::min(d_in, spe + SPW);           // the next super-panel's end
                if (far_pending) {   // the previous super-panel's far update wrote these columns
                    KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[0], 0));
                    far_pending = false;
                }
                st = trail_tc_long(maps, d_out, d_in, sp0, static_cast<int>(spe - sp0), spe, sp1, info, stream);
                if (st != KQ_OK) return st;
                if (sp1 < d_in) {
                    if (side) KQ_CUDA(cudaStreamWaitEvent(s_far, side->ev[0], 0));
                    st = trail_tc_long(maps, d_out, d_in, sp0, static_cast<int>(spe - sp0), sp1, d_in, info, s_far);
                    if (st != KQ_OK) return st;
                    if (side) {
                        KQ_CUDA(cudaEventRecord(side->ev2[0], s_far));
                        far_pending = true;
                    }
                }
            }
        }
        if (in_pending) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));
        if (far_pending) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[0], 0));
    } else if (fuse && tc) {
        // Pairs of blocks (2s, 2s + 1). Block 2s + 1 applies block 2s's update of its columns
        // itself; after the pair, its update (K = 256, still applied 128 of K at a time) of
        // the next pair's columns runs on the caller's stream just before the next pair,
        // and that of the columns beyond on the side stream beside the next pair. The
        // next-pair update waits for the side update of the pair before (it wrote the same
        // columns); the side updates alternate two events.
        bool rest_pending[2] = {false, false};
        for (int64_t b = 0; b < nblk; ++b) {
            const int64_t i0 = b * BLK;
            const int64_t pr = b / 2;
            kq_status st;
            if ((b & 1) == 0 && b >= 2) {
                if (rest_pending[pr & 1]) {   // the side update of pair pr - 2
                    KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[pr & 1], 0));
                    rest_pending[pr & 1] = false;
                }
                st = trailing(i0 - 2 * BLK, 2 * BLK, i0, std::min<int64_t>(d_in, i0 + 2 * BLK), stream);
                if (st != KQ_OK) return st;
            }
            block_launch(b, (b & 1) ? o.Rq + (b - 1) * BLK * BLK : nullptr);
            KQ_LAUNCH_CHECK("obs_block_kernel");
            if ((b & 1) == 0) continue;
            const int64_t nb2 = std::min<int64_t>(d_in, i0 + 3 * BLK);   // beyond the next pair
            if (nb2 >= d_in) continue;
            cudaStream_t fs = stream;
            if (side) {
                KQ_CUDA(cudaEventRecord(side->ev[0], stream));   // E of the pair ready
                KQ_CUDA(cudaStreamWaitEvent(side->s, side->ev[0], 0));
                fs = side->s;
            }
            st = trailing(i0 - BLK, 2 * BLK, nb2, d_in, fs);
            if (st != KQ_OK) return st;
            if (side) {
                KQ_CUDA(cudaEventRecord(side->ev2[pr & 1], side->s));
                rest_pending[pr & 1] = true;
            }
        }
        for (int q = 0; q < 2; ++q)
            if (rest_pending[q]) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[q], 0));
    } else {
        for (int64_t i0 = 0; i0 < d_in; i0 += BLK) {
            const int64_t b = i0 / BLK;
            const int kb = static_cast<int>(std::min<int64_t>(BLK, d_in - i0));
            const float* rq = fuse && b > 0 ? o.Rq + (b - 1) * BLK * BLK : nullptr;
            if (fuse && far_pending[b & 1]) {   // the far update of block b - 2
                KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[b & 1], 0));
                far_pending[b & 1] = false;
            }
            block_launch(b, rq);
            KQ_LAUNCH_CHECK("obs_block_kernel");
            const int64_t nb0 = i0 + kb;                                // next block column
            if (nb0 >= d_in) break;
            const int64_t nb1 = std::min<int64_t>(d_in, nb0 + BLK);    // columns beyond it: [nb1, d_in)
            const bool fork = side && nb1 < d_in;
            if (fork) KQ_CUDA(cudaEventRecord(side->ev[0], stream));           // E of this block ready
            kq_status st;
            if (!fuse) {
                if (forked) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));  // previous far update done
                st = trailing(i0, kb, nb0, nb1, stream);
                if (st != KQ_OK) return st;
            }
            if (nb1 < d_in) {
                cudaStream_t fs = stream;
                if (fork) {
                    KQ_CUDA(cudaStreamWaitEvent(side->s, side->ev[0], 0));
                    fs = side->s;
                }
                st = trailing(i0, kb, nb1, d_in, fs);
                if (st != KQ_OK) return st;
                if (fork) {
                    KQ_CUDA(cudaEventRecord(fuse ? side->ev2[b & 1] : side->ev[1], side->s));
                    if (fuse)
                        far_pending[b & 1] = true;
                    else
                        forked = true;
                }
            }
        }
        for (int q = 0; q < 2; ++q)
            if (far_pending[q]) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[q], 0));
    }
    if (forked) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));
    if (col_loss) {
        colloss_kernel<<<static_cast<unsigned>(cdiv(d_in, CS_X)), dim3(CS_X, CS_Y), 0, stream>>>(o.E, d_out, d_in, col_loss);
        KQ_LAUNCH_CHECK("colloss_kernel");
    }
    return KQ_OK;
}
