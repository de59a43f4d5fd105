// Stage 3: damped inverse Cholesky.
//
// Paper: Algorithm 2 ("H_X <- H_X + lambda mean(diag(H_X)) I; L <- Inverse_Cholesky(H_X)")
// and Proposition 1 (H_X^-1 = L L^T, L lower). The OBS sweep (Eq. obs_update) uses row j of
// R = L^T.
//
// Route (2 n^3 / 3 flops instead of factor -> invert -> factor): with J the index
// reversal, the lower Cholesky factor C of A = J H J gives H = (J C J)(J C J)^T, J C J
// upper, hence H^-1 = (J C^-T J)(J C^-T J)^T and L = J C^-T J, i.e. L[i][j] = C^-1[n-1-j][n-1-i].
// One right-looking blocked sweep (block nb = 128) computes C and Z = C^-1 together:
//   step k: diag  -- factor A_kk = C_kk C_kk^T in registers and keep C_kk^-1 (1 CTA);
//           panel -- C_ik = A_ik C_kk^-T (i > k) and Z_kj = C_kk^-1 B_kj (j < k);
//           update-- A_ij -= C_ik C_jk^T (k < j <= i) and B_ij -= C_ik Z_kj (j <= k < i),
// where B (stored in Z's blocks) is the right-hand side I of C Z = I after the earlier
// steps' eliminations. The matrix is padded to a multiple of nb with an identity block.
// Look-ahead: the update is split into the tiles step k + 1 reads first (row and column
// block k + 1; the next diagonal tile alone on the caller's stream, the rest on a library
// side stream) and the rest of the step's tiles (side stream, beside step k + 1's diagonal
// factorization and panel). The diagonal kernel is fp32 SIMT with fused multiply-add; the
// panel and the tile updates multiply on the tensor cores (mma.sync tf32 with the 3xTF32
// split, operands split as they are loaded).
// Two levels when n > 8 NB: steps are grouped in super-panels S of 8 blocks (D: the rows
// below S, P: the columns left of it). The steps of S touch only S's diagonal block (A's
// lower tiles and B's tiles in rows and columns S), so they stay small kernels. S's panel
// below and its rows of Z to the left then follow from the inverse of its diagonal block,
// Z_SS = C_SS^-1, which those steps built: with A' and B' as the earlier super-panels left
// them, A'_DS = C_DS C_SS^T (the Schur complement's block) and C_SS Z_SP = B'_SP (forward
// substitution), so C_DS = A'_DS Z_SS^T and Z_SP = Z_SS B'_SP, two K = 8 NB products on the
// tensor cores (3xTF32, trail_tc.cu's two-CTA kernel, each tile's K bounded by the
// triangle of Z_SS). Every tile beyond S then takes the whole super-panel's update at once
// (K = 8 NB): the next super-panel's diagonal block first, on the caller's stream (the next
// steps read only it), every other tile on a second library stream beside the next
// super-panel's steps, leaving them a few SMs. The products and the update read tf32 hi / lo
// splits of their operands (split_block_kernel); the split sets alternate between
// super-panels, so a super-panel's splits do not overwrite the operands the previous
// super-panel's update reads. The trailing matrix is read and written once per super-panel
// rather than once per step (at n = 28672, ~90 GB of HBM traffic instead of ~700 GB).
#include <math.h>

#include <cstdlib>

#include "kq_common.cuh"
#include "tile_gemm.cuh"
#include "trail_tc.cuh"

namespace kq {
namespace {

constexpr int NB = 128;

constexpr int SPB = 8;                          // blocks per super-panel

struct Work {
    float* A;      // npad x npad, reversed damped H -> C (lower)
    float* Z;      // npad x npad, B -> C^-1 (lower)
    float* split[8];  // per set: Ch, Cl (split C panel), Zh, Zl (split Z rows, transposed)
    double* dsum;  // sum of diag(H)
};

inline size_t npad_of(int64_t n) { return static_cast<size_t>(cdiv(n, NB) * NB); }

// Split operand width and number of sets: two sets of a super-panel's width when the matrix
// takes more than one super-panel; none otherwise (the one-level schedule multiplies on the
// strip kernels, which split their operands as they load them).
constexpr size_t split_width(size_t) { return static_cast<size_t>(SPB) * NB; }
constexpr size_t split_sets(size_t np) { return np / NB > static_cast<size_t>(SPB) ? 2 : 0; }
constexpr size_t ws_bytes_for(size_t np) {
    return (2 * np * np + split_sets(np) * 4 * np * split_width(np)) * sizeof(float) + 256;
}

// --------------------------------------------------------------------- prep
__global__ void diag_sum_kernel(const float* __restrict__ H, int64_t n, double* out) {
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

// A[i][j] = H[n-1-i][n-1-j] + delta [i == j] inside n; identity in the padding; Z = 0.
__global__ void prep_kernel(const float* __restrict__ H, int64_t n, int64_t npad, float damp_rel,
                            const double* __restrict__ dsum, float* __restrict__ A,
                            float* __restrict__ Z) {
    const float delta = static_cast<float>(static_cast<double>(damp_rel) * (*dsum / static_cast<double>(n)));
    const int64_t total = npad * npad;
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t i = e / npad, j = e % npad;
        float v;
        if (i < n && j < n) {
            v = H[(n - 1 - i) * n + (n - 1 - j)];
            if (i == j) v += delta;
        } else {
            v = (i == j) ? 1.0f : 0.0f;
        }
        if (KQ_IN_RANGE(e, total)) {
            A[e] = v;
            Z[e] = 0.0f;
        }
    }
}

// The same with 16-byte accesses (n % 4 == 0, H 16-byte aligned): four columns per
// thread and step, H's row read as reversed float4 quads.
__global__ void prep4_kernel(const float* __restrict__ H, int64_t n, int64_t npad, float damp_rel,
                             const double* __restrict__ dsum, float* __restrict__ A, float* __restrict__ Z) {
    const float delta = static_cast<float>(static_cast<double>(damp_rel) * (*dsum / static_cast<double>(n)));
    const int64_t nq = npad / 4, total = npad * nq;
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t i = e / nq, j = 4 * (e - i * nq);
        float v[4];
        if (i < n && j < n) {   // the whole quad (n % 4 == 0): A[i][j + t] = H[n-1-i][n-1-j-t]
            const float4 h = *reinterpret_cast<const float4*>(H + (n - 1 - i) * n + (n - 4 - j));
            v[0] = h.w;
            v[1] = h.z;
            v[2] = h.y;
            v[3] = h.x;
#pragma unroll
            for (int t = 0; t < 4; ++t)
                if (i == j + t) v[t] += delta;
        } else {
#pragma unroll
            for (int t = 0; t < 4; ++t) v[t] = (i == j + t) ? 1.0f : 0.0f;
        }
        if (KQ_IN_RANGE(4 * e + 3, npad * npad)) {
            reinterpret_cast<float4*>(A)[e] = make_float4(v[0], v[1], v[2], v[3]);
            reinterpret_cast<float4*>(Z)[e] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        }
    }
}

// ---------------------------------------------------------------- diag block
// Factor A_kk = C C^T and invert C on one CTA, as an L D L^T sweep that builds L^-1 in
// place (Gauss-Jordan on the lower triangle), four columns per barrier.
//
// Scalar step j (the definition): with the "hook" h (row j left of the diagonal, column j
// below it, h_j = 0), pivot d_j and multipliers u_i = M_ij / d_j, every row i > j updates
//   M_ik -= u_i h_k      (k != j; k > j: Schur complement, k < j: rows of L^-1)
// and column j keeps its value, the unscaled column j of L D. So M ends up holding, below
// the diagonal, R = -L^-1 D (column-scaled), and C^-1 = D^-1/2 L^-1 has entries
// -R_ik / (d_k sqrt(d_i)). C = L D^1/2 itself is not stored: the panel and the updates read
// only C^-1 of the diagonal block.
//
// Four steps at once (block column q, rows j..j+3, j = 4q): with the 4 x 4 pivot block
// factored as L_b D_b L_b^T (raw columns g = L_b D_b, raw inverse rows b of the block),
// a panel row p below it gives w = L_b^-1 p (the raw hook values of the four steps) and
// u = w / d; a block-row column x (left of the block) gives h = L_b^-1 x; the four scalar
// updates of a below-block entry sum to M_ik -= sum_t u_i^t h_k^t with h = w for columns
// right of the block. Panel entries end as w_s - sum_{t>s} u^t b_ts, block-row entries as
// h, and the pivot block as b. The pivot block's owner factors it once and publishes the
// record; panel rows and block-row rows are published raw by their owners. One barrier
// per block column; the staging is double-buffered.
//
// Thread t < 528 owns one 4 x 4 block of the lower triangle (row-major block order) in
// registers. Pivots are checked by thread 0 (first non-positive one reported).
constexpr int DIAG_THREADS = 544;                            // 528 owners + 16 idle lanes
constexpr int DG_OWNERS = (NB / 4) * (NB / 4 + 1) / 2;       // 528
constexpr int DG_PIV = 32;                                   // floats per pivot record
constexpr size_t DIAG_SMEM =
    (2 * NB * 4 + 2 * 4 * NB + 2 * DG_PIV + NB) * sizeof(float);

struct Piv4 {   // factored 4 x 4 pivot block: 1 / d, unit-lower L_b, raw inverse rows b
    float rd[4], l10, l20, l30, l21, l31, l32, b10, b20, b30, b21, b31, b32;
};

__device__ __forceinline__ float rcp_approx(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// x <- L_b^-1 x
__device__ __forceinline__ void unit_lower_solve(float& x0, float& x1, float& x2, float& x3, const Piv4& p) {
    x1 = fmaf(-p.l10, x0, x1);
    x2 = fmaf(-p.l20, x0, x2);
    x3 = fmaf(-p.l30, x0, x3);
    x2 = fmaf(-p.l21, x1, x2);
    x3 = fmaf(-p.l31, x1, x3);
    x3 = fmaf(-p.l32, x2, x3);
}

// Publish the inputs of block step q (buffer q & 1): block-row rows (left of the pivot),
// panel rows (below it), and the factored pivot, whose owner also sets its block final.
__device__ __forceinline__ void diag_publish(int q, float (&m)[4][4], int bi, int bk, float* Pst, float* Qst,
                                             float* Pv) {
    const int buf = q & 1;
    const int i0 = 4 * bi, k0 = 4 * bk;
    if (bi == q && bk < q) {
#pragma unroll
        for (int r = 0; r < 4; ++r)
            *reinterpret_cast<float4*>(Qst + buf * 4 * NB + r * NB + k0) = make_float4(m[r][0], m[r][1], m[r][2], m[r][3]);
    }
    if (bk == q && bi > q) {
#pragma unroll
        for (int r = 0; r < 4; ++r)
            *reinterpret_cast<float4*>(Pst + buf * NB * 4 + (i0 + r) * 4) = make_float4(m[r][0], m[r][1], m[r][2], m[r][3]);
    }
    if (bi == q && bk == q) {
        float a11 = m[1][1], a21 = m[2][1], a31 = m[3][1], a22 = m[2][2], a32 = m[3][2], a33 = m[3][3];
        const float d0 = m[0][0], g10 = m[1][0], g20 = m[2][0], g30 = m[3][0];
        const float r0 = rcp_approx(d0);
        const float l10 = g10 * r0, l20 = g20 * r0, l30 = g30 * r0;
        a11 = fmaf(-l10, g10, a11);
        a21 = fmaf(-l20, g10, a21);
        a31 = fmaf(-l30, g10, a31);
        a22 = fmaf(-l20, g20, a22);
        a32 = fmaf(-l30, g20, a32);
        a33 = fmaf(-l30, g30, a33);
        const float d1 = a11, g21 = a21, g31 = a31;
        const float r1 = rcp_approx(d1);
        const float l21 = g21 * r1, l31 = g31 * r1;
        a22 = fmaf(-l21, g21, a22);
        a32 = fmaf(-l31, g21, a32);
        a33 = fmaf(-l31, g31, a33);
        const float d2 = a22, g32 = a32;
        const float r2 = rcp_approx(d2);
        const float l32 = g32 * r2;
        a33 = fmaf(-l32, g32, a33);
        const float d3 = a33;
        const float r3 = rcp_approx(d3);
        const float b10 = g10, b21 = g21, b32 = g32;
        const float b20 = fmaf(-l21, b10, g20);
        const float b31 = fmaf(-l32, b21, g31);
        const float b30 = fmaf(-l32, b20, fmaf(-l31, b10, g30));
        float* pv = Pv + buf * DG_PIV;
        *reinterpret_cast<float4*>(pv) = make_float4(r0, r1, r2, r3);
        *reinterpret_cast<float4*>(pv + 4) = make_float4(l10, l20, l30, l21);
        *reinterpret_cast<float4*>(pv + 8) = make_float4(l31, l32, b10, b20);
        *reinterpret_cast<float4*>(pv + 12) = make_float4(b30, b21, b31, b32);
        *reinterpret_cast<float4*>(pv + 16) = make_float4(d0, d1, d2, d3);
        m[1][0] = b10;
        m[2][0] = b20;
        m[3][0] = b30;
        m[2][1] = b21;
        m[3][1] = b31;
        m[3][2] = b32;
    }
}

__global__ void __launch_bounds__(DIAG_THREADS) chol_diag_kernel(Work w, int64_t n, int64_t npad, int k, int* info) {
    extern __shared__ __align__(16) float sm[];
    float* Pst = sm;                      // [2][NB][4]   panel rows
    float* Qst = Pst + 2 * NB * 4;        // [2][4][NB]   block-row rows
    float* Pv = Qst + 2 * 4 * NB;         // [2][DG_PIV]  pivot records
    float* dv = Pv + 2 * DG_PIV;          // [NB]         pivots d
    const int tid = threadIdx.x;
    const int64_t off = static_cast<int64_t>(k) * NB;
    const bool owner = tid < DG_OWNERS;
    int bi = 0, bk = 0;
    if (owner) {
        int rem = tid;
        while (rem > bi) {
            rem -= bi + 1;
            ++bi;
        }
        bk = rem;
    }
    const int i0 = 4 * bi, k0 = 4 * bk;
    float m[4][4];
    if (owner) {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const float4 v = *reinterpret_cast<const float4*>(w.A + (off + i0 + r) * npad + off + k0);
            m[r][0] = v.x;
            m[r][1] = v.y;
            m[r][2] = v.z;
            m[r][3] = v.w;
        }
        diag_publish(0, m, bi, bk, Pst, Qst, Pv);
    }
    __syncthreads();
#pragma unroll 1
    for (int q = 0; q < NB / 4; ++q) {
        const int buf = q & 1;
        const float* pv = Pv + buf * DG_PIV;
        if (tid == 0) {
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                const float d = pv[16 + t];
                dv[4 * q + t] = d;
                if (!(d > 0.0f)) {
                    const int64_t rev = off + 4 * q + t;
                    if (rev < n) record_error(info, static_cast<int>(n - rev));
                }
            }
        }
        if (owner && bi >= q && !(bi == q && bk >= q)) {
            Piv4 p;
            {
                const float4 v0 = *reinterpret_cast<const float4*>(pv);
                const float4 v1 = *reinterpret_cast<const float4*>(pv + 4);
                const float4 v2 = *reinterpret_cast<const float4*>(pv + 8);
                const float4 v3 = *reinterpret_cast<const float4*>(pv + 12);
                p.rd[0] = v0.x;
                p.rd[1] = v0.y;
                p.rd[2] = v0.z;
                p.rd[3] = v0.w;
                p.l10 = v1.x;
                p.l20 = v1.y;
                p.l30 = v1.z;
                p.l21 = v1.w;
                p.l31 = v2.x;
                p.l32 = v2.y;
                p.b10 = v2.z;
                p.b20 = v2.w;
                p.b30 = v3.x;
                p.b21 = v3.y;
                p.b31 = v3.z;
                p.b32 = v3.w;
            }
            if (bi == q) {
                // block row, left of the pivot: rows become L_b^-1 x (final)
#pragma unroll
                for (int c = 0; c < 4; ++c) unit_lower_solve(m[0][c], m[1][c], m[2][c], m[3][c], p);
            } else {
                // my rows below the pivot: w = L_b^-1 p, u = w / d
                float u[4][4], wv[4][4];
                const float* pr = Pst + buf * NB * 4 + i0 * 4;
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const float4 x = *reinterpret_cast<const float4*>(pr + 4 * r);
                    float x0 = x.x, x1 = x.y, x2 = x.z, x3 = x.w;
                    unit_lower_solve(x0, x1, x2, x3, p);
                    wv[r][0] = x0;
                    wv[r][1] = x1;
                    wv[r][2] = x2;
                    wv[r][3] = x3;
                    u[r][0] = x0 * p.rd[0];
                    u[r][1] = x1 * p.rd[1];
                    u[r][2] = x2 * p.rd[2];
                    u[r][3] = x3 * p.rd[3];
                }
                if (bk == q) {
                    // panel: final raw inverse columns
#pragma unroll
                    for (int r = 0; r < 4; ++r) {
                        m[r][0] = fmaf(-u[r][3], p.b30, fmaf(-u[r][2], p.b20, fmaf(-u[r][1], p.b10, wv[r][0])));
                        m[r][1] = fmaf(-u[r][3], p.b31, fmaf(-u[r][2], p.b21, wv[r][1]));
                        m[r][2] = fmaf(-u[r][3], p.b32, wv[r][2]);
                        m[r][3] = wv[r][3];
                    }
                } else {
                    // h = L_b^-1 x, x from the block row (left columns) or the panel (right)
                    float h[4][4];   // h[t][c]
                    if (bk < q) {
                        const float* qr = Qst + buf * 4 * NB + k0;
#pragma unroll
                        for (int t = 0; t < 4; ++t) {
                            const float4 x = *reinterpret_cast<const float4*>(qr + t * NB);
                            h[t][0] = x.x;
                            h[t][1] = x.y;
                            h[t][2] = x.z;
                            h[t][3] = x.w;
                        }
                    } else {
                        const float* pc = Pst + buf * NB * 4 + k0 * 4;
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            const float4 x = *reinterpret_cast<const float4*>(pc + 4 * c);
                            h[0][c] = x.x;
                            h[1][c] = x.y;
                            h[2][c] = x.z;
                            h[3][c] = x.w;
                        }
                    }
#pragma unroll
                    for (int c = 0; c < 4; ++c) unit_lower_solve(h[0][c], h[1][c], h[2][c], h[3][c], p);
#pragma unroll
                    for (int t = 0; t < 4; ++t)
#pragma unroll
                        for (int r = 0; r < 4; ++r)
#pragma unroll
                            for (int c = 0; c < 4; ++c) m[r][c] = fmaf(-u[r][t], h[t][c], m[r][c]);
                }
            }
        }
        if (owner && q + 1 < NB / 4) diag_publish(q + 1, m, bi, bk, Pst, Qst, Pv);
        __syncthreads();
    }
    // Scales (the staging is free now): 1 / sqrt(d), 1 / d.
    float* isq = Pst;
    float* idv = Qst;
    if (tid < NB) {
        const float d = dv[tid];
        isq[tid] = __frcp_rn(sqrtf(d));
        idv[tid] = __frcp_rn(d);
    }
    __syncthreads();
    // C^-1 = D^-1/2 L^-1 with L^-1_ik = -R_ik / d_k (k < i); the upper blocks of Z stay 0.
    // C_kk itself is not stored: later steps read only C^-1_kk and the blocks below it.
    if (owner) {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int i = i0 + r;
            const float si = isq[i];
            float o[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int kk = k0 + c;
                o[c] = kk < i ? -m[r][c] * idv[kk] * si : (kk == i ? si : 0.0f);
            }
            if (KQ_IN_RANGE((off + i) * npad + off + k0 + 3, npad * npad))
                *reinterpret_cast<float4*>(w.Z + (off + i) * npad + off + k0) = make_float4(o[0], o[1], o[2], o[3]);
        }
    }
}

// ---------------------------------------------------------- strips of one tile
// The panel and the first tiles of the next step are on the critical path and come in
// ~nbk tiles, so each 128 x 128 tile is split over 4 CTAs (strips or quadrants) with the
// whole K = 128 staged in shared memory at once (two cp.async groups of 64).
constexpr int SK = NB;
constexpr int SLD = SK + 4;   // row stride of K-contiguous slabs (conflict-free float4 rows)

template <int BM, int BNc, bool BNL>
struct Strip {
    static constexpr int RM = BM / 16, CN = BNc / 16;
    static constexpr int A_FLOATS = BM * SLD;
    static constexpr int B_FLOATS = BNL ? SK * (BNc + 4) : BNc * SLD;
    static constexpr size_t SMEM = static_cast<size_t>(A_FLOATS + B_FLOATS) * sizeof(float);
};
constexpr size_t smax(size_t a, size_t b) { return a > b ? a : b; }
constexpr size_t STRIP_SMEM = smax(smax(Strip<128, 32, true>::SMEM, Strip<32, 128, false>::SMEM),
                                   smax(Strip<64, 64, true>::SMEM, Strip<64, 64, false>::SMEM));

// acc[i][j] = sum over k < 128 of A[ty + 16 i][k] * B(k, col_j), 256 threads (ty, tx) =
// (tid / 16, tid % 16). A is K-contiguous (row r at A + r ld). BNL = false: B(k, c) at
// B + c ld + k, col_j = tx + 16 j; BNL = true: B(k, c) at B + k ld + c, col_j = CN tx + j.
// All global reads finish before the function returns (the output may alias an input
// row or column strip of this CTA).
// The products run on the tensor cores: mma.sync m16n8k8 in tf32 with the 3xTF32 split
// (A_lo B_hi + A_hi B_lo + A_hi B_hi, fp32 accumulation), each of the 8 warps owning a
// 16 x 32 block of the BM x BNc output (BM BNc = 8 x 512 for the three strip shapes); the
// fragments are read from the padded shared-memory operands (row stride SLD = 132: the 32
// lanes of a fragment load hit 32 banks), and the results go back through shared memory
// into the layout above.
template <int BM, int BNc, bool BNL>
__device__ __forceinline__ void strip_gemm(const float* __restrict__ A, const float* __restrict__ B, int64_t ld,
                                           float (&acc)[BM / 16][BNc / 16], float* sm) {
    using S = Strip<BM, BNc, BNL>;
    constexpr int RM = S::RM, CN = S::CN, BLD = BNc + 4;
    float* As = sm;
    float* Bs = sm + S::A_FLOATS;
    const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int kh = h * (SK / 2);
        for (int q = tid; q < BM * (SK / 8); q += G_THREADS) {
            const int r = q / (SK / 8), k4 = q % (SK / 8);
            cp_async16(As + r * SLD + kh + 4 * k4, A + r * ld + kh + 4 * k4, 16);
        }
        if (BNL) {
            for (int q = tid; q < (SK / 2) * (BNc / 4); q += G_THREADS) {
                const int kk = q / (BNc / 4), c4 = q % (BNc / 4);
                cp_async16(Bs + (kh + kk) * BLD + 4 * c4, B + (kh + kk) * ld + 4 * c4, 16);
            }
        } else {
            for (int q = tid; q < BNc * (SK / 8); q += G_THREADS) {
                const int c = q / (SK / 8), k4 = q % (SK / 8);
                cp_async16(Bs + c * SLD + kh + 4 * k4, B + c * ld + kh + 4 * k4, 16);
            }
        }
        cp_async_commit();
    }
    const int lane = tid & 31, wid = tid >> 5, g = lane >> 2, t4 = lane & 3;
    constexpr int WC = BNc / 32;                 // warp columns of 32
    static_assert((BM / 16) * WC == G_THREADS / 32, "8 warps of 16 x 32");
    const int wr = wid / WC, wc = wid % WC;
    float c[4][4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) c[nt][e] = 0.0f;
    const float* arow0 = As + (16 * wr + g) * SLD;
    const float* arow1 = arow0 + 8 * SLD;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        if (h == 0)
            cp_async_wait<1>();
        else
            cp_async_wait<0>();
        __syncthreads();
#pragma unroll 2
        for (int ks = h * (SK / 2); ks < (h + 1) * (SK / 2); ks += 8) {
            const float a[4] = {arow0[ks + t4], arow1[ks + t4], arow0[ks + t4 + 4], arow1[ks + t4 + 4]};
            uint32_t ah[4], al[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float hi = tf32_hi(a[e]);
                ah[e] = __float_as_uint(hi);
                al[e] = __float_as_uint(a[e] - hi);
            }
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
                const int n = 32 * wc + 8 * nt + g;
                const float b0 = BNL ? Bs[(ks + t4) * BLD + n] : Bs[n * SLD + ks + t4];
                const float b1 = BNL ? Bs[(ks + t4 + 4) * BLD + n] : Bs[n * SLD + ks + t4 + 4];
                const float bh0 = tf32_hi(b0), bh1 = tf32_hi(b1);
                const uint32_t bh[2] = {__float_as_uint(bh0), __float_as_uint(bh1)};
                const uint32_t bl[2] = {__float_as_uint(b0 - bh0), __float_as_uint(b1 - bh1)};
                mma_tf32(c[nt], al, bh);
                mma_tf32(c[nt], ah, bl);
                mma_tf32(c[nt], ah, bh);
            }
        }
    }
    __syncthreads();   // every warp is done with As and Bs
    constexpr int CLD = BNc + 4;
    float* Cs = sm;    // [BM][CLD], within As and Bs
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
        const int r = 16 * wr + g, col = 32 * wc + 8 * nt + 2 * t4;
        Cs[r * CLD + col] = c[nt][0];
        Cs[r * CLD + col + 1] = c[nt][1];
        Cs[(r + 8) * CLD + col] = c[nt][2];
        Cs[(r + 8) * CLD + col + 1] = c[nt][3];
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < RM; ++i)
#pragma unroll
        for (int j = 0; j < CN; ++j) acc[i][j] = Cs[(ty + 16 * i) * CLD + (BNL ? CN * tx + j : tx + 16 * j)];
}

__global__ void __launch_bounds__(G_THREADS, 2) chol_panel_kernel(Work w, int64_t npad, int k, int b0) {
    extern __shared__ __align__(16) float sm[];
    const int b = static_cast<int>(blockIdx.x) + b0, s = blockIdx.y;
    const int64_t off = static_cast<int64_t>(k) * NB;
    const float* cinv = w.Z + off * npad + off;
    const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
    if (b < k) {
        float* out = w.Z + off * npad + static_cast<int64_t>(b) * NB + 32 * s;
        float acc[8][2];
        strip_gemm<128, 32, true>(cinv, out, npad, acc, sm);
#pragma unroll
        for (int i = 0; i < 8; ++i)
            if (KQ_IN_RANGE((out - w.Z) + (ty + 16 * i) * npad + 2 * tx + 1, npad * npad))
                *reinterpret_cast<float2*>(out + (ty + 16 * i) * npad + 2 * tx) = make_float2(acc[i][0], acc[i][1]);
    } else {
        float* out = w.A + (static_cast<int64_t>(b + 1) * NB + 32 * s) * npad + off;
        float acc[2][8];
        strip_gemm<32, 128, false>(out, cinv, npad, acc, sm);
#pragma unroll
        for (int i = 0; i < 2; ++i)
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (KQ_IN_RANGE((out - w.A) + (ty + 16 * i) * npad + tx + 16 * j, npad * npad))
                    out[(ty + 16 * i) * npad + tx + 16 * j] = acc[i][j];
    }
}

// Quadrant q (rows 64 (q / 2), columns 64 (q % 2)) of update tile (i, j) of step k.
__device__ __forceinline__ void update_quad(const Work& w, int64_t npad, int k, int i, int j, int q, float* sm) {
    const int64_t ko = static_cast<int64_t>(k) * NB;
    const int64_t r0 = static_cast<int64_t>(i) * NB + 64 * (q >> 1);
    const int64_t c0 = static_cast<int64_t>(j) * NB + 64 * (q & 1);
    const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
    const float* cik = w.A + r0 * npad + ko;
    float acc[4][4];
    if (j > k) {
        strip_gemm<64, 64, false>(cik, w.A + c0 * npad + ko, npad, acc, sm);
        float* out = w.A + r0 * npad + c0;
        float o[4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c = 0; c < 4; ++c) o[a][c] = out[(ty + 16 * a) * npad + tx + 16 * c];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (KQ_IN_RANGE((out - w.A) + (ty + 16 * a) * npad + tx + 16 * c, npad * npad))
                    out[(ty + 16 * a) * npad + tx + 16 * c] = o[a][c] - acc[a][c];
    } else {
        strip_gemm<64, 64, true>(cik, w.Z + ko * npad + c0, npad, acc, sm);
        float* out = w.Z + r0 * npad + c0;
        float4 o[4];
#pragma unroll
        for (int a = 0; a < 4; ++a) o[a] = *reinterpret_cast<const float4*>(out + (ty + 16 * a) * npad + 4 * tx);
#pragma unroll
        for (int a = 0; a < 4; ++a)
            if (KQ_IN_RANGE((out - w.Z) + (ty + 16 * a) * npad + 4 * tx + 3, npad * npad))
                *reinterpret_cast<float4*>(out + (ty + 16 * a) * npad + 4 * tx) =
                    make_float4(o[a].x - acc[a][0], o[a].y - acc[a][1], o[a].z - acc[a][2], o[a].w - acc[a][3]);
    }
}

// The tiles that step k + 1 reads first: row block k + 1 (tiles (k + 1, j), b0 <= j <= k + 1)
// and block column k + 1 below it (tiles (i, k + 1), k + 1 < i < b0 + gridDim.x); one tile
// x 4 quadrants per block index from b0. part 0: all of them; part 1: only the diagonal
// tile (k + 1, k + 1), which is all the next diagonal step needs (grid 1 x 4); part 2: all
// but that tile, for the next panel.
__global__ void __launch_bounds__(G_THREADS, 2) chol_next_kernel(Work w, int64_t npad, int k, int part, int b0) {
    extern __shared__ __align__(16) float sm[];
    const int bid = part == 1 ? k + 1 : static_cast<int>(blockIdx.x) + b0;
    if (part == 2 && bid == k + 1) return;
    if (bid < k + 2)
        update_quad(w, npad, k, k + 1, bid, blockIdx.y, sm);
    else
        update_quad(w, npad, k, bid, k + 1, blockIdx.y, sm);
}

// The rest of step k's update inside the blocks [k0, k1): the lower tiles (i, j) of A with
// k + 2 <= j <= i < k1, then the tiles (i, j) of B with k + 2 <= i < k1, k0 <= j <= k;
// one tile x 4 quadrants per block index.
__global__ void __launch_bounds__(G_THREADS, 2) chol_rest_kernel(Work w, int64_t npad, int k, int k0, int k1) {
    extern __shared__ __align__(16) float sm[];
    const int m = k1 - k - 2;
    int t = static_cast<int>(blockIdx.x), i, j;
    if (t < m * (m + 1) / 2) {
        j = k + 2;
        while (t >= k1 - j) {
            t -= k1 - j;
            ++j;
        }
        i = j + t;
    } else {
        t -= m * (m + 1) / 2;
        const int nzc = k - k0 + 1;
        i = k + 2 + t / nzc;
        j = k0 + t % nzc;
    }
    update_quad(w, npad, k, i, j, blockIdx.y, sm);
}

// hi / lo = tf32 split of sign * src over a [rows x cols] block of a row-major matrix
// (leading dimension lds; rows and cols multiples of 64), written as [rows x cols] (trans = 0)
// or transposed, [cols x rows] (trans = 1), with leading dimension ldd; zero_src: the block
// of src is set to 0 after it is read. src_n / dst_n: elements addressable from src / hi.
// Block (32, 8) walking 64 x 64 tiles (persistent grid): each thread has its 16 loads of a
// tile in flight before the stores; the transposed tile goes through shared memory.
constexpr int SPLIT_T = 64;
__global__ void __launch_bounds__(256) split_block_kernel(float* __restrict__ src, int64_t lds, int64_t rows,
                                                          int64_t cols, float* __restrict__ hi,
                                                          float* __restrict__ lo, int64_t ldd, int trans, float sign,
                                                          int zero_src, int64_t src_n, int64_t dst_n) {
    __shared__ float t[SPLIT_T][SPLIT_T + 1];
    const int64_t nct = cols / SPLIT_T, ntiles = (rows / SPLIT_T) * nct;
    const int tx = threadIdx.x, ty = threadIdx.y;
    for (int64_t b = blockIdx.x; b < ntiles; b += gridDim.x) {
        const int64_t r0 = (b / nct) * SPLIT_T, c0 = (b % nct) * SPLIT_T;
        float v[8][2];
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int64_t si = (r0 + ty + 8 * i) * lds + c0 + 32 * h + tx;
                v[i][h] = KQ_IN_RANGE(si, src_n) ? src[si] : 0.0f;
            }
        if (zero_src) {
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int64_t si = (r0 + ty + 8 * i) * lds + c0 + 32 * h + tx;
                    if (KQ_IN_RANGE(si, src_n)) src[si] = 0.0f;
                }
        }
        if (!trans) {
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int64_t di = (r0 + ty + 8 * i) * ldd + c0 + 32 * h + tx;
                    if (!KQ_IN_RANGE(di, dst_n)) continue;
                    const float x = sign * v[i][h];
                    const float hv = tf32_hi(x);
                    hi[di] = hv;
                    lo[di] = x - hv;
                }
            continue;
        }
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int h = 0; h < 2; ++h) t[ty + 8 * i][32 * h + tx] = v[i][h];
        __syncthreads();
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int c = ty + 8 * i, r = 32 * h + tx;   // src[r0 + r][c0 + c]
                const int64_t di = (c0 + c) * ldd + r0 + r;
                if (!KQ_IN_RANGE(di, dst_n)) continue;
                const float x = sign * t[r][c];
                const float hv = tf32_hi(x);
                hi[di] = hv;
                lo[di] = x - hv;
            }
        __syncthreads();
    }
}

kq_status split_block(float* src, int64_t lds, int64_t rows, int64_t cols, float* hi, float* lo, int64_t ldd,
                      int trans, float sign, int zero_src, int64_t src_n, int64_t dst_n, cudaStream_t stream) {
    if (rows <= 0 || cols <= 0) return KQ_OK;
    if (rows % SPLIT_T || cols % SPLIT_T) {
        set_error("kq_chol_inv: split block %lld x %lld is not whole %d x %d tiles", (long long)rows,
                  (long long)cols, SPLIT_T, SPLIT_T);
        return KQ_ERR_INVALID_ARG;
    }
    const int64_t tiles = (rows / SPLIT_T) * (cols / SPLIT_T);
    const int64_t grid = std::min<int64_t>(tiles, static_cast<int64_t>(num_sms()) * 8);
    split_block_kernel<<<static_cast<unsigned>(grid), dim3(32, 8), 0, stream>>>(src, lds, rows, cols, hi, lo, ldd,
                                                                                trans, sign, zero_src, src_n, dst_n);
    KQ_LAUNCH_CHECK("split_block_kernel");
    return KQ_OK;
}

// SMs left to the next super-panel's steps while the update of the tiles beyond the
// next super-panel runs beside them (its grid is that many SMs short of all resident
// clusters): KQ_CHOL_FREE_SMS, an even number below the SM count, else FAR_FREE_SMS.
constexpr int FAR_FREE_SMS = 16;
int far_free_sms() {
    static const int v = [] {
        const char* e = std::getenv("KQ_CHOL_FREE_SMS");
        const int x = e ? std::atoi(e) : FAR_FREE_SMS;
        return (x >= 0 && x % 2 == 0 && x < num_sms()) ? x : FAR_FREE_SMS;
    }();
    return v;
}

// -------------------------------------------------------------------- finish
// Lt[i][j] = Z[n-1-j][n-1-i] for j <= i < n, 0 above the diagonal (32 x 32 smem transpose).
__global__ void finish_kernel(const float* __restrict__ Z, int64_t n, int64_t npad, float* __restrict__ Lt) {
    __shared__ float t[32][33];
    const int64_t i0 = static_cast<int64_t>(blockIdx.y) * 32, j0 = static_cast<int64_t>(blockIdx.x) * 32;
    // Source block: rows a = n-1-j (j in [j0, j0+32)), cols b = n-1-i.
    for (int r = threadIdx.y; r < 32; r += blockDim.y) {
        const int64_t j = j0 + r;
        const int64_t i = i0 + threadIdx.x;
        float v = 0.0f;
        if (i < n && j < n && j <= i) v = Z[(n - 1 - j) * npad + (n - 1 - i)];
        t[r][threadIdx.x] = v;
    }
    __syncthreads();
    for (int r = threadIdx.y; r < 32; r += blockDim.y) {
        const int64_t i = i0 + r, j = j0 + threadIdx.x;
        if (i < n && j < n && KQ_IN_RANGE(i * n + j, n * n)) Lt[i * n + j] = t[threadIdx.x][r];
    }
}

// The same with 64 x 64 tiles and 16-byte accesses (n % 4 == 0, Lt 16-byte aligned): the
// tile of Lt at (i0, j0) reads rows a = n-1-j of Z over columns n-1-i, a quad at a time
// (reversed into shared memory), and writes quads of Lt's rows; tiles wholly above the
// diagonal only write zeros.
__global__ void __launch_bounds__(256) finish4_kernel(const float* __restrict__ Z, int64_t n, int64_t npad,
                                                      float* __restrict__ Lt) {
    __shared__ float t[64][65];   // t[jj][ii] = Lt[i0 + ii][j0 + jj]
    const int64_t i0 = static_cast<int64_t>(blockIdx.y) * 64, j0 = static_cast<int64_t>(blockIdx.x) * 64;
    const int q = threadIdx.x & 15, r0 = threadIdx.x >> 4;   // 16 quads x 16 rows per pass
    const bool above = j0 > i0 + 63;
    if (!above) {
        for (int jj = r0; jj < 64; jj += 16) {
            const int64_t j = j0 + jj;
            // Z row n-1-j, columns n-64-i0 + 4q .. +3, i.e. ii = 63-4q-u for u = 0..3
            const int64_t c = n - 64 - i0 + 4 * q;
            float4 z = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (j < n && c >= 0) z = *reinterpret_cast<const float4*>(Z + (n - 1 - j) * npad + c);
            const float zv[4] = {z.x, z.y, z.z, z.w};
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int ii = 63 - 4 * q - u;
                const int64_t i = i0 + ii;
                t[jj][ii] = (j < n && i < n && j <= i) ? zv[u] : 0.0f;
            }
        }
    }
    __syncthreads();
    for (int ii = r0; ii < 64; ii += 16) {
        const int64_t i = i0 + ii, j = j0 + 4 * q;
        if (i >= n || j >= n) continue;   // whole quads (n % 4 == 0)
        float4 v = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        if (!above) v = make_float4(t[4 * q][ii], t[4 * q + 1][ii], t[4 * q + 2][ii], t[4 * q + 3][ii]);
        if (KQ_IN_RANGE(i * n + j + 3, n * n)) *reinterpret_cast<float4*>(Lt + i * n + j) = v;
    }
}

}  // namespace

KQ_DEBUG_UNIT(chol)
}  // namespace kq

using namespace kq;

extern "C" size_t kq_chol_inv_workspace(int64_t n) {
    if (n < 1) return 0;
    return ws_bytes_for(npad_of(n));
}

extern "C" kq_status kq_chol_inv(const float* H, int64_t n, float damp_rel, float* Lt, int* info, void* ws,
                                 size_t ws_bytes, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!H || !Lt || n < 1 || n > 65536 || !(damp_rel >= 0.0f)) {
        set_error("kq_chol_inv: invalid arguments (n=%lld)", (long long)n);
        return KQ_ERR_INVALID_ARG;
    }
    if (!ws || ws_bytes < kq_chol_inv_workspace(n) || (reinterpret_cast<uintptr_t>(ws) & 15u)) {
        set_error("kq_chol_inv: workspace must be 16-byte aligned and hold %zu bytes",
                  kq_chol_inv_workspace(n));
        return KQ_ERR_WORKSPACE;
    }
    const int64_t npad = static_cast<int64_t>(npad_of(n));
    const int nbk = static_cast<int>(npad / NB);
    const int width = static_cast<int>(split_width(static_cast<size_t>(npad)));
    const int nsets = static_cast<int>(split_sets(static_cast<size_t>(npad)));
    const bool two_level = nbk > SPB;
    Work w;
    w.A = static_cast<float*>(ws);
    w.Z = w.A + npad * npad;
    float* sp = w.Z + npad * npad;
    for (int q = 0; q < 4 * nsets; ++q, sp += npad * width) w.split[q] = sp;
    w.dsum = reinterpret_cast<double*>(sp);
    CholTcMaps maps;
    if (two_level) {
        kq_status st = maps.init(w.A, w.Z, npad, width, nsets, w.split);
        if (st != KQ_OK) return st;
    }
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(chol_diag_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(DIAG_SMEM)));
        KQ_CUDA(cudaFuncSetAttribute(chol_panel_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(STRIP_SMEM)));
        KQ_CUDA(cudaFuncSetAttribute(chol_next_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(STRIP_SMEM)));
        KQ_CUDA(cudaFuncSetAttribute(chol_rest_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(STRIP_SMEM)));
        return KQ_OK;
    }));
    diag_sum_kernel<<<1, 1024, 0, stream>>>(H, n, w.dsum);
    KQ_LAUNCH_CHECK("diag_sum_kernel");
    const int64_t total = npad * npad;
    if (n % 4 == 0 && (reinterpret_cast<uintptr_t>(H) & 15u) == 0) {
        const int64_t g4 = std::min<int64_t>(cdiv(total / 4, 256), static_cast<int64_t>(num_sms()) * 32);
        prep4_kernel<<<static_cast<unsigned>(g4), 256, 0, stream>>>(H, n, npad, damp_rel, w.dsum, w.A, w.Z);
        KQ_LAUNCH_CHECK("prep4_kernel");
    } else {
        const int64_t pgrid = std::min<int64_t>(cdiv(total, 256), static_cast<int64_t>(num_sms()) * 32);
        prep_kernel<<<static_cast<unsigned>(pgrid), 256, 0, stream>>>(H, n, npad, damp_rel, w.dsum, w.A, w.Z);
        KQ_LAUNCH_CHECK("prep_kernel");
    }
    SideStream* side = nbk > 2 ? side_stream(stream) : nullptr;
    bool forked = false, remote_pending = false;
    bool next_pending = false;   // the next panel's tiles, updated on the side stream
    const int free_sms = far_free_sms();
    for (int k0 = 0; k0 < nbk; k0 += (two_level ? SPB : nbk)) {
        const int k1 = two_level ? std::min(nbk, k0 + SPB) : nbk;   // this super-panel: blocks [k0, k1)
        const int set = two_level ? (k0 / SPB) & 1 : 0;
        const bool far_after = two_level && k1 < nbk;
        // The steps of the super-panel inside its own blocks: A's lower tiles in rows and
        // columns [k0, k1) and B's tiles in rows and columns [k0, k1).
        for (int k = k0; k < k1; ++k) {
            chol_diag_kernel<<<1, DIAG_THREADS, DIAG_SMEM, stream>>>(w, n, npad, k, info);
            KQ_LAUNCH_CHECK("chol_diag_kernel");
            if (next_pending) {   // the tiles of this panel, updated beside the diagonal step
                KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[2], 0));
                next_pending = false;
            }
            if (k1 - 1 - k0 > 0) {
                chol_panel_kernel<<<dim3(k1 - 1 - k0, 4), G_THREADS, STRIP_SMEM, stream>>>(w, npad, k, k0);
                KQ_LAUNCH_CHECK("chol_panel_kernel");
            }
            if (k + 1 >= k1) break;
            const bool has_rest = k + 2 < k1;   // tiles of this super-panel beyond k + 1
            if (side) KQ_CUDA(cudaEventRecord(side->ev[0], stream));       // panel k done
            if (forked) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));   // rest of step k - 1 done
            if (side) {
                // Step k's update of the next diagonal tile alone on this stream, so the next
                // diagonal step starts at once; the other tiles the next panel reads, then the
                // rest of the step's update (other tiles), on the side stream beside it.
                KQ_CUDA(cudaStreamWaitEvent(side->s, side->ev[0], 0));
                chol_next_kernel<<<dim3(k1 - k0, 4), G_THREADS, STRIP_SMEM, side->s>>>(w, npad, k, 2, k0);
                KQ_LAUNCH_CHECK("chol_next_kernel");
                KQ_CUDA(cudaEventRecord(side->ev2[2], side->s));
                next_pending = true;
                chol_next_kernel<<<dim3(1, 4), G_THREADS, STRIP_SMEM, stream>>>(w, npad, k, 1, k0);
            } else {
                chol_next_kernel<<<dim3(k1 - k0, 4), G_THREADS, STRIP_SMEM, stream>>>(w, npad, k, 0, k0);
            }
            KQ_LAUNCH_CHECK("chol_next_kernel");
            if (has_rest) {
                const int m = k1 - k - 2;
                const unsigned tiles = static_cast<unsigned>(m * (m + 1) / 2 + m * (k - k0 + 1));
                chol_rest_kernel<<<dim3(tiles, 4), G_THREADS, STRIP_SMEM, side ? side->s : stream>>>(w, npad, k, k0, k1);
                KQ_LAUNCH_CHECK("chol_rest_kernel");
                if (side) {
                    KQ_CUDA(cudaEventRecord(side->ev[1], side->s));
                    forked = true;
                }
            }
        }
        if (!two_level) continue;
        if (forked) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));
        if (next_pending) {
            KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[2], 0));
            next_pending = false;
        }
        // the previous super-panel's update of the tiles beyond its successor's diagonal block
        if (remote_pending) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[1], 0));
        // The super-panel's blocks of C below it and of Z left of it, from its diagonal block
        // of Z (= C_SS^-1, lower triangular), as two products on the tensor cores:
        //   C_DS = A'_DS C_SS^-T = A'_DS Z_SS^T,   Z_SP = C_SS^-1 B'_SP = Z_SS B'_SP,
        // A' and B' as the earlier super-panels' updates left them (D: the rows below the
        // super-panel, P: the columns left of it). Operands in split set `set`: -A'_DS in the
        // C slices' rows of D, Z_SS in the Z slices' rows of S, -B'_SP transposed in the Z
        // slices' rows of P; the output blocks are cleared as their operands are read.
        // C_DS and the next diagonal block's update are on the caller's stream (the next
        // super-panel's steps wait for them); Z_SP, the Z operands of the update of the tiles
        // beyond and that update on the second library stream, beside the next steps.
        const int64_t sw = static_cast<int64_t>(k1 - k0) * NB;
        const int64_t s0 = static_cast<int64_t>(k0) * NB, s1 = static_cast<int64_t>(k1) * NB;
        float* const* sp4 = w.split + 4 * set;
        const int64_t nsplit = npad * width;
        float* a_ds = w.A + s1 * npad + s0;
        float* z_sp = w.Z + s0 * npad;
        cudaStream_t rs = side ? side->s2 : stream;
        KQ_TRY(split_block(z_sp + s0, npad, sw, sw, sp4[2] + s0 * width, sp4[3] + s0 * width, width, 0, 1.0f, 0,
                           npad * npad - (s0 * npad + s0), nsplit - s0 * width, stream));
        if (side) {
            KQ_CUDA(cudaEventRecord(side->ev2[0], stream));   // Z_SS split; the earlier updates done
            KQ_CUDA(cudaStreamWaitEvent(side->s2, side->ev2[0], 0));
        }
        KQ_TRY(split_block(z_sp, npad, sw, s0, sp4[2], sp4[3], width, 1, -1.0f, 1, npad * npad - s0 * npad, nsplit,
                           rs));
        KQ_TRY(chol_gemm_tc(z_sp, npad, sw, s0, sp4[2] + s0 * width, sp4[3] + s0 * width, sp4[2], sp4[3], width,
                            static_cast<int>(sw), 2, info, rs));
        if (far_after) {
            KQ_TRY(split_block(a_ds, npad, npad - s1, sw, sp4[0] + s1 * width, sp4[1] + s1 * width, width, 0, -1.0f,
                               1, npad * npad - (s1 * npad + s0), nsplit - s1 * width, stream));
            KQ_TRY(chol_gemm_tc(a_ds, npad, npad - s1, sw, sp4[0] + s1 * width, sp4[1] + s1 * width,
                                sp4[2] + s0 * width, sp4[3] + s0 * width, width, static_cast<int>(sw), 1, info,
                                stream));
            // operands of the update of every tile beyond the super-panel (K = its width):
            // C_DS in the C slices' rows of D ...
            KQ_TRY(split_block(a_ds, npad, npad - s1, sw, sp4[0] + s1 * width, sp4[1] + s1 * width, width, 0, 1.0f,
                               0, npad * npad - (s1 * npad + s0), nsplit - s1 * width, stream));
            if (side) {
                KQ_CUDA(cudaEventRecord(side->ev2[3], stream));   // C_DS split; Z_SS no longer read here
                KQ_CUDA(cudaStreamWaitEvent(side->s2, side->ev2[3], 0));
            }
            // ... and Z_S. (the columns left of the super-panel's end) transposed in the Z
            // slices' rows, over Z_SS's split once both products have read it
            KQ_TRY(split_block(z_sp, npad, sw, s1, sp4[2], sp4[3], width, 1, 1.0f, 0, npad * npad - s0 * npad, nsplit,
                               rs));
            // The update of the tiles beyond: the next super-panel's diagonal block on the
            // caller's stream (all the next super-panel's steps read it), every other tile --
            // A's block columns from k1 below row block k2, A beyond, Z's rows from k1 left of
            // column block k1 -- on the second library stream on all SMs but free_sms.
            const int k2 = std::min(nbk, k1 + SPB);
            const int nslab = (k1 - k0) * NB / 32;
            KQ_TRY(chol_update_tc(maps, set, nbk, k1, k2, 0, 0, 0, 0, nslab, info, stream, 0, 0, k2));
            KQ_TRY(chol_update_tc(maps, set, nbk, k1, nbk, k1, nbk, k1, 0, nslab, info, rs, side ? free_sms : 0, k2,
                                  nbk));
        }
        if (side) {
            KQ_CUDA(cudaEventRecord(side->ev2[1], side->s2));
            remote_pending = true;
        }
    }
    if (forked) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));
    if (next_pending) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[2], 0));
    if (remote_pending) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev2[1], 0));
    if (n % 4 == 0 && (reinterpret_cast<uintptr_t>(Lt) & 15u) == 0) {
        finish4_kernel<<<dim3(static_cast<unsigned>(cdiv(n, 64)), static_cast<unsigned>(cdiv(n, 64))), 256, 0,
                         stream>>>(w.Z, n, npad, Lt);
        KQ_LAUNCH_CHECK("finish4_kernel");
    } else {
        finish_kernel<<<dim3(static_cast<unsigned>(cdiv(n, 32)), static_cast<unsigned>(cdiv(n, 32))),
                        dim3(32, 8), 0, stream>>>(w.Z, n, npad, Lt);
        KQ_LAUNCH_CHECK("finish_kernel");
    }
    return KQ_OK;
}

// ------------------------------------------------------------ no-allocation variant
// kq_chol_inv_noalloc runs the same kernels as kq_chol_inv, with the scratch space taken
// from a fixed array in device memory that the library owns, so the caller passes only
// inputs and outputs. The array is sized for n <= KQ_CHOL_NOALLOC_MAX_N and is held by
// every device that loads the library until the process exits. Its device address is
// looked up once per device (with that device current) on the first call there.
#include <mutex>

namespace {
constexpr size_t kNoallocBytes = kq::ws_bytes_for(KQ_CHOL_NOALLOC_MAX_N);
static __device__ __align__(256) unsigned char g_chol_scratch[kNoallocBytes];
static_assert(kNoallocBytes == KQ_CHOL_NOALLOC_SCRATCH_BYTES,
              "the documented size of the allocation-free scratch array must match the one it has");
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[64] = {};
}  // namespace

extern "C" kq_status kq_chol_inv_noalloc(const float* H, int64_t n, float damp_rel, float* Lt, int* info,
                                         kq_stream_t stream) {
    if (n < 1 || n > KQ_CHOL_NOALLOC_MAX_N) {
        set_error("kq_chol_inv_noalloc: n=%lld is outside [1, %d], the size its fixed scratch array holds; "
                  "use kq_chol_inv with a caller workspace",
                  (long long)n, KQ_CHOL_NOALLOC_MAX_N);
        return KQ_ERR_WORKSPACE;
    }
    int dev = 0;
    KQ_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= 64) {
        set_error("kq_chol_inv_noalloc: device index %d not supported", dev);
        return KQ_ERR_INVALID_ARG;
    }
    void* ws = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_noalloc_mu);
        if (!g_noalloc_ptr[dev]) {
            void* p = nullptr;
            const cudaError_t e = cudaGetSymbolAddress(&p, g_chol_scratch);
            if (e != cudaSuccess) return cuda_status(e, "cudaGetSymbolAddress(g_chol_scratch)");
            if (!p) {
                set_error("kq_chol_inv_noalloc: cudaGetSymbolAddress(g_chol_scratch) gave a null address");
                return KQ_ERR_CUDA;
            }
            g_noalloc_ptr[dev] = p;
        }
        ws = g_noalloc_ptr[dev];
    }
    return kq_chol_inv(H, n, damp_rel, Lt, info, ws, kNoallocBytes, stream);
}
