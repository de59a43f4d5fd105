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
//   step k: diag  -- factor A_kk = C_kk C_kk^T and invert C_kk in shared memory (1 CTA);
//           panel -- C_ik = A_ik C_kk^-T (i > k) and Z_kj = C_kk^-1 B_kj (j < k);
//           update-- A_ij -= C_ik C_jk^T (k < j <= i) and B_ij -= C_ik Z_kj (j <= k < i),
// where B (stored in Z's blocks) is the right-hand side I of C Z = I after the earlier
// steps' eliminations. The matrix is padded to a multiple of nb with an identity block.
// Look-ahead: the update is split into the tiles step k + 1 reads first (row and column
// block k + 1, on the caller's stream, on the critical path) and the rest (on a library
// side stream, beside step k + 1's diagonal factorization and panel); step k + 1's own
// first tiles wait for that rest, which also writes them.
// All arithmetic is fp32 with fused multiply-add.
#include <math.h>

#include "kq_common.cuh"
#include "tile_gemm.cuh"

namespace kq {
namespace {

constexpr int NB = 128;
constexpr int LD = NB + 1;                      // padded shared-memory row
constexpr int TILE_FLOATS = NB * LD;

struct Work {
    float* A;      // npad x npad, reversed damped H -> C (lower)
    float* Z;      // npad x npad, B -> C^-1 (lower)
    double* dsum;  // sum of diag(H)
};

inline size_t npad_of(int64_t n) { return static_cast<size_t>(cdiv(n, NB) * NB); }

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
        A[e] = v;
        Z[e] = 0.0f;
    }
}

// ---------------------------------------------------------------- diag block
constexpr int DIAG_THREADS = 512;
constexpr int SB = 32;                        // leaf size inside the diagonal block
constexpr int TLDD = SB + 1;
constexpr size_t DIAG_SMEM = (2 * TILE_FLOATS + NB * TLDD + 2 * NB) * sizeof(float);

__device__ __forceinline__ void named_barrier(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// Leaf factor by 128 threads (warps 0..3, named barrier 1): thread t owns row t / 4 of the
// 32 x 32 leaf at s and the columns k = t (mod 4). Step j updates the trailing part with
// the pivot scaling deferred, a_ik -= (a_ij / p_j) a_kj; afterwards C_ij = a_ij / sqrt(p_j),
// C_jj = sqrt(p_j), and dv[j] = 1 / C_jj. Returns the first non-positive pivot, or -1.
__device__ __forceinline__ int leaf_factor128(float* s, int ld, float* pv, float* dv, int t) {
    const int i = t >> 2, q = t & 3;
    int bad = -1;
#pragma unroll 1
    for (int j = 0; j < SB; ++j) {
        const float p = s[j * ld + j];
        if (!(p > 0.0f) && bad < 0) bad = j;
        if (i > j) {
            const float f = s[i * ld + j] * __fdiv_rn(1.0f, p);
            // at most 8 columns per thread: unrolled so all loads are issued together
            float sk[8], si[8];
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                const int k = j + 1 + q + 4 * m;
                if (k <= i) {
                    sk[m] = s[k * ld + j];
                    si[m] = s[i * ld + k];
                }
            }
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                const int k = j + 1 + q + 4 * m;
                if (k <= i) s[i * ld + k] = fmaf(-f, sk[m], si[m]);
            }
        }
        if (t == 0) pv[j] = p;
        named_barrier(1, 128);
    }
    for (int e = t; e < SB * SB; e += 128) {
        const int r = e >> 5, c = e & 31;
        const float d = sqrtf(pv[c]);
        if (c < r) s[r * ld + c] = __fdiv_rn(s[r * ld + c], d);
        else if (c == r) s[r * ld + c] = d;
        else s[r * ld + c] = 0.0f;
        if (r == 0) dv[c] = __fdiv_rn(1.0f, d);
    }
    named_barrier(1, 128);
    return bad;
}

// Leaf inverse by 128 threads without block barriers: four lanes per column c (8 columns
// per warp), lane q of the group owning rows i = q (mod 4). Step i: the owner of row i
// finalizes x_ic = b_ic / C_ii and shuffles it to the group, which updates
// b_i'c -= C_i'i x_ic for its rows i' > i. X (stride ld) starts as the identity.
__device__ __forceinline__ void leaf_inverse128(const float* L, float* X, int ld, const float* dv, int t) {
    const int c = t >> 2, q = t & 3;
    const int lane = threadIdx.x & 31, gbase = lane & ~3;
    for (int r = q; r < SB; r += 4) X[r * ld + c] = (r == c) ? 1.0f : 0.0f;
    __syncwarp();
#pragma unroll 1
    for (int i = 0; i < SB; ++i) {
        float xi = 0.0f;
        if ((i & 3) == q) {
            xi = X[i * ld + c] * dv[i];
            X[i * ld + c] = xi;
        }
        xi = __shfl_sync(0xffffffffu, xi, gbase | (i & 3));
        const int r0 = i + 1 + ((q - i - 1) & 3);   // first row > i owned by this lane
        float lr[8], xr[8];
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const int r = r0 + 4 * m;
            if (r < SB) {
                lr[m] = L[r * ld + i];
                xr[m] = X[r * ld + c];
            }
        }
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const int r = r0 + 4 * m;
            if (r < SB) X[r * ld + c] = fmaf(-lr[m], xi, xr[m]);
        }
        __syncwarp();
    }
}

// Factor A_kk = C C^T and invert C in shared memory, blocked by 32 x 32 leaves:
//   leaf p: warps 0..3 factor leaf (p, p) while warps 4..7 invert leaf p - 1; then one warp
//   per row solves the rows below against the leaf (C_qp = A_qp C_pp^-T) and all warps
//   update the trailing part with 4 x 4 register tiles;
//   after the last leaf: X_qp = -X_qq sum_{r=p}^{q-1} C_qr X_rp by increasing q - p.
// Writes C to A_kk and X = C^-1 to Z_kk. A non-positive pivot records its index in H's
// own numbering (1-based).
__global__ void __launch_bounds__(DIAG_THREADS) chol_diag_kernel(Work w, int64_t n, int64_t npad, int k, int* info) {
    extern __shared__ float sm[];
    float* a = sm;                        // [NB][LD]  A_kk -> C
    float* x = sm + TILE_FLOATS;          // [NB][LD]  C^-1
    float* t = sm + 2 * TILE_FLOATS;      // [NB][TLDD] temporaries
    float* pv = t + NB * TLDD;            // [NB] pivots
    float* dv = pv + NB;                  // [NB] 1 / C_jj
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr int NW = DIAG_THREADS / 32;
    const int64_t off = static_cast<int64_t>(k) * NB;
    for (int e = tid; e < NB * NB; e += blockDim.x) {
        const int r = e / NB, c = e % NB;
        a[r * LD + c] = c <= r ? w.A[(off + r) * npad + off + c] : 0.0f;
        x[r * LD + c] = 0.0f;
    }
    __syncthreads();
    for (int p = 0; p <= NB / SB; ++p) {
        const int o = p * SB;
        if (p < NB / SB && warp < 4) {
            const int bad = leaf_factor128(a + o * LD + o, LD, pv + o, dv + o, tid);
            if (bad >= 0 && tid == 0) {
                const int64_t rev = off + o + bad;
                if (rev < n) record_error(info, static_cast<int>(n - rev));
            }
        } else if (p > 0 && warp >= 4 && warp < 8) {
            const int po = o - SB;
            leaf_inverse128(a + po * LD + po, x + po * LD + po, LD, dv + po, tid - 128);
        }
        __syncthreads();
        if (p == NB / SB) break;
        const int nr = NB - o - SB;
        // rows below: warp per row (3 rows interleaved), lane = column of the leaf
        for (int r0 = warp; r0 < nr; r0 += 3 * NW) {
            float v[3];
            int rr[3];
#pragma unroll
            for (int u = 0; u < 3; ++u) {
                rr[u] = r0 + u * NW;
                v[u] = rr[u] < nr ? a[(o + SB + rr[u]) * LD + o + lane] : 0.0f;
            }
            const float* L = a + o * LD + o;
#pragma unroll 4
            for (int m = 0; m < SB; ++m) {
                const float lm = L[lane * LD + m];
                const float dm = dv[o + m];
#pragma unroll
                for (int u = 0; u < 3; ++u) {
                    const float vm = __shfl_sync(0xffffffffu, v[u], m) * dm;
                    if (lane == m) v[u] = vm;
                    else if (lane > m) v[u] = fmaf(-vm, lm, v[u]);
                }
            }
#pragma unroll
            for (int u = 0; u < 3; ++u)
                if (rr[u] < nr) a[(o + SB + rr[u]) * LD + o + lane] = v[u];
        }
        __syncthreads();
        // trailing update of rows/cols [o + SB, NB): 4 x 4 register tiles of the lower part
        const int nt = nr / 4;
        for (int e = tid; e < nt * nt; e += blockDim.x) {
            const int tr = e / nt, tc = e % nt;
            if (tc > tr) continue;
            const int r0 = o + SB + 4 * tr, c0 = o + SB + 4 * tc;
            float acc[4][4] = {};
#pragma unroll 4
            for (int m = 0; m < SB; ++m) {
                float ra[4], cb[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    ra[u] = a[(r0 + u) * LD + o + m];
                    cb[u] = a[(c0 + u) * LD + o + m];
                }
#pragma unroll
                for (int u = 0; u < 4; ++u)
#pragma unroll
                    for (int v2 = 0; v2 < 4; ++v2) acc[u][v2] = fmaf(ra[u], cb[v2], acc[u][v2]);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v2 = 0; v2 < 4; ++v2)
                    if (c0 + v2 <= r0 + u) a[(r0 + u) * LD + c0 + v2] -= acc[u][v2];
        }
        __syncthreads();
    }
    // off-diagonal leaves of X, by distance d = q - p, 4 x 4 register tiles
    for (int d = 1; d < NB / SB; ++d) {
        const int nblk = NB / SB - d;
        for (int e = tid; e < nblk * 64; e += blockDim.x) {   // T_qp = sum_r C_qr X_rp
            const int b = e >> 6, ti = (e >> 3) & 7, tj = e & 7;
            const int pp = b, qq = b + d;
            float acc[4][4] = {};
            for (int r2 = pp; r2 < qq; ++r2) {
#pragma unroll 4
                for (int m = 0; m < SB; ++m) {
                    float ca[4], xb[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        ca[u] = a[(qq * SB + 4 * ti + u) * LD + r2 * SB + m];
                        xb[u] = x[(r2 * SB + m) * LD + pp * SB + 4 * tj + u];
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u)
#pragma unroll
                        for (int v2 = 0; v2 < 4; ++v2) acc[u][v2] = fmaf(ca[u], xb[v2], acc[u][v2]);
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v2 = 0; v2 < 4; ++v2) t[(b * SB + 4 * ti + u) * TLDD + 4 * tj + v2] = acc[u][v2];
        }
        __syncthreads();
        for (int e = tid; e < nblk * 64; e += blockDim.x) {   // X_qp = -X_qq T_qp
            const int b = e >> 6, ti = (e >> 3) & 7, tj = e & 7;
            const int pp = b, qq = b + d;
            float acc[4][4] = {};
#pragma unroll 4
            for (int m = 0; m < SB; ++m) {
                float xa[4], tb[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    xa[u] = x[(qq * SB + 4 * ti + u) * LD + qq * SB + m];
                    tb[u] = t[(b * SB + m) * TLDD + 4 * tj + u];
                }
#pragma unroll
                for (int u = 0; u < 4; ++u)
#pragma unroll
                    for (int v2 = 0; v2 < 4; ++v2) acc[u][v2] = fmaf(xa[u], tb[v2], acc[u][v2]);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v2 = 0; v2 < 4; ++v2) x[(qq * SB + 4 * ti + u) * LD + pp * SB + 4 * tj + v2] = -acc[u][v2];
        }
        __syncthreads();
    }
    for (int e = tid; e < NB * NB; e += blockDim.x) {
        const int r = e / NB, c = e % NB;
        w.A[(off + r) * npad + off + c] = c <= r ? a[r * LD + c] : 0.0f;
        w.Z[(off + r) * npad + off + c] = c <= r ? x[r * LD + c] : 0.0f;
    }
}

// --------------------------------------------------------------------- panel
// CTA b < k: Z_kb <- C_kk^-1 Z_kb.  CTA b >= k: i = b + 1, A_ik <- A_ik C_kk^-T. The whole
// input tile is consumed before the in-place write (gemm_tile ends with a barrier).
__global__ void __launch_bounds__(G_THREADS, 2) chol_panel_kernel(Work w, int64_t npad, int k) {
    extern __shared__ __align__(16) float sm[];
    const int b = blockIdx.x;
    const int64_t off = static_cast<int64_t>(k) * NB;
    const float* cinv = w.Z + off * npad + off;
    float acc[8][8];
    float* out;
    bool nn;
    if (b < k) {
        out = w.Z + off * npad + static_cast<int64_t>(b) * NB;
        gemm_tile<true, true>(cinv, npad, NB, out, npad, NB, NB, acc, sm);   // C^-1 x B (B N-contiguous)
        nn = true;
    } else {
        out = w.A + static_cast<int64_t>(b + 1) * NB * npad + off;
        gemm_tile<false, true>(out, npad, NB, cinv, npad, NB, NB, acc, sm);  // A x (C^-1)^T
        nn = false;
    }
    const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int c = nn ? gt_col<true>(tx, j) : gt_col<false>(tx, j);
            out[static_cast<int64_t>(gt_row(ty, i)) * npad + c] = acc[i][j];
        }
}

// out[tile] -= acc, loads of 32 values issued before their stores.
template <bool BN>
__device__ __forceinline__ void sub_tile(float* out, int64_t ld, const float (&acc)[8][8]) {
    const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        float ov[4][8];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 8; ++b)
                ov[a][b] = out[static_cast<int64_t>(gt_row(ty, 4 * h + a)) * ld + gt_col<BN>(tx, b)];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 8; ++b)
                out[static_cast<int64_t>(gt_row(ty, 4 * h + a)) * ld + gt_col<BN>(tx, b)] = ov[a][b] - acc[4 * h + a][b];
    }
}

// -------------------------------------------------------------------- update
// Tile (i, j) of step k, k < i < nbk, 0 <= j <= i:
//   j > k : A_ij -= C_ik C_jk^T;     j <= k : Z_ij -= C_ik Z_kj.
__device__ __forceinline__ void update_tile(const Work& w, int64_t npad, int k, int i, int j, float* sm) {
    const int64_t ko = static_cast<int64_t>(k) * NB;
    const float* cik = w.A + static_cast<int64_t>(i) * NB * npad + ko;
    const bool apart = j > k;
    float acc[8][8];
    if (apart)
        gemm_tile<false, true>(cik, npad, NB, w.A + static_cast<int64_t>(j) * NB * npad + ko, npad, NB, NB, acc, sm);
    else
        gemm_tile<true, true>(cik, npad, NB, w.Z + ko * npad + static_cast<int64_t>(j) * NB, npad, NB, NB, acc, sm);
    float* out = (apart ? w.A : w.Z) + static_cast<int64_t>(i) * NB * npad + static_cast<int64_t>(j) * NB;
    if (apart)
        sub_tile<false>(out, npad, acc);
    else
        sub_tile<true>(out, npad, acc);
}

// The tiles that step k + 1 reads first: row block k + 1 (tiles (k + 1, j), j <= k + 1)
// and block column k + 1 below it (tiles (i, k + 1), i > k + 1). nbk CTAs.
__global__ void __launch_bounds__(G_THREADS, 2) chol_next_kernel(Work w, int64_t npad, int k) {
    extern __shared__ __align__(16) float sm[];
    const int bid = blockIdx.x;
    if (bid < k + 2)
        update_tile(w, npad, k, k + 1, bid, sm);
    else
        update_tile(w, npad, k, bid, k + 1, sm);
}

// The other tiles of step k: (i, j) with i > k + 1 and j != k + 1 (i tiles in row block i).
__global__ void __launch_bounds__(G_THREADS, 2) chol_rest_kernel(Work w, int64_t npad, int k) {
    extern __shared__ __align__(16) float sm[];
    int bid = blockIdx.x;
    int i = k + 2;
    while (bid >= i) {
        bid -= i;
        ++i;
    }
    update_tile(w, npad, k, i, bid < k + 1 ? bid : bid + 1, sm);
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
        if (i < n && j < n) Lt[i * n + j] = t[threadIdx.x][r];
    }
}

}  // namespace
}  // namespace kq

using namespace kq;

extern "C" size_t kq_chol_inv_workspace(int64_t n) {
    if (n < 1) return 0;
    const size_t np = npad_of(n);
    return 2 * np * np * sizeof(float) + 256;
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
    Work w;
    w.A = static_cast<float*>(ws);
    w.Z = w.A + npad * npad;
    w.dsum = reinterpret_cast<double*>(w.Z + npad * npad);
    static bool attr = false;
    if (!attr) {
        KQ_CUDA(cudaFuncSetAttribute(chol_diag_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(DIAG_SMEM)));
        KQ_CUDA(cudaFuncSetAttribute(chol_panel_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(G_SMEM)));
        KQ_CUDA(cudaFuncSetAttribute(chol_next_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(G_SMEM)));
        KQ_CUDA(cudaFuncSetAttribute(chol_rest_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(G_SMEM)));
        attr = true;
    }
    diag_sum_kernel<<<1, 1024, 0, stream>>>(H, n, w.dsum);
    KQ_LAUNCH_CHECK("diag_sum_kernel");
    const int64_t total = npad * npad;
    const int64_t pgrid = std::min<int64_t>(cdiv(total, 256), static_cast<int64_t>(num_sms()) * 32);
    prep_kernel<<<static_cast<unsigned>(pgrid), 256, 0, stream>>>(H, n, npad, damp_rel, w.dsum, w.A, w.Z);
    KQ_LAUNCH_CHECK("prep_kernel");
    SideStream* side = nbk > 2 ? side_stream(stream) : nullptr;
    bool forked = false;
    for (int k = 0; k < nbk; ++k) {
        chol_diag_kernel<<<1, DIAG_THREADS, DIAG_SMEM, stream>>>(w, n, npad, k, info);
        KQ_LAUNCH_CHECK("chol_diag_kernel");
        if (nbk > 1) {
            chol_panel_kernel<<<nbk - 1, G_THREADS, G_SMEM, stream>>>(w, npad, k);
            KQ_LAUNCH_CHECK("chol_panel_kernel");
        }
        if (k + 1 >= nbk) break;
        int64_t rest = 0;
        for (int i = k + 2; i < nbk; ++i) rest += i;
        const bool fork = side && rest > 0;
        if (fork) KQ_CUDA(cudaEventRecord(side->ev[0], stream));      // panel k done
        if (forked) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));  // rest of step k - 1 done
        chol_next_kernel<<<nbk, G_THREADS, G_SMEM, stream>>>(w, npad, k);
        KQ_LAUNCH_CHECK("chol_next_kernel");
        if (rest > 0) {
            cudaStream_t rs = stream;
            if (fork) {
                KQ_CUDA(cudaStreamWaitEvent(side->s, side->ev[0], 0));
                rs = side->s;
            }
            chol_rest_kernel<<<static_cast<unsigned>(rest), G_THREADS, G_SMEM, rs>>>(w, npad, k);
            KQ_LAUNCH_CHECK("chol_rest_kernel");
            if (fork) {
                KQ_CUDA(cudaEventRecord(side->ev[1], side->s));
                forked = true;
            }
        }
    }
    if (forked) KQ_CUDA(cudaStreamWaitEvent(stream, side->ev[1], 0));
    finish_kernel<<<dim3(static_cast<unsigned>(cdiv(n, 32)), static_cast<unsigned>(cdiv(n, 32))),
                    dim3(32, 8), 0, stream>>>(w.Z, n, npad, Lt);
    KQ_LAUNCH_CHECK("finish_kernel");
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
constexpr size_t kNoallocBytes =
    2 * static_cast<size_t>(KQ_CHOL_NOALLOC_MAX_N) * KQ_CHOL_NOALLOC_MAX_N * sizeof(float) + 256;
static __device__ __align__(256) unsigned char g_chol_scratch[kNoallocBytes];
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
            if (e != cudaSuccess || !p) return cuda_status(e, "cudaGetSymbolAddress(g_chol_scratch)");
            g_noalloc_ptr[dev] = p;
        }
        ws = g_noalloc_ptr[dev];
    }
    return kq_chol_inv(H, n, damp_rel, Lt, info, ws, kNoallocBytes, stream);
}
