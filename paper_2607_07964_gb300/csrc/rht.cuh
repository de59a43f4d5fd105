// Randomized Hadamard transform building blocks shared by the BiIP rotations (biip.cu) and
// inference (infer.cu): the H_28 construction, the +-1 28-point mix, radix-2/4/8 butterflies
// over a shared-memory vector, and the per-index factors (sign, scale) applied around them.
#pragma once

#include <stdint.h>

#include <utility>

#include "kq_common.cuh"

namespace kq {
namespace {

// ---------------------------------------------------------------------------------------
// H_28 by Paley's second construction over GF(13): the symmetric conference matrix
// C = [[0, 1^T], [1, Q]], Q[i][j] = chi(j - i) (chi = quadratic character mod 13), with
// every entry replaced by a 2 x 2 block: 0 -> [[1,-1],[-1,-1]], c = +-1 -> c [[1,1],[1,-1]].
// Stored as 28 row masks; bit a of row r is set when H_28[r][a] = -1.
constexpr int chi13(int a) {
    a %= 13;
    if (a < 0) a += 13;
    if (a == 0) return 0;
    for (int x = 1; x < 13; ++x)
        if ((x * x) % 13 == a) return 1;
    return -1;
}
constexpr int conf14(int i, int j) {
    if (i == 0 && j == 0) return 0;
    if (i == 0 || j == 0) return 1;
    return chi13((j - 1) - (i - 1));
}
constexpr int h28_entry(int r, int a) {
    const int c = conf14(r / 2, a / 2);
    const int u = r % 2, v = a % 2;
    if (c == 0) return (u == 0 && v == 0) ? 1 : -1;   // [[1,-1],[-1,-1]]
    const int blk = (u == 1 && v == 1) ? -1 : 1;     // [[1,1],[1,-1]]
    return c * blk;
}
struct H28Masks {
    uint32_t m[28];
};
constexpr H28Masks make_h28() {
    H28Masks t{};
    for (int r = 0; r < 28; ++r) {
        uint32_t m = 0;
        for (int a = 0; a < 28; ++a)
            if (h28_entry(r, a) < 0) m |= 1u << a;
        t.m[r] = m;
    }
    return t;
}
constexpr bool h28_is_hadamard() {
    for (int r = 0; r < 28; ++r)
        for (int q = 0; q < 28; ++q) {
            int dot = 0;
            for (int a = 0; a < 28; ++a) dot += h28_entry(r, a) * h28_entry(q, a);
            if (dot != (r == q ? 28 : 0)) return false;
            if (h28_entry(r, q) != h28_entry(q, r)) return false;
        }
    return true;
}
static_assert(h28_is_hadamard(), "H_28 must satisfy H H^T = 28 I and be symmetric");

// Factor applied to element index j before (pre) or after (post) a transform.
enum FactorMode { F_NONE = 0, F_SMUL = 1, F_SDIV = 2, F_SIGN = 3 };

// F_SDIV's sign / s is +-1 over s correctly rounded, i.e. +-__frcp_rn(s): the same bits as
// the division for a numerator of +-1, without its slower sequence.
__device__ __forceinline__ float factor(int mode, const int8_t* sign, const float* s, int64_t j) {
    if (mode == F_NONE) return 1.0f;
    const float sg = static_cast<float>(sign[j]);
    if (mode == F_SIGN || s == nullptr) return sg;
    if (mode == F_SMUL) return sg * s[j];
    const float r = __frcp_rn(s[j]);
    return sg < 0.0f ? -r : r;
}

// factor() for the 16 consecutive indices j0 .. j0 + 15 (j0 a multiple of 16; sign and s
// 16-byte aligned): one 16-byte load of the signs and four of the scales.
__device__ __forceinline__ void factors16(int mode, const int8_t* sign, const float* s, int64_t j0,
                                          float (&f)[16]) {
    if (mode == F_NONE) {
#pragma unroll
        for (int k = 0; k < 16; ++k) f[k] = 1.0f;
        return;
    }
    const int4 sg4 = __ldg(reinterpret_cast<const int4*>(sign + j0));
    const int32_t sw[4] = {sg4.x, sg4.y, sg4.z, sg4.w};
    float sv[16];
    if (mode != F_SIGN && s != nullptr) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float4 v = __ldg(reinterpret_cast<const float4*>(s + j0) + q);
            sv[4 * q] = v.x;
            sv[4 * q + 1] = v.y;
            sv[4 * q + 2] = v.z;
            sv[4 * q + 3] = v.w;
        }
    }
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        const int8_t b = static_cast<int8_t>((sw[k >> 2] >> (8 * (k & 3))) & 0xff);
        const bool neg = b < 0;
        float m;
        if (mode == F_SIGN || s == nullptr) m = 1.0f;
        else if (mode == F_SMUL) m = sv[k];
        else m = __frcp_rn(sv[k]);
        f[k] = neg ? -m : m;
    }
}

// y = H_28 x for 28 values in registers, each output handed to out(r, y_r) as soon as it is
// formed (only x stays live). Each row's sign mask is a template argument taken from the
// compile-time table kH28, so every term is a plain add or subtract.
constexpr H28Masks kH28 = make_h28();

template <uint32_t M>
__device__ __forceinline__ float pm_sum28(const float (&x)[28]) {
    float acc = 0.0f;
#pragma unroll
    for (int a = 0; a < 28; ++a) acc = ((M >> a) & 1u) ? acc - x[a] : acc + x[a];
    return acc;
}

template <typename Out, int... R>
__device__ __forceinline__ void mix28_rows(const float (&x)[28], Out& out, std::integer_sequence<int, R...>) {
    (out(R, pm_sum28<kH28.m[R]>(x)), ...);
}

// Rows BASE .. BASE + sizeof...(R) - 1 of y = H_28 x.
template <int BASE, typename Out, int... R>
__device__ __forceinline__ void mix28_rows_at(const float (&x)[28], Out& out, std::integer_sequence<int, R...>) {
    (out(BASE + R, pm_sum28<kH28.m[BASE + R]>(x)), ...);
}

template <typename Out>
__device__ __forceinline__ void mix28(const float (&x)[28], Out out) {
    mix28_rows(x, out, std::make_integer_sequence<int, 28>{});
}

// In-register Walsh-Hadamard transform of R = 2, 4 or 8 values (natural order).
template <int R>
__device__ __forceinline__ void fwht_reg(float (&x)[8]) {
#pragma unroll
    for (int h = 1; h < R; h <<= 1)
#pragma unroll
        for (int i = 0; i < R; ++i)
            if ((i & h) == 0) {
                const float a = x[i], b = x[i + h];
                x[i] = a + b;
                x[i + h] = a - b;
            }
}
__device__ __forceinline__ void fwht_reg_r(float (&x)[8], int r) {
    if (r == 8) fwht_reg<8>(x);
    else if (r == 4) fwht_reg<4>(x);
    else if (r == 2) fwht_reg<2>(x);
}

// One radix-r pass (span h = 2^lgh) of the Walsh-Hadamard transform over a shared vector
// of n elements (every h*r-aligned block independently). Index math is shifts and masks.
// FIRST: multiply each element by its pre-factor while reading. LAST: instead of writing
// back, store (value * post-factor * scale) to dst (global).
template <bool FIRST, bool LAST>
__device__ __forceinline__ void fwht_pass(float* v, int n, int lgh, int lgr, int pre_mode, int post_mode,
                                          const int8_t* sign, const float* s, float scale, float* dst) {
    const int h = 1 << lgh, r = 1 << lgr;
    for (int g = threadIdx.x; g < (n >> lgr); g += blockDim.x) {
        const int base = ((g >> lgh) << (lgh + lgr)) | (g & (h - 1));
        float x[8];
#pragma unroll
        for (int q = 0; q < 8; ++q)
            if (q < r) {
                x[q] = v[base + q * h];
                if (FIRST) x[q] *= factor(pre_mode, sign, s, base + q * h);
            }
        fwht_reg_r(x, r);
#pragma unroll
        for (int q = 0; q < 8; ++q)
            if (q < r) {
                if (LAST) dst[base + q * h] = x[q] * (factor(post_mode, sign, s, base + q * h) * scale);
                else v[base + q * h] = x[q];
            }
    }
}

// Stage n contiguous floats from global into shared memory with 16-byte cp.async copies
// (scalar copies when the row is not 16-byte aligned).
__device__ __forceinline__ void stage_row(float* v, const float* src, int n) {
    if ((reinterpret_cast<uintptr_t>(src) & 15u) == 0 && (n & 3) == 0) {
        for (int q = threadIdx.x; q < (n >> 2); q += blockDim.x) cp_async16(v + 4 * q, src + 4 * q, 16);
        cp_async_commit();
        cp_async_wait<0>();
    } else {
        for (int j = threadIdx.x; j < n; j += blockDim.x) v[j] = src[j];
    }
    __syncthreads();
}


// v (shared, n floats) <- post (.) (T (pre (.) v)) * scale in place, T = H_28 (x) H_P when
// has28 else H_P (n = 28 P or P), by the whole CTA; returns after a barrier.
__device__ __forceinline__ void block_rht_inplace(float* v, int n, int lgP, bool has28, int pre_mode, int post_mode,
                                                  const int8_t* sign, const float* s, float scale) {
    const int P = 1 << lgP;
    bool first = true;
    if (!has28 && lgP == 0) {
        for (int j = threadIdx.x; j < n; j += blockDim.x)
            v[j] = v[j] * factor(pre_mode, sign, s, j) * (factor(post_mode, sign, s, j) * scale);
        __syncthreads();
        return;
    }
    for (int lgh = 0; lgh < lgP;) {
        const int lgr = min(3, lgP - lgh);
        const bool last = !has28 && lgh + lgr == lgP;
        if (first && last) fwht_pass<true, true>(v, n, lgh, lgr, pre_mode, post_mode, sign, s, scale, v);
        else if (first) fwht_pass<true, false>(v, n, lgh, lgr, pre_mode, post_mode, sign, s, scale, v);
        else if (last) fwht_pass<false, true>(v, n, lgh, lgr, pre_mode, post_mode, sign, s, scale, v);
        else fwht_pass<false, false>(v, n, lgh, lgr, pre_mode, post_mode, sign, s, scale, v);
        first = false;
        __syncthreads();
        lgh += lgr;
    }
    if (has28) {
        for (int b = threadIdx.x; b < P; b += blockDim.x) {
            float x[28];
#pragma unroll
            for (int a = 0; a < 28; ++a) {
                x[a] = v[a * P + b];
                if (first) x[a] *= factor(pre_mode, sign, s, a * P + b);
            }
            mix28(x, [&](int a, float y) { v[a * P + b] = y * (factor(post_mode, sign, s, a * P + b) * scale); });
        }
        __syncthreads();
    }
}

// y = H_28 x by the block structure of Paley's construction: with s_a = x_2a + x_2a+1 and
// d_a = x_2a - x_2a+1 (a < 14), every nonzero entry c of the conference matrix C contributes
// c [[1, 1], [1, -1]], i.e. c s_a to y_2r and c d_a to y_2r+1, and the zero diagonal entry
// [[1, -1], [-1, -1]], i.e. d_r to y_2r and -s_r to y_2r+1. So y_2r = (C s)_r + d_r and
// y_2r+1 = (C d)_r - s_r: 390 additions instead of the 756 of the dense +-1 sums. The
// signs of C come from the same constexpr table (row masks of H_28: the sign of entry
// (2r, 2a) is c for a != r). out(r, y_r) receives every output.
template <int R, uint32_t M>
__device__ __forceinline__ float conf_row_sum(const float (&v)[14]) {
    float acc = 0.0f;
#pragma unroll
    for (int a = 0; a < 14; ++a)
        if (a != R) acc = ((M >> (2 * a)) & 1u) ? acc - v[a] : acc + v[a];
    return acc;
}
template <typename Out, int... R>
__device__ __forceinline__ void mix28_paley_rows(const float (&sv)[14], const float (&dv)[14], Out& out,
                                                 std::integer_sequence<int, R...>) {
    ((out(2 * R, conf_row_sum<R, kH28.m[2 * R]>(sv) + dv[R]),
      out(2 * R + 1, conf_row_sum<R, kH28.m[2 * R]>(dv) - sv[R])),
     ...);
}
template <typename Out>
__device__ __forceinline__ void mix28_paley(const float (&x)[28], Out out) {
    float sv[14], dv[14];
#pragma unroll
    for (int a = 0; a < 14; ++a) {
        sv[a] = x[2 * a] + x[2 * a + 1];
        dv[a] = x[2 * a] - x[2 * a + 1];
    }
    mix28_paley_rows(sv, dv, out, std::make_integer_sequence<int, 14>{});
}
// The block structure above, checked on the table at compile time.
constexpr bool h28_has_paley_blocks() {
    for (int r = 0; r < 14; ++r)
        for (int a = 0; a < 14; ++a) {
            const int e00 = h28_entry(2 * r, 2 * a), e01 = h28_entry(2 * r, 2 * a + 1);
            const int e10 = h28_entry(2 * r + 1, 2 * a), e11 = h28_entry(2 * r + 1, 2 * a + 1);
            if (a == r) {
                if (e00 != 1 || e01 != -1 || e10 != -1 || e11 != -1) return false;
            } else if (e01 != e00 || e10 != e00 || e11 != -e00) {
                return false;
            }
        }
    return true;
}
static_assert(h28_has_paley_blocks(), "H_28 must have the 2 x 2 block structure mix28_paley relies on");

// ---------------------------------------------------------------------------------------
// Walsh-Hadamard transform of n = 2^LG values held in registers, 16 per thread (n / 16
// threads, LG in [9, 14]). Phase q transforms the index bits in rr_mask(LG, q); thread t
// holds the 16 elements that differ in those bits (value k at the bits of the mask, t
// spread over the other bits in order). Phase 0 is the thread's 16 contiguous elements;
// between phases the values move through shared memory (padded one float in 32: at most
// four-way bank conflicts, two for n = 4096); the last phase covers the top four bits, so
// consecutive threads hold consecutive elements. When LG is not a multiple of 4, one phase
// transforms the few remaining bits and carries some already transformed low bits.
__host__ __device__ constexpr int rr_phases(int LG) { return LG / 4 + (LG % 4 ? 1 : 0); }
__host__ __device__ constexpr uint32_t rr_mask(int LG, int q) {
    const int nf = LG / 4, rem = LG % 4;
    if (rem == 0 || q < nf - 1) return 0xFu << (4 * q);
    const int p = 4 * (nf - 1);
    if (q == nf - 1) return (((1u << rem) - 1u) << p) | ((1u << (4 - rem)) - 1u);
    return 0xFu << (p + rem);
}
// The k bits (of a 4-bit k deposited into rr_mask(LG, q)) whose index bits phase q is the
// first to transform.
__host__ __device__ constexpr uint32_t rr_new_kbits(int LG, int q) {
    uint32_t before = 0;
    for (int i = 0; i < q; ++i) before |= rr_mask(LG, i);
    const uint32_t m = rr_mask(LG, q);
    uint32_t kb = 0;
    for (int i = 0, b = 0; i < 32; ++i)
        if ((m >> i) & 1u) {
            if (!((before >> i) & 1u)) kb |= 1u << b;
            ++b;
        }
    return kb;
}

// The low bits of v scattered into the set bits of MASK, in order.
template <uint32_t MASK>
__device__ __forceinline__ int deposit_bits(int v) {
    int out = 0, b = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i)
        if ((MASK >> i) & 1u) {
            out |= ((v >> b) & 1) << i;
            ++b;
        }
    return out;
}

template <uint32_t KB>
__device__ __forceinline__ void fwht_kbits(float (&x)[16]) {
#pragma unroll
    for (int b = 0; b < 4; ++b)
        if ((KB >> b) & 1u)
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if ((i & (1 << b)) == 0) {
                    const float a = x[i], c = x[i | (1 << b)];
                    x[i] = a + c;
                    x[i | (1 << b)] = a - c;
                }
}

__device__ __forceinline__ int pad32(int j) { return j + (j >> 5); }

// Exchange-buffer addresses without padding for LG = 9 and 10 (P = 512, 1024): element j
// goes to j with the row bits r = j >> 5 XORed into its bank bits through a GF(2)-linear
// map chosen so that, for each of the four access patterns of the two exchanges (a warp's 32
// threads vary index bits {4..8}, {2, 3, 6, 7, 8} or {0..4} for LG = 10; {4..8}, {3, 5..8} or
// {0..4} for LG = 9), the 32 addresses fall in 32 distinct banks. A permutation of [0, P)
// within each 32-float row, so the buffer needs no padding.
template <int LG>
__device__ __forceinline__ int swz_bank(int j) {
    static_assert(LG == 9 || LG == 10, "exchange swizzle for P = 512 and 1024");
    const int r = j >> 5;
    int m;
    if constexpr (LG == 10)
        m = ((r & 1) << 3) | ((r >> 1) & 1) | (((r >> 2) & 1) << 1) | (((r >> 3) & 1) * 0x14);
    else
        m = (r & 7) | (((r >> 3) & 1) * 0x18);
    return j ^ m;
}

// Values of phase Q - 1 to shared memory, those of phase Q back, and phase Q's butterflies.
// Every thread of the CTA calls it (two barriers); threads with act false hold no values.
// SWZ: the buffer holds P floats addressed through swz_bank (LG = 9, 10), else P + P / 32
// padded one float in 32.
template <int LG, int Q, bool SWZ = false>
__device__ __forceinline__ void rr_transpose(float (&x)[16], float* buf, int t, bool act = true) {
    constexpr uint32_t N1 = (1u << LG) - 1u;
    constexpr uint32_t MW = rr_mask(LG, Q - 1), MR = rr_mask(LG, Q);
    const int tw = deposit_bits<N1 & ~MW>(t), tr = deposit_bits<N1 & ~MR>(t);
    auto at = [](int j) {
        if constexpr (SWZ)
            return swz_bank<LG>(j);
        else
            return pad32(j);
    };
    __syncthreads();   // the previous reads of buf are done
    if (act) {
#pragma unroll
        for (int k = 0; k < 16; ++k) buf[at(tw | deposit_bits<MW>(k))] = x[k];
    }
    __syncthreads();
    if (act) {
#pragma unroll
        for (int k = 0; k < 16; ++k) x[k] = buf[at(tr | deposit_bits<MR>(k))];
        fwht_kbits<rr_new_kbits(LG, Q)>(x);
    }
}


}  // namespace
}  // namespace kq
