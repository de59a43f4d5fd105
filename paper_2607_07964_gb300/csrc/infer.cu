// Inference with a quantized layer: y = W^ x with the incoherence processing reverted
// online (Sec. 3.2: "At inference, BiIP introduces no additional overhead beyond QuIP#";
// the reverted weight of Algorithm 2 is W^ = S_G^-1 U^T Q' V S_X^-1, Q' the dequantized
// codes). The dense W^ is never formed:
//   x' = V S_X^-1 x        fast Hadamard transform of each token (biip.cu row transform)
//   y' = Q' x'             dequantizing matrix-vector product over packed codes (this file)
//   y  = S_G^-1 U^T y'     fast Hadamard transform of each output
// so the cost is the code stream plus O(d log d) per token.
//
// Packed codes: each row of codes is stored as 32-bit words along d_in, word w holding codes
// w * (32 / pb) .. + (32 / pb) - 1, code t of the word in bits [t pb, t pb + pb); pb = bits for
// 2, 4 and 8-bit codes, and 4 for 3-bit codes (3-bit codes travel in 4-bit lanes).
//
// Fused kernel (when B max(d_in, d_out) floats fit in shared memory): every CTA of a
// persistent grid first forms x' = V S_X^-1 x in shared memory (the transform is O(d log d),
// cheap next to the code stream, so each CTA does it rather than wait for one) and the sums
// of x' over each 128-column group; then warps stream rows of codes, lane i taking words
// i, i + 32, ... with eight words in flight, and accumulate
//   y'_r = sum_g scale_rg (sum_{c in g} q_rc x'_c) - sum_g scale_rg zero_rg X'_g;
// a code q becomes the exact float q by a byte permute that places it under the exponent of
// 2^23 (the float 2^23 + q) and one subtraction. The last CTA to finish (an atomic ticket
// after a memory fence; no CTA waits for another) applies y = S_G^-1 U^T y' to the gathered
// y'. Larger B d: three kernels (row transform, the same product reading x' through L1 with
// per-16-column sums, row transform).
#include "kq_common.cuh"
#include "rht.cuh"

namespace kq {
kq_status rotate_rows_pre_div(float* M, int64_t rows, int64_t n, const float* s, const int8_t* sign,
                              cudaStream_t stream);
kq_status rotate_rows_inv(float* M, int64_t rows, int64_t n, const float* s, const int8_t* sign,
                          cudaStream_t stream);

namespace {

constexpr int KQ_INFER_MAX_B = 8;

inline int lane_bits(int bits) { return bits == 3 ? 4 : bits; }

// packed[r][w] = sum_t codes[r][w * cpw + t] << (t pb), one thread per word.
__global__ void pack_kernel(const uint8_t* __restrict__ codes, int64_t d_out, int64_t d_in, int pb,
                            uint32_t* __restrict__ packed) {
    const int cpw = 32 / pb;
    const int64_t wpr = d_in / cpw;
    const int64_t total = d_out * wpr;
    const uint32_t mask = (1u << pb) - 1u;
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t r = e / wpr, w = e - r * wpr;
        const uint8_t* src = codes + r * d_in + w * cpw;
        uint32_t v = 0;
        for (int t = 0; t < cpw; ++t) v |= (static_cast<uint32_t>(src[t]) & mask) << (t * pb);
        packed[e] = v;
    }
}

// xs[b][k] = sum of x'[b][16 k .. 16 k + 15] (fp32, in order).
__global__ void runsum16_kernel(const float* __restrict__ x, int64_t B, int64_t d_in, float* __restrict__ xs) {
    const int64_t runs = d_in / 16;
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < B * runs;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const float4* p = reinterpret_cast<const float4*>(x + (e / runs) * d_in + (e % runs) * 16);
        float a = 0.0f;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float4 v = p[q];
            a = a + v.x;
            a = a + v.y;
            a = a + v.z;
            a = a + v.w;
        }
        xs[e] = a;
    }
}

// The float q for the byte k (0..3) of w: the bits 0x4B0000qq are 2^23 + q.
__device__ __forceinline__ float byte_as_float(uint32_t w, int k) {
    return __int_as_float(static_cast<int>(__byte_perm(w, 0x4B000000u, 0x7440u | static_cast<uint32_t>(k)))) - 8388608.0f;
}

// Codes of one 32-bit word as floats, in code order (PB bits each).
template <int PB>
__device__ __forceinline__ void word_codes(uint32_t w, float (&q)[32 / PB]) {
    if constexpr (PB == 8) {
#pragma unroll
        for (int k = 0; k < 4; ++k) q[k] = byte_as_float(w, k);
    } else if constexpr (PB == 4) {
        const uint32_t lo = w & 0x0F0F0F0Fu, hi = (w >> 4) & 0x0F0F0F0Fu;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            q[2 * k] = byte_as_float(lo, k);
            q[2 * k + 1] = byte_as_float(hi, k);
        }
    } else {
#pragma unroll
        for (int sft = 0; sft < 4; ++sft) {
            const uint32_t m = (w >> (2 * sft)) & 0x03030303u;
#pragma unroll
            for (int k = 0; k < 4; ++k) q[4 * k + sft] = byte_as_float(m, k);
        }
    }
}

// y'[b][r] = sum_g scale[r][g] (sum_{c in g} q_rc x'[b][c] - zero[r][g] sum_{c in g} x'[b][c]).
template <int PB, int B>
__global__ void __launch_bounds__(256) dequant_gemv_kernel(const uint32_t* __restrict__ packed,
                                                           const float* __restrict__ scale,
                                                           const int32_t* __restrict__ zero, int64_t d_out,
                                                           int64_t d_in, int group, const float* __restrict__ x,
                                                           const float* __restrict__ xs, float* __restrict__ y) {
    constexpr int CPW = 32 / PB;          // codes per word
    constexpr int CPC = 4 * CPW;          // codes per 16-byte chunk
    const int lane = threadIdx.x & 31;
    const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
    const int64_t chunks = d_in / CPC;
    const int64_t ng = group ? d_in / group : 1;
    const int64_t runs = d_in / 16;
    for (int64_t r = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5); r < d_out; r += warps) {
        const uint4* row = reinterpret_cast<const uint4*>(packed + r * (d_in / CPW));
        float acc[B];
#pragma unroll
        for (int b = 0; b < B; ++b) acc[b] = 0.0f;
        for (int64_t c = lane; c < chunks; c += 32) {
            const uint4 wv = __ldg(row + c);
            const uint32_t ws[4] = {wv.x, wv.y, wv.z, wv.w};
            const int64_t col0 = c * CPC;
            float dot[B];
#pragma unroll
            for (int b = 0; b < B; ++b) dot[b] = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                float q[CPW];
                word_codes<PB>(ws[k], q);
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const float4* xp = reinterpret_cast<const float4*>(x + b * d_in + col0 + k * CPW);
#pragma unroll
                    for (int v = 0; v < CPW / 4; ++v) {
                        const float4 xv = __ldg(xp + v);
                        dot[b] = fmaf(q[4 * v], xv.x, dot[b]);
                        dot[b] = fmaf(q[4 * v + 1], xv.y, dot[b]);
                        dot[b] = fmaf(q[4 * v + 2], xv.z, dot[b]);
                        dot[b] = fmaf(q[4 * v + 3], xv.w, dot[b]);
                    }
                }
            }
            // a chunk lies inside one group (groups are 128 columns, chunks 16 to 64)
            const int64_t gi = r * ng + (group ? col0 / group : 0);
            const float sc = __ldg(scale + gi);
            const float z = static_cast<float>(__ldg(zero + gi));
#pragma unroll
            for (int b = 0; b < B; ++b) {
                float sx = 0.0f;
#pragma unroll
                for (int u = 0; u < CPC / 16; ++u) sx += __ldg(xs + b * runs + col0 / 16 + u);
                acc[b] = fmaf(sc, fmaf(-z, sx, dot[b]), acc[b]);
            }
        }
#pragma unroll
        for (int b = 0; b < B; ++b) {
            float v = acc[b];
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) y[b * d_out + r] = v;
        }
    }
}

constexpr int FU = 8;   // words in flight per lane

template <int PB, int B>
__global__ void __launch_bounds__(256) infer_fused_kernel(
    const uint32_t* __restrict__ packed, const float* __restrict__ scale, const int32_t* __restrict__ zero, int d_out,
    int d_in, int group, const float* __restrict__ s_x, const float* __restrict__ s_g,
    const int8_t* __restrict__ sign_u, const int8_t* __restrict__ sign_v, int lg_in, int has28_in, int lg_out,
    int has28_out, const float* __restrict__ x, float* __restrict__ yp, float* __restrict__ y,
    unsigned int* __restrict__ ticket) {
    extern __shared__ __align__(16) float fsm[];
    constexpr int CPW = 32 / PB;
    const int dmax = max(d_in, d_out);
    const int gsz = group ? group : d_in;
    const int ng = d_in / gsz;
    float* xv = fsm;                           // B x d_in: x'; the last CTA reuses it for y'
    float* gs = fsm + static_cast<int64_t>(B) * dmax;   // B x ng: group sums of x'
    __shared__ int is_last;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarp = blockDim.x >> 5;
    const int wpr = d_in / CPW;
    // first batch of this warp's first row, in flight while x' is formed
    int r = blockIdx.x * nwarp + warp;
    uint32_t cur[FU];
#pragma unroll
    for (int u = 0; u < FU; ++u) {
        const int w = lane + 32 * u;
        cur[u] = (r < d_out && w < wpr) ? __ldg(packed + static_cast<int64_t>(r) * wpr + w) : 0u;
    }
    // x' = V S_X^-1 x per token
    const float isn_in = rsqrtf(static_cast<float>(d_in));
    // the factors sigma_V / s_X are applied while loading (independent vector loads), so the
    // butterflies below run on shared memory alone
    // (four vectors per thread per step, all loads issued before use)
    {
        const float4* s4 = reinterpret_cast<const float4*>(s_x);
        const char4* g4 = reinterpret_cast<const char4*>(sign_v);
        const int nq = d_in / 4;
        for (int q0 = threadIdx.x; q0 < nq; q0 += 4 * blockDim.x) {
            float4 f[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int q = q0 + u * blockDim.x;
                if (q < nq) {
                    const float4 sc = __ldg(s4 + q);
                    const char4 sg = g4[q];
                    f[u] = make_float4(static_cast<float>(sg.x) / sc.x, static_cast<float>(sg.y) / sc.y,
                                       static_cast<float>(sg.z) / sc.z, static_cast<float>(sg.w) / sc.w);
                }
            }
#pragma unroll
            for (int b = 0; b < B; ++b) {
                float4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int q = q0 + u * blockDim.x;
                    if (q < nq) v[u] = __ldg(reinterpret_cast<const float4*>(x + static_cast<int64_t>(b) * d_in) + q);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int q = q0 + u * blockDim.x;
                    if (q < nq)
                        reinterpret_cast<float4*>(xv + b * d_in)[q] =
                            make_float4(v[u].x * f[u].x, v[u].y * f[u].y, v[u].z * f[u].z, v[u].w * f[u].w);
                }
            }
        }
    }
    __syncthreads();
    for (int b = 0; b < B; ++b)
        block_rht_inplace(xv + b * d_in, d_in, lg_in, has28_in != 0, F_NONE, F_NONE, sign_v, s_x, isn_in);
    for (int e = warp; e < B * ng; e += nwarp) {
        const float* p = xv + (e / ng) * d_in + (e % ng) * gsz;
        float a = 0.0f;
        for (int j = lane; j < gsz; j += 32) a += p[j];
        for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
        if (lane == 0) gs[e] = a;
    }
    __syncthreads();
    const int rstride = gridDim.x * nwarp;
    const int gshift = group ? 7 : 30;   // group of a column: col >> 7 (128 columns) or 0 (whole row)
    for (; r < d_out; r += rstride) {
        const float* srow = scale + static_cast<int64_t>(r) * ng;
        float acc[B];
#pragma unroll
        for (int b = 0; b < B; ++b) acc[b] = 0.0f;
        for (int w0 = lane; w0 < wpr; w0 += 32 * FU) {
            // next batch: the rest of this row, else the next row's first batch
            uint32_t nxt[FU];
            const int nw0 = w0 + 32 * FU;
            const int nr = nw0 < wpr ? r : r + rstride;
            const int nb = nw0 < wpr ? nw0 : lane;
#pragma unroll
            for (int u = 0; u < FU; ++u) {
                const int w = nb + 32 * u;
                nxt[u] = (nr < d_out && w < wpr) ? __ldg(packed + static_cast<int64_t>(nr) * wpr + w) : 0u;
            }
#pragma unroll
            for (int u = 0; u < FU; ++u) {
                const int w = w0 + 32 * u;
                if (w < wpr) {
                    float q[CPW];
                    word_codes<PB>(cur[u], q);
                    const int col = w * CPW;
                    const float sc = __ldg(srow + (col >> gshift));
#pragma unroll
                    for (int b = 0; b < B; ++b) {
                        const float4* xp = reinterpret_cast<const float4*>(xv + b * d_in + col);
                        float d = 0.0f;
#pragma unroll
                        for (int v = 0; v < CPW / 4; ++v) {
                            const float4 xq = xp[v];
                            d = fmaf(q[4 * v], xq.x, d);
                            d = fmaf(q[4 * v + 1], xq.y, d);
                            d = fmaf(q[4 * v + 2], xq.z, d);
                            d = fmaf(q[4 * v + 3], xq.w, d);
                        }
                        acc[b] = fmaf(sc, d, acc[b]);
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < FU; ++u) cur[u] = nxt[u];
        }
        // zero points: - sum_g scale_g zero_g X'_g
        for (int g = lane; g < ng; g += 32) {
            const int64_t gi = static_cast<int64_t>(r) * ng + g;
            const float sz = __ldg(scale + gi) * static_cast<float>(__ldg(zero + gi));
#pragma unroll
            for (int b = 0; b < B; ++b) acc[b] = fmaf(-sz, gs[b * ng + g], acc[b]);
        }
#pragma unroll
        for (int b = 0; b < B; ++b) {
            float v = acc[b];
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) yp[static_cast<int64_t>(b) * d_out + r] = v;
        }
    }
    // the last CTA to finish applies y = S_G^-1 U^T y'
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) is_last = atomicAdd(ticket, 1u) == gridDim.x - 1;
    __syncthreads();
    if (!is_last) return;
    __threadfence();
    const float isn_out = rsqrtf(static_cast<float>(d_out));
    const int mq = B * d_out / 4;   // y' gathered as float4, four per thread per step
    for (int q0 = threadIdx.x; q0 < mq; q0 += 4 * blockDim.x) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int q = q0 + u * blockDim.x;
            if (q < mq) v[u] = __ldcg(reinterpret_cast<const float4*>(yp) + q);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int q = q0 + u * blockDim.x;
            if (q < mq) reinterpret_cast<float4*>(xv)[q] = v[u];
        }
    }
    __syncthreads();
    for (int b = 0; b < B; ++b)
        block_rht_inplace(xv + b * d_out, d_out, lg_out, has28_out != 0, F_NONE, F_NONE, sign_u, s_g, isn_out);
    // sigma_U / s_G on the way out (the same vectorized, loads-first pattern)
    const int oq = d_out / 4;
    for (int q0 = threadIdx.x; q0 < oq; q0 += 4 * blockDim.x) {
        float4 f[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int q = q0 + u * blockDim.x;
            if (q < oq) {
                const float4 sc = __ldg(reinterpret_cast<const float4*>(s_g) + q);
                const char4 sg = reinterpret_cast<const char4*>(sign_u)[q];
                f[u] = make_float4(static_cast<float>(sg.x) / sc.x, static_cast<float>(sg.y) / sc.y,
                                   static_cast<float>(sg.z) / sc.z, static_cast<float>(sg.w) / sc.w);
            }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int q = q0 + u * blockDim.x;
            if (q < oq)
                for (int b = 0; b < B; ++b) {
                    const float4 t = reinterpret_cast<const float4*>(xv + b * d_out)[q];
                    reinterpret_cast<float4*>(y + static_cast<int64_t>(b) * d_out)[q] =
                        make_float4(t.x * f[u].x, t.y * f[u].y, t.z * f[u].z, t.w * f[u].w);
                }
        }
    }
}

template <int PB>
kq_status launch_fused(int64_t B, unsigned grid, size_t smem, cudaStream_t st, const uint32_t* packed,
                       const float* scale, const int32_t* zero, int d_out, int d_in, int group, const float* s_x,
                       const float* s_g, const int8_t* su, const int8_t* sv, int lgi, int h28i, int lgo, int h28o,
                       const float* x, float* yp, float* y, unsigned* ticket) {
#define KQ_FUSED_CASE(NB)                                                                                     \
    case NB: {                                                                                               \
        static bool attr = false;                                                                            \
        if (!attr) {                                                                                         \
            KQ_CUDA(cudaFuncSetAttribute(infer_fused_kernel<PB, NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                         210 * 1024));                                                       \
            attr = true;                                                                                     \
        }                                                                                                    \
        infer_fused_kernel<PB, NB><<<grid, 256, smem, st>>>(packed, scale, zero, d_out, d_in, group, s_x, s_g, su, \
                                                          sv, lgi, h28i, lgo, h28o, x, yp, y, ticket);       \
        break;                                                                                               \
    }
    switch (B) {
        KQ_FUSED_CASE(1)
        KQ_FUSED_CASE(2)
        KQ_FUSED_CASE(3)
        KQ_FUSED_CASE(4)
        KQ_FUSED_CASE(5)
        KQ_FUSED_CASE(6)
        KQ_FUSED_CASE(7)
        KQ_FUSED_CASE(8)
        default:
            return KQ_ERR_INVALID_ARG;
    }
#undef KQ_FUSED_CASE
    KQ_LAUNCH_CHECK("infer_fused_kernel");
    return KQ_OK;
}

// n = 28 * 2^k or 2^k: (k, has28); false if neither.
inline bool rht_plan(int64_t n, int* lg, int* h28) {
    int64_t p = n;
    *h28 = 0;
    if (n % 28 == 0) {
        p = n / 28;
        *h28 = 1;
    }
    if (p < 1 || (p & (p - 1))) return false;
    int k = 0;
    while ((int64_t{1} << k) < p) ++k;
    *lg = k;
    return true;
}

template <int PB>
kq_status launch_gemv(int64_t B, dim3 grid, cudaStream_t st, const uint32_t* packed, const float* scale,
                      const int32_t* zero, int64_t d_out, int64_t d_in, int group, const float* x, const float* xs,
                      float* y) {
#define KQ_GEMV_CASE(NB)                                                                                  \
    case NB:                                                                                             \
        dequant_gemv_kernel<PB, NB><<<grid, 256, 0, st>>>(packed, scale, zero, d_out, d_in, group, x, xs, y); \
        break;
    switch (B) {
        KQ_GEMV_CASE(1)
        KQ_GEMV_CASE(2)
        KQ_GEMV_CASE(3)
        KQ_GEMV_CASE(4)
        KQ_GEMV_CASE(5)
        KQ_GEMV_CASE(6)
        KQ_GEMV_CASE(7)
        KQ_GEMV_CASE(8)
        default:
            return KQ_ERR_INVALID_ARG;
    }
#undef KQ_GEMV_CASE
    KQ_LAUNCH_CHECK("dequant_gemv_kernel");
    return KQ_OK;
}

inline size_t al256(size_t b) { return (b + 255) & ~static_cast<size_t>(255); }

}  // namespace
}  // namespace kq

using namespace kq;

extern "C" size_t kq_packed_codes_bytes(int64_t d_out, int64_t d_in, int bits) {
    if (d_out < 1 || d_in < 1 || bits < 1 || bits > 8 || bits == 5 || bits == 6 || bits == 7 || bits == 1) return 0;
    return static_cast<size_t>(d_out) * static_cast<size_t>(d_in) * lane_bits(bits) / 8;
}

extern "C" kq_status kq_pack_codes(const uint8_t* codes, int64_t d_out, int64_t d_in, int bits, uint32_t* packed,
                                   kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!codes || !packed || d_out < 1 || d_in < 1) {
        set_error("kq_pack_codes: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (kq_packed_codes_bytes(d_out, d_in, bits) == 0 || (d_in % 128) != 0 ||
        (reinterpret_cast<uintptr_t>(packed) & 15u)) {
        set_error("kq_pack_codes: bits must be 2, 3, 4 or 8, d_in a multiple of 128, packed 16-byte aligned");
        return KQ_ERR_UNSUPPORTED;
    }
    const int pb = lane_bits(bits);
    const int64_t words = d_out * d_in / (32 / pb);
    const int64_t grid = std::min<int64_t>(cdiv(words, 256), static_cast<int64_t>(num_sms()) * 16);
    pack_kernel<<<static_cast<unsigned>(grid), 256, 0, stream>>>(codes, d_out, d_in, pb, packed);
    KQ_LAUNCH_CHECK("pack_kernel");
    return KQ_OK;
}

extern "C" size_t kq_infer_workspace(int64_t B, int64_t d_in, int64_t d_out) {
    if (B < 1 || d_in < 1 || d_out < 1) return 0;
    return al256(static_cast<size_t>(B) * d_in * sizeof(float)) + al256(static_cast<size_t>(B) * (d_in / 16) * sizeof(float)) +
           al256(static_cast<size_t>(B) * d_out * sizeof(float)) + 256 + 256;
}

extern "C" kq_status kq_infer(const uint32_t* packed, const float* scale, const int32_t* zero, int64_t d_out,
                              int64_t d_in, int bits, int group, const float* s_x, const float* s_g,
                              const int8_t* sign_u, const int8_t* sign_v, const float* x, int64_t B, float* y,
                              void* ws, size_t ws_bytes, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!packed || !scale || !zero || !s_x || !s_g || !sign_u || !sign_v || !x || !y || d_out < 1 || d_in < 1 || B < 1 ||
        B > KQ_INFER_MAX_B) {
        set_error("kq_infer: invalid arguments (B must be 1..%d)", KQ_INFER_MAX_B);
        return KQ_ERR_INVALID_ARG;
    }
    if (kq_packed_codes_bytes(d_out, d_in, bits) == 0 || (d_in % 128) != 0 || (group != 0 && group != 128) ||
        (reinterpret_cast<uintptr_t>(packed) & 15u) || (reinterpret_cast<uintptr_t>(x) & 15u) ||
        (reinterpret_cast<uintptr_t>(s_x) & 15u) || (reinterpret_cast<uintptr_t>(sign_v) & 3u) ||
        (reinterpret_cast<uintptr_t>(s_g) & 15u) || (reinterpret_cast<uintptr_t>(sign_u) & 3u) ||
        (reinterpret_cast<uintptr_t>(y) & 15u) || (d_out % 4) != 0) {
        set_error("kq_infer: bits in {2, 3, 4, 8}, d_in %% 128 == 0, d_out %% 4 == 0, group 0 or 128, 16-byte "
                  "aligned codes, x, y, s_x, s_g, 4-byte aligned signs");
        return KQ_ERR_UNSUPPORTED;
    }
    if (!ws || ws_bytes < kq_infer_workspace(B, d_in, d_out) || (reinterpret_cast<uintptr_t>(ws) & 255u)) {
        set_error("kq_infer: workspace must be 256-byte aligned and hold %zu bytes", kq_infer_workspace(B, d_in, d_out));
        return KQ_ERR_WORKSPACE;
    }
    float* xt = static_cast<float*>(ws);
    float* xs = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + al256(static_cast<size_t>(B) * d_in * sizeof(float)));
    uint8_t* after_xs = reinterpret_cast<uint8_t*>(xs) + al256(static_cast<size_t>(B) * (d_in / 16) * sizeof(float));
    float* yp = reinterpret_cast<float*>(after_xs);
    unsigned* ticket = reinterpret_cast<unsigned*>(after_xs + al256(static_cast<size_t>(B) * d_out * sizeof(float)));
    const int pb = lane_bits(bits);
    int lgi = 0, h28i = 0, lgo = 0, h28o = 0;
    if (!rht_plan(d_in, &lgi, &h28i) || !rht_plan(d_out, &lgo, &h28o)) {
        set_error("kq_infer: d_in=%lld or d_out=%lld has no Hadamard construction", (long long)d_in, (long long)d_out);
        return KQ_ERR_UNSUPPORTED;
    }
    const int ng = group ? static_cast<int>(d_in / group) : 1;
    const size_t fsmem = (static_cast<size_t>(B) * std::max(d_in, d_out) + static_cast<size_t>(B) * ng) * sizeof(float);
    if (fsmem <= 200 * 1024) {
        // persistent grid: three CTAs per SM (the register budget at 84 registers), fewer if
        // shared memory says so
        const int per_sm = static_cast<int>(std::max<size_t>(1, std::min<size_t>(3, (227 * 1024) / (fsmem + 1024))));
        const unsigned grid = static_cast<unsigned>(std::min<int64_t>(cdiv(d_out, 8), static_cast<int64_t>(num_sms()) * per_sm));
        KQ_CUDA(cudaMemsetAsync(ticket, 0, sizeof(unsigned), stream));
        kq_status fs;
        if (pb == 2)
            fs = launch_fused<2>(B, grid, fsmem, stream, packed, scale, zero, static_cast<int>(d_out), static_cast<int>(d_in),
                                 group, s_x, s_g, sign_u, sign_v, lgi, h28i, lgo, h28o, x, yp, y, ticket);
        else if (pb == 4)
            fs = launch_fused<4>(B, grid, fsmem, stream, packed, scale, zero, static_cast<int>(d_out), static_cast<int>(d_in),
                                 group, s_x, s_g, sign_u, sign_v, lgi, h28i, lgo, h28o, x, yp, y, ticket);
        else
            fs = launch_fused<8>(B, grid, fsmem, stream, packed, scale, zero, static_cast<int>(d_out), static_cast<int>(d_in),
                                 group, s_x, s_g, sign_u, sign_v, lgi, h28i, lgo, h28o, x, yp, y, ticket);
        return fs;
    }
    // x' = V S_X^-1 x
    KQ_CUDA(cudaMemcpyAsync(xt, x, static_cast<size_t>(B) * d_in * sizeof(float), cudaMemcpyDeviceToDevice, stream));
    kq_status st = rotate_rows_pre_div(xt, B, d_in, s_x, sign_v, stream);
    if (st != KQ_OK) return st;
    const int64_t runs = B * (d_in / 16);
    runsum16_kernel<<<static_cast<unsigned>(std::max<int64_t>(1, std::min<int64_t>(cdiv(runs, 256), num_sms() * 8))), 256, 0,
                      stream>>>(xt, B, d_in, xs);
    KQ_LAUNCH_CHECK("runsum16_kernel");
    // y' = Q' x'
    const dim3 grid(static_cast<unsigned>(std::min<int64_t>(cdiv(d_out, 8), static_cast<int64_t>(num_sms()) * 16)));
    if (pb == 2) st = launch_gemv<2>(B, grid, stream, packed, scale, zero, d_out, d_in, group, xt, xs, y);
    else if (pb == 4) st = launch_gemv<4>(B, grid, stream, packed, scale, zero, d_out, d_in, group, xt, xs, y);
    else st = launch_gemv<8>(B, grid, stream, packed, scale, zero, d_out, d_in, group, xt, xs, y);
    if (st != KQ_OK) return st;
    // y = S_G^-1 U^T y'
    return rotate_rows_inv(y, B, d_out, s_g, sign_u, stream);
}
