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
// Streamed path (when x' of the B tokens and two ring slots fit in shared memory, and y'
// of one token): two kernels. The first runs one CTA per SM over a contiguous range of rows
// and moves the weights with TMA bulk copies through a ring of shared-memory slots while it
// forms x' = V S_X^-1 x; a code q becomes an exact float by a byte permute that places it
// under the exponent of 2^23 (the float 2^23 + q), and the zero point goes in the same
// subtraction. The second applies y = S_G^-1 U^T y', one CTA per token. Both are launched as
// programmatic dependents, so the next call's weights are on their way into L2 while this
// call finishes. Larger B d: three kernels (row transform, a product reading x' through L1
// with per-16-column sums, row transform).
#include <cooperative_groups.h>

#include "kq_common.cuh"
#include "rht.cuh"

namespace cg = cooperative_groups;

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

// ------------------------------------------------------------------------- streamed path
// y' = Q' x' with the weights streamed through shared memory by TMA bulk copies, then
// y = S_G^-1 U^T y' by a second kernel. Both launch as programmatic dependents of the work
// before them on the stream: a CTA asks L2 for its whole weight slab (codes, scales, zeros)
// before it waits for the preceding kernel (a prefetch hint: L2 is the point of coherence,
// so nothing stale can be read), and touches x, y' and y only after that wait.
constexpr int IS_WARPS = 8;    // warps of the streaming kernel
constexpr int IS_SLOTS = 8;    // most ring slots
constexpr int XREG = 16;       // x' values a thread holds while reordering it
constexpr int XB = 132;        // floats per block of the reordered x' (128 used: 32 lanes x 4)

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ void prefetch_l2(const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(src)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Words a 32-bit word of codes is split into, one code per byte.
template <int PB>
__host__ __device__ constexpr int byte_words() { return PB == 2 ? 4 : (PB == 4 ? 2 : 1); }

// 2^23 + code for the byte k of w (the bits 0x4B0000qq).
__device__ __forceinline__ float byte_raw(uint32_t w, int k) {
    return __int_as_float(static_cast<int>(__byte_perm(w, 0x4B000000u, 0x7440u | static_cast<uint32_t>(k))));
}

// Codes 2j and 2j + 1 of a word as the pair (2^23 + q_2j, 2^23 + q_2j+1); m holds the word
// split into bytes: PB = 8: m[0] = w; PB = 4: m[0] = even codes, m[1] = odd codes; PB = 2:
// m[s] = codes s, s + 4, s + 8, s + 12.
template <int PB>
__device__ __forceinline__ void split_bytes(uint32_t w, uint32_t (&m)[byte_words<PB>()]) {
    if constexpr (PB == 8) {
        m[0] = w;
    } else if constexpr (PB == 4) {
        m[0] = w & 0x0F0F0F0Fu;
        m[1] = (w >> 4) & 0x0F0F0F0Fu;
    } else {
#pragma unroll
        for (int s = 0; s < 4; ++s) m[s] = (w >> (2 * s)) & 0x03030303u;
    }
}
template <int PB>
__device__ __forceinline__ float2 raw_pair(const uint32_t (&m)[byte_words<PB>()], int j) {
    constexpr int NS = byte_words<PB>();
    const int c0 = 2 * j, c1 = 2 * j + 1;
    return make_float2(byte_raw(m[c0 % NS], c0 / NS), byte_raw(m[c1 % NS], c1 / NS));
}

// One CTA per SM; CTA c owns the rows of quads [c Q / grid, (c + 1) Q / grid) (a quad = 4
// rows, so every slab of scales and zeros starts on 16 bytes). Its rows pass through a ring
// of nslot shared-memory slots, qps quads per stage; a slot holds the stage's codes, scales
// and zeros, loaded by one mbarrier-tracked bulk copy each. A unit of work is one quad and
// one lane step: lane l covers the 16-byte chunk 32 s + l of each of the quad's rows (32 / PB
// codes a word, 4 words; a chunk lies inside one group of 128 columns), with x' of the chunk
// loaded once for the four rows. Units are dealt to the warps round-robin across stages.
// A code q and its zero z become (2^23 + q) - (2^23 + z) = q - z exactly (pairs of codes
// with the packed f32x2 add), so
//   y'_r = sum_chunks scale_rg sum_{c in chunk} (q_rc - z_rg) x'_c,
// the products summed in pairs by f32x2 fma. Lane sums of a unit are reduced in the warp and
// parked per (row, step); the warp that finishes a stage last adds them up in step order,
// writes the stage's rows of y' and refills the slot with the stage nslot ahead.
// CTAs per SM of the streaming kernel: two for one token (at most 128 registers a thread).
__host__ __device__ constexpr int stream_ctas_per_sm(int B) { return B == 1 ? 2 : 1; }

template <int PB, int B>
__global__ void __launch_bounds__(IS_WARPS * 32, stream_ctas_per_sm(B)) infer_stream_kernel(
    const uint32_t* __restrict__ packed, const float* __restrict__ scale, const int32_t* __restrict__ zero, int d_out,
    int d_in, int ng, int grouped, const float* __restrict__ s_x, const int8_t* __restrict__ sign_v, int lg_in,
    int has28_in, const float* __restrict__ x, float* __restrict__ yp, int qps, int nslot, int part_slot,
    int slot_bytes, int xp, int* info) {
    extern __shared__ __align__(128) uint8_t ism[];
    __shared__ uint64_t full[IS_SLOTS];
    __shared__ int done[IS_SLOTS];
    __shared__ int abort_flag;
    __shared__ int issued_hi;   // stages whose copies have been issued: [0, issued_hi)
    constexpr int CPW = 32 / PB;   // codes per word
    constexpr int CPC = 4 * CPW;   // codes per 16-byte chunk
    constexpr int NS = byte_words<PB>();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rowbytes = d_in / 8 * PB;
    const int CH = rowbytes / 16;         // chunks per row
    const int S = (CH + 31) / 32;         // lane steps per row
    const int Q = d_out / 4;
    const int qa = static_cast<int>(static_cast<int64_t>(blockIdx.x) * Q / gridDim.x);
    const int qb = static_cast<int>(static_cast<int64_t>(blockIdx.x + 1) * Q / gridDim.x);
    const int nst = (qb - qa + qps - 1) / qps;
    const int codes_bytes = qps * 4 * rowbytes;
    const int sc_bytes = qps * 4 * ng * 4;
    const bool reg12 = d_in == 4096;   // x' transform in registers (16 values per thread)
    float* xv = reinterpret_cast<float*>(ism);                                    // B x xp
    float* xbuf = xv + static_cast<int64_t>(B) * xp;                              // 4096 + 128 (reg12)
    float* part = xbuf + (reg12 ? 4096 + 128 : 0);                                // nslot x part_slot
    uint8_t* slots = reinterpret_cast<uint8_t*>(part + static_cast<int64_t>(nslot) * part_slot);
    const uint8_t* pk = reinterpret_cast<const uint8_t*>(packed);

    if (threadIdx.x == 0) {
        for (int k = 0; k < nslot; ++k) mbar_init(&full[k], 1);
        fence_mbar_init();
        abort_flag = 0;
        issued_hi = 0;
    }
    if (threadIdx.x < IS_SLOTS) done[threadIdx.x] = 0;
    // the weights do not depend on the preceding kernel: ask L2 for them now
    if (threadIdx.x == 0 && qb > qa) {
        const int64_t r0 = static_cast<int64_t>(qa) * 4, nr = static_cast<int64_t>(qb - qa) * 4;
        prefetch_l2(pk + r0 * rowbytes, static_cast<uint32_t>(nr * rowbytes));
        prefetch_l2(scale + r0 * ng, static_cast<uint32_t>(nr * ng * 4));
        prefetch_l2(zero + r0 * ng, static_cast<uint32_t>(nr * ng * 4));
    }
    // sign / s of V S_X^-1 (= sign RN(1 / s) exactly) does not depend on the preceding kernel
    // either: thread t's 16 contiguous elements in registers (reg12), else the whole vector in
    // token 0's x' buffer
    float fx[16];
    if (reg12) {
        const float4* s4 = reinterpret_cast<const float4*>(s_x) + 4 * threadIdx.x;
        const char4* g4 = reinterpret_cast<const char4*>(sign_v) + 4 * threadIdx.x;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float4 sc = __ldg(s4 + q);
            const char4 sg = g4[q];
            fx[4 * q] = sg.x < 0 ? -__frcp_rn(sc.x) : __frcp_rn(sc.x);
            fx[4 * q + 1] = sg.y < 0 ? -__frcp_rn(sc.y) : __frcp_rn(sc.y);
            fx[4 * q + 2] = sg.z < 0 ? -__frcp_rn(sc.z) : __frcp_rn(sc.z);
            fx[4 * q + 3] = sg.w < 0 ? -__frcp_rn(sc.w) : __frcp_rn(sc.w);
        }
    } else {
        for (int j = threadIdx.x; j < d_in; j += blockDim.x) {
            const float r = __frcp_rn(__ldg(s_x + j));
            xv[j] = sign_v[j] < 0 ? -r : r;
        }
    }
    pdl_launch_dependents();
    pdl_wait();
    __syncthreads();
    auto issue = [&](int t) {
        const int k = t % nslot;
        const int q0 = qa + t * qps, nq = min(qps, qb - q0);
        const int64_t r0 = static_cast<int64_t>(q0) * 4;
        const uint32_t cb = static_cast<uint32_t>(nq * 4 * rowbytes), sb = static_cast<uint32_t>(nq * 4 * ng * 4);
        uint8_t* dst = slots + static_cast<int64_t>(k) * slot_bytes;
        atomicMax(&issued_hi, t + 1);
        mbar_arrive_expect_tx(&full[k], cb + 2 * sb);
        bulk_g2s(dst, pk + r0 * rowbytes, cb, &full[k]);
        bulk_g2s(dst + codes_bytes, scale + r0 * ng, sb, &full[k]);
        bulk_g2s(dst + codes_bytes + sc_bytes, zero + r0 * ng, sb, &full[k]);
    };
    if (threadIdx.x == 0)
        for (int t = 0; t < min(nslot, nst); ++t) issue(t);
    // x' = V S_X^-1 x per token, while the first stages land, stored reordered for the
    // product: for lane step s, word kw and quadruple v of the chunk, the 32 lanes' four floats
    // are consecutive (conflict-free 16-byte loads; in natural order the lanes' chunks are CPC
    // floats apart), blocks of 128 floats XB apart.
    auto xpos = [&](int col) {
        const int c = col / CPC, w = col - c * CPC;
        const int kw = w / CPW, v = (w - kw * CPW) >> 2;
        return (((c >> 5) * 4 + kw) * (CPW / 4) + v) * XB + (c & 31) * 4 + (col & 3);
    };
    const float isn_in = rsqrtf(static_cast<float>(d_in));
    if (reg12) {
        // Walsh-Hadamard transform of 4096 values, 16 per thread: the thread's 16 contiguous
        // values, then two transpositions through shared memory; the last phase holds
        // element j = t | k << 8 and writes it straight to its reordered place.
        const int t = threadIdx.x;
        for (int b = 0; b < B; ++b) {
            float xr[16];
            // x may come from the kernel this one overlapped: read it through L2
            const float4* xs4 = reinterpret_cast<const float4*>(x + static_cast<int64_t>(b) * d_in) + 4 * t;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float4 v = __ldcg(xs4 + q);
                xr[4 * q] = v.x * fx[4 * q];
                xr[4 * q + 1] = v.y * fx[4 * q + 1];
                xr[4 * q + 2] = v.z * fx[4 * q + 2];
                xr[4 * q + 3] = v.w * fx[4 * q + 3];
            }
            fwht_kbits<0xFu>(xr);
            rr_transpose<12, 1>(xr, xbuf, t);
            rr_transpose<12, 2>(xr, xbuf, t);
#pragma unroll
            for (int k = 0; k < 16; ++k) xv[b * xp + xpos(t | (k << 8))] = xr[k] * isn_in;
        }
        __syncthreads();
    } else {
        const int nq4 = d_in / 4;
        for (int b = B - 1; b >= 0; --b) {   // token 0 last: its buffer holds the factors
            for (int q0 = threadIdx.x; q0 < nq4; q0 += 4 * blockDim.x) {
                float4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int q = q0 + u * blockDim.x;
                    if (q < nq4) v[u] = __ldcg(reinterpret_cast<const float4*>(x + static_cast<int64_t>(b) * d_in) + q);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int q = q0 + u * blockDim.x;
                    if (q < nq4) {
                        const float4 f = reinterpret_cast<const float4*>(xv)[q];
                        reinterpret_cast<float4*>(xv + b * xp)[q] =
                            make_float4(v[u].x * f.x, v[u].y * f.y, v[u].z * f.z, v[u].w * f.w);
                    }
                }
            }
        }
        __syncthreads();
        // transform in natural order, then reorder in place through registers, XREG values a
        // thread per round; a round's places lie at or above its own columns and below the
        // places of the rounds after it, so the rounds go from the last one down
        for (int b = 0; b < B; ++b) {
            float* xb = xv + b * xp;
            block_rht_inplace(xb, d_in, lg_in, has28_in != 0, F_NONE, F_NONE, sign_v, s_x, isn_in);
            const int R = XREG * IS_WARPS * 32;
            for (int base = (d_in - 1) / R * R; base >= 0; base -= R) {
                float tv[XREG];
#pragma unroll
                for (int i = 0; i < XREG; ++i) {
                    const int col = base + i * IS_WARPS * 32 + static_cast<int>(threadIdx.x);
                    if (col < d_in) tv[i] = xb[col];
                }
                __syncthreads();
#pragma unroll
                for (int i = 0; i < XREG; ++i) {
                    const int col = base + i * IS_WARPS * 32 + static_cast<int>(threadIdx.x);
                    if (col < d_in) xb[xpos(col)] = tv[i];
                }
                __syncthreads();
            }
        }
    }

    int ubase = 0;   // units of the stages before this one (round-robin over warps)
    for (int t = 0; t < nst; ++t) {
        const int k = t % nslot;
        const int q0 = qa + t * qps, nq = min(qps, qb - q0);
        const int units = nq * S;
        if (!mbar_wait(&full[k], static_cast<uint32_t>((t / nslot) & 1), &abort_flag)) break;
        const uint8_t* sl = slots + static_cast<int64_t>(k) * slot_bytes;
        const float* ss = reinterpret_cast<const float*>(sl + codes_bytes);
        const int32_t* zz = reinterpret_cast<const int32_t*>(sl + codes_bytes + sc_bytes);
        float* pp = part + static_cast<int64_t>(k) * part_slot;
        for (int u = ((warp - ubase) % IS_WARPS + IS_WARPS) % IS_WARPS; u < units; u += IS_WARPS) {
            const int ql = u / S, s = u - ql * S;
            const int c = s * 32 + lane;
            float2 dot[4][B];
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int b = 0; b < B; ++b) dot[r][b] = make_float2(0.0f, 0.0f);
            float scl[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            if (c < CH) {
                const int col0 = c * CPC;
                const int g = grouped ? (col0 >> 7) : 0;
                uint4 wv[4];
                float2 zo[4];
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const int rl = ql * 4 + r;
                    wv[r] = *reinterpret_cast<const uint4*>(sl + static_cast<int64_t>(rl) * rowbytes + c * 16);
                    scl[r] = ss[rl * ng + g];
                    const float z = 8388608.0f + static_cast<float>(zz[rl * ng + g]);
                    zo[r] = make_float2(-z, -z);
                }
#pragma unroll
                for (int kw = 0; kw < 4; ++kw) {
                    const int xo = ((s * 4 + kw) * (CPW / 4)) * XB + lane * 4;   // reordered x' of word kw
                    if constexpr (B * CPW <= 32) {
                        float2 xk[B][CPW / 2];
#pragma unroll
                        for (int b = 0; b < B; ++b)
#pragma unroll
                            for (int v = 0; v < CPW / 4; ++v) {
                                const float4 t4 = *reinterpret_cast<const float4*>(xv + b * xp + xo + XB * v);
                                xk[b][2 * v] = make_float2(t4.x, t4.y);
                                xk[b][2 * v + 1] = make_float2(t4.z, t4.w);
                            }
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            const uint32_t wd = kw == 0 ? wv[r].x : kw == 1 ? wv[r].y : kw == 2 ? wv[r].z : wv[r].w;
                            uint32_t m[NS];
                            split_bytes<PB>(wd, m);
#pragma unroll
                            for (int j = 0; j < CPW / 2; ++j) {
                                const float2 q2 = __fadd2_rn(raw_pair<PB>(m, j), zo[r]);
#pragma unroll
                                for (int b = 0; b < B; ++b) dot[r][b] = __ffma2_rn(q2, xk[b][j], dot[r][b]);
                            }
                        }
                    } else {
#pragma unroll
                        for (int b = 0; b < B; ++b) {
                            float2 xk[CPW / 2];
#pragma unroll
                            for (int v = 0; v < CPW / 4; ++v) {
                                const float4 t4 = *reinterpret_cast<const float4*>(xv + b * xp + xo + XB * v);
                                xk[2 * v] = make_float2(t4.x, t4.y);
                                xk[2 * v + 1] = make_float2(t4.z, t4.w);
                            }
#pragma unroll
                            for (int r = 0; r < 4; ++r) {
                                const uint32_t wd = kw == 0 ? wv[r].x : kw == 1 ? wv[r].y : kw == 2 ? wv[r].z : wv[r].w;
                                uint32_t m[NS];
                                split_bytes<PB>(wd, m);
#pragma unroll
                                for (int j = 0; j < CPW / 2; ++j)
                                    dot[r][b] = __ffma2_rn(__fadd2_rn(raw_pair<PB>(m, j), zo[r]), xk[j], dot[r][b]);
                            }
                        }
                    }
                }
            }
            // scale the chunk, reduce over the lanes, park per (row, step)
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    float v = scl[r] * (dot[r][b].x + dot[r][b].y);
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                    if (lane == 0) pp[((ql * 4 + r) * S + s) * B + b] = v;
                }
        }
        ubase += units;
        // the last warp through the stage writes its rows of y' and refills the slot
        __syncwarp();
        int last = 0;
        if (lane == 0) {
            __threadfence_block();
            last = atomicAdd(&done[k], 1) == (t / nslot + 1) * IS_WARPS - 1;
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        if (last) {
            __threadfence_block();
            for (int e = lane; e < nq * 4 * B; e += 32) {
                const int rl = e / B, b = e - rl * B;
                float a = 0.0f;
                for (int s2 = 0; s2 < S; ++s2) a += pp[(rl * S + s2) * B + b];
                if (KQ_IN_RANGE(static_cast<int64_t>(b) * d_out + static_cast<int64_t>(q0) * 4 + rl,
                                static_cast<int64_t>(B) * d_out))
                    yp[static_cast<int64_t>(b) * d_out + static_cast<int64_t>(q0) * 4 + rl] = a;
            }
            __syncwarp();
            if (lane == 0 && t + nslot < nst) {
                fence_proxy_async_smem();
                issue(t + nslot);
            }
        }
    }
    // A wait that gave up (the copies never landed): report KQ_ERR_TIMEOUT in the device
    // error word, give the latest stage issued into each slot one more bounded wait, so that
    // no copy still in flight lands in shared memory after the CTA has exited, and leave y'
    // as NaN for this CTA's rows.
    __syncthreads();
    if (abort_flag) {
        if (threadIdx.x == 0) {
            record_error(info, -KQ_ERR_TIMEOUT);
            for (int t = max(0, issued_hi - nslot); t < issued_hi; ++t) {
                int quiet = 0;
                mbar_wait(&full[t % nslot], static_cast<uint32_t>((t / nslot) & 1), &quiet);
            }
        }
        for (int e = threadIdx.x; e < (qb - qa) * 4 * B; e += blockDim.x) {
            const int rl = e / B, b = e - rl * B;
            yp[static_cast<int64_t>(b) * d_out + static_cast<int64_t>(qa) * 4 + rl] = __int_as_float(0x7fc00000);
        }
    }
}

// y = S_G^-1 U^T y' by one cluster of NC CTAs per token, CTA c holding the slice
// [c L, c L + L) of y' (L = n / NC). With T = H_A (x) H_P (index a P + b, b fastest): for
// n = 2^k, NC = 8 CTAs (A = 8, P = L) or one CTA for n < 64; for n = 28 P, NC = 7 CTAs of four
// length-P pieces each (A = 28). Each CTA applies H_P to its pieces in shared memory; after a
// cluster barrier, column b of the A x P array is gathered from the CTAs' shared memory
// (distributed shared memory), mixed by H_A, scaled by sigma_U / s_G / sqrt(n) and written.
template <int NC>
__global__ void __launch_bounds__(256) infer_out_kernel(const float* __restrict__ yp, int d_out, int lg_p,
                                                        const float* __restrict__ s_g,
                                                        const int8_t* __restrict__ sign_u, float* __restrict__ y) {
    extern __shared__ __align__(16) float ov[];
    constexpr int A = NC == 7 ? 28 : NC;    // rows of the A x P array
    constexpr int PER = A / NC;              // rows a CTA holds
    const int P = 1 << lg_p;
    const int L = PER * P;
    cg::cluster_group cl = cg::this_cluster();
    const int rank = NC > 1 ? static_cast<int>(cl.block_rank()) : 0;
    const int64_t b = blockIdx.x / NC;
    pdl_launch_dependents();
    pdl_wait();
    const float* src = yp + b * d_out + static_cast<int64_t>(rank) * L;
    if ((L & 3) == 0) {
        for (int q = threadIdx.x; q < L / 4; q += blockDim.x)
            reinterpret_cast<float4*>(ov)[q] = __ldcg(reinterpret_cast<const float4*>(src) + q);
    } else {
        for (int q = threadIdx.x; q < L; q += blockDim.x) ov[q] = __ldcg(src + q);
    }
    __syncthreads();
    block_rht_inplace(ov, L, lg_p, false, F_NONE, F_NONE, sign_u, s_g, 1.0f);
    if constexpr (NC > 1) cl.sync();
    const float isn = rsqrtf(static_cast<float>(d_out));
    // columns [c0, c1) of this CTA; for A = 28 two threads share a column, 14 rows each
    constexpr int SPLIT = A == 28 ? 2 : 1;
    constexpr int RA = A / SPLIT;
    const int per_cta = (P + NC - 1) / NC;
    const int c0 = rank * per_cta, c1 = min(P, c0 + per_cta);
    float* yb = y + b * d_out;
    for (int task = threadIdx.x; task < (c1 - c0) * SPLIT; task += blockDim.x) {
        const int col = c0 + task / SPLIT, a0 = (task % SPLIT) * RA;
        // sigma_U / s_G of this thread's outputs first (sign / s = sign RN(1 / s) exactly)
        float f[RA];
#pragma unroll
        for (int q = 0; q < RA; ++q) {
            const int64_t j = static_cast<int64_t>(a0 + q) * P + col;
            const float r = __frcp_rn(__ldg(s_g + j));
            f[q] = sign_u[j] < 0 ? -r : r;
        }
        float xa[A];
#pragma unroll
        for (int c = 0; c < NC; ++c) {
            const float* rv = NC > 1 ? cl.map_shared_rank(ov, c) : ov;
#pragma unroll
            for (int q = 0; q < PER; ++q) xa[c * PER + q] = rv[q * P + col];
        }
        auto put = [&](int a, float v) { yb[static_cast<int64_t>(a) * P + col] = v * isn * f[a - a0]; };
        if constexpr (A == 28) {
            if (a0 == 0) mix28_rows_at<0>(xa, put, std::make_integer_sequence<int, 14>{});
            else mix28_rows_at<14>(xa, put, std::make_integer_sequence<int, 14>{});
        } else {
            float x8[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) x8[q] = q < A ? xa[q] : 0.0f;
            if constexpr (A == 8) fwht_reg<8>(x8);
#pragma unroll
            for (int q = 0; q < A; ++q) put(q, x8[q]);
        }
    }
    if constexpr (NC > 1) cl.sync();   // keep this CTA's slice alive until every CTA has read it
}

// y = S_G^-1 U^T y' for one token per CTA with the transform in registers (16 values a
// thread): n = 2^LG (n / 16 threads) or, when H28, n = 28 P with P = 2^LG (28 rows of P / 16
// threads each, one row's Walsh-Hadamard transform per group; then the 28-point mix of every
// column from shared memory, two threads a column with 14 rows each). The factors
// sigma_U / s_G of each thread's outputs are loaded before the wait for the preceding kernel.
template <int LG, bool H28>
__global__ void __launch_bounds__((H28 ? 28 : 1) * (1 << LG) / 16) infer_out_reg_kernel(
    const float* __restrict__ yp, int d_out, const float* __restrict__ s_g, const int8_t* __restrict__ sign_u,
    float* __restrict__ y) {
    constexpr int P = 1 << LG, TR = P / 16, NPH = rr_phases(LG);
    constexpr uint32_t ML = rr_mask(LG, NPH - 1);
    constexpr int NT = (H28 ? 28 : 1) * TR;
    constexpr int NF = H28 ? 28 : 16;   // factors a thread holds
    extern __shared__ __align__(16) float osm[];
    const int tid = threadIdx.x, row = tid / TR, t = tid - row * TR;
    const int tl = deposit_bits<((1u << LG) - 1u) & ~ML>(t);
    float f[NF];
    auto fac = [&](int64_t j) {
        const float r = __frcp_rn(__ldg(s_g + j));
        return sign_u[j] < 0 ? -r : r;
    };
    if constexpr (H28) {
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int task = tid + u * NT, col = task >> 1, a0 = (task & 1) * 14;
#pragma unroll
            for (int q = 0; q < 14; ++q) f[u * 14 + q] = task < 2 * P ? fac(static_cast<int64_t>(a0 + q) * P + col) : 0.0f;
        }
    } else {
#pragma unroll
        for (int k = 0; k < 16; ++k) f[k] = fac(tl | deposit_bits<ML>(k));
    }
    pdl_launch_dependents();
    pdl_wait();
    const float isn = rsqrtf(static_cast<float>(d_out));
    const int64_t b = blockIdx.x;
    float xr[16];
    const float4* src = reinterpret_cast<const float4*>(yp + b * d_out + row * P + 16 * t);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const float4 v = __ldcg(src + q);
        xr[4 * q] = v.x;
        xr[4 * q + 1] = v.y;
        xr[4 * q + 2] = v.z;
        xr[4 * q + 3] = v.w;
    }
    float* buf = osm + row * (P + P / 32);
    fwht_kbits<0xFu>(xr);
    rr_transpose<LG, 1>(xr, buf, t);
    if constexpr (NPH > 2) rr_transpose<LG, 2>(xr, buf, t);
    if constexpr (NPH > 3) rr_transpose<LG, 3>(xr, buf, t);
    float* yb = y + b * d_out;
    if constexpr (!H28) {
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const int j = tl | deposit_bits<ML>(k);
            yb[j] = xr[k] * isn * f[k];
        }
    } else {
        __syncthreads();   // every row's transposition buffer has been read
#pragma unroll
        for (int k = 0; k < 16; ++k) osm[row * P + (tl | deposit_bits<ML>(k))] = xr[k];
        __syncthreads();
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int task = tid + u * NT, col = task >> 1, a0 = (task & 1) * 14;
            if (task < 2 * P) {
                float xa[28];
#pragma unroll
                for (int a = 0; a < 28; ++a) xa[a] = osm[a * P + col];
                auto put = [&](int a, float v) { yb[static_cast<int64_t>(a) * P + col] = v * isn * f[u * 14 + a - a0]; };
                if (a0 == 0) mix28_rows_at<0>(xa, put, std::make_integer_sequence<int, 14>{});
                else mix28_rows_at<14>(xa, put, std::make_integer_sequence<int, 14>{});
            }
        }
    }
}

// Launch as a programmatic dependent of the preceding work on the stream, in clusters of
// `cluster` CTAs when cluster > 1.
template <typename... Params, typename... Args>
cudaError_t launch_dependent(void (*kern)(Params...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                             unsigned cluster, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = cluster;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = cluster > 1 ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<Params>(args)...);
}

// Shared-memory plan of the streaming kernel: x' (B d_in floats), then per slot the parked
// lane sums (qps 4 S B floats, rounded to 16 bytes) and the stage's codes, scales and zeros.
struct StreamPlan {
    int grid, qps, nslot, part_slot, slot_bytes, xp;
    size_t smem;
};
constexpr size_t kStreamSmemMax = 226 * 1024;

// Two CTAs per SM when the kernel allows it and two ring slots fit in half the shared
// memory, else one CTA per SM.
inline bool stream_plan_at(int64_t B, int64_t d_out, int64_t d_in, int pb, int64_t ng, int per_sm, StreamPlan* p) {
    const int64_t rowbytes = d_in / 8 * pb;
    const int64_t quad = 4 * rowbytes + 2 * 4 * ng * 4;
    const int64_t Q = d_out / 4;
    const int64_t smem_max = per_sm == 1 ? static_cast<int64_t>(kStreamSmemMax) : 112 * 1024;
    const int grid = static_cast<int>(std::min<int64_t>(Q, static_cast<int64_t>(num_sms()) * per_sm));
    const int64_t qmax = cdiv(Q, grid);
    const int64_t S = cdiv(rowbytes / 16, 32);
    const int64_t xp = S * (32 / pb) * XB;   // reordered x' per token (whole lane steps)
    const int64_t xbytes = B * xp * 4 + (d_in == 4096 ? (4096 + 128) * 4 : 0);
    int64_t qps = std::max<int64_t>(1, std::min<int64_t>(qmax, (24 * 1024) / quad));
    for (; qps >= 1; --qps) {
        const int64_t part = (qps * 4 * S * B + 3) / 4 * 4;
        const int64_t per_slot = qps * quad + part * 4;
        const int64_t stages = cdiv(qmax, qps);
        const int64_t room = (smem_max - xbytes) / per_slot;
        const int64_t ns = std::min(std::min(static_cast<int64_t>(IS_SLOTS), stages), room);
        if (ns >= 2 || (ns == 1 && stages == 1)) {
            *p = StreamPlan{grid, static_cast<int>(qps), static_cast<int>(ns), static_cast<int>(part),
                            static_cast<int>(qps * quad), static_cast<int>(xp),
                            static_cast<size_t>(xbytes + ns * per_slot)};
            return true;
        }
    }
    return false;
}
inline bool stream_plan(int64_t B, int64_t d_out, int64_t d_in, int pb, int64_t ng, StreamPlan* p) {
    const int per_sm = stream_ctas_per_sm(static_cast<int>(B));
    return (per_sm > 1 && stream_plan_at(B, d_out, d_in, pb, ng, per_sm, p)) ||
           stream_plan_at(B, d_out, d_in, pb, ng, 1, p);
}

// y = S_G^-1 U^T y' for B tokens: in registers for n = 2^k (9 <= k <= 14) and n = 28 * 512,
// else infer_out_kernel (n = 28 P: clusters of 7, n = 2^k >= 64: clusters of 8, smaller: one
// CTA).
template <int LG, bool H28>
kq_status launch_out_reg(int64_t B, cudaStream_t st, const float* yp, int d_out, const float* s_g, const int8_t* su,
                         float* y) {
    constexpr int P = 1 << LG, NT = (H28 ? 28 : 1) * P / 16;
    const size_t smem = static_cast<size_t>(H28 ? 28 : 1) * (P + P / 32) * sizeof(float);
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(infer_out_reg_kernel<LG, H28>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(smem)));
        return KQ_OK;
    }));
    KQ_CUDA(launch_dependent(infer_out_reg_kernel<LG, H28>, dim3(static_cast<unsigned>(B)), dim3(NT), smem, st, 1u, yp,
                             d_out, s_g, su, y));
    KQ_LAUNCH_CHECK("infer_out_reg_kernel");
    return KQ_OK;
}

inline kq_status launch_out(int64_t B, cudaStream_t st, const float* yp, int d_out, const float* s_g, const int8_t* su,
                            int lgo, int h28o, float* y) {
    if (h28o && lgo == 9) return launch_out_reg<9, true>(B, st, yp, d_out, s_g, su, y);
    if (!h28o) {
        switch (lgo) {
            case 9: return launch_out_reg<9, false>(B, st, yp, d_out, s_g, su, y);
            case 10: return launch_out_reg<10, false>(B, st, yp, d_out, s_g, su, y);
            case 11: return launch_out_reg<11, false>(B, st, yp, d_out, s_g, su, y);
            case 12: return launch_out_reg<12, false>(B, st, yp, d_out, s_g, su, y);
            case 13: return launch_out_reg<13, false>(B, st, yp, d_out, s_g, su, y);
            case 14: return launch_out_reg<14, false>(B, st, yp, d_out, s_g, su, y);
            default: break;
        }
    }
    if (h28o) {
        KQ_CUDA(launch_dependent(infer_out_kernel<7>, dim3(static_cast<unsigned>(7 * B)), dim3(256),
                                 static_cast<size_t>(4) * (size_t{1} << lgo) * sizeof(float), st, 7u, yp, d_out, lgo, s_g,
                                 su, y));
    } else if (d_out >= 64) {
        KQ_CUDA(launch_dependent(infer_out_kernel<8>, dim3(static_cast<unsigned>(8 * B)), dim3(256),
                                 (size_t{1} << (lgo - 3)) * sizeof(float), st, 8u, yp, d_out, lgo - 3, s_g, su, y));
    } else {
        KQ_CUDA(launch_dependent(infer_out_kernel<1>, dim3(static_cast<unsigned>(B)), dim3(256),
                                 static_cast<size_t>(d_out) * sizeof(float), st, 1u, yp, d_out, lgo, s_g, su, y));
    }
    KQ_LAUNCH_CHECK("infer_out_kernel");
    return KQ_OK;
}

template <int PB, int B>
kq_status launch_stream_b(const StreamPlan& sp, cudaStream_t st, const uint32_t* packed, const float* scale,
                          const int32_t* zero, int d_out, int d_in, int ng, int grouped, const float* s_x,
                          const float* s_g, const int8_t* su, const int8_t* sv, int lgi, int h28i, int lgo, int h28o,
                          const float* x, float* yp, float* y, int* info) {
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(infer_stream_kernel<PB, B>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(kStreamSmemMax)));
        return KQ_OK;
    }));
    KQ_CUDA(launch_dependent(infer_stream_kernel<PB, B>, dim3(sp.grid), dim3(IS_WARPS * 32), sp.smem, st, 1u, packed, scale,
                             zero, d_out, d_in, ng, grouped, s_x, sv, lgi, h28i, x, yp, sp.qps, sp.nslot, sp.part_slot,
                             sp.slot_bytes, sp.xp, info));
    KQ_LAUNCH_CHECK("infer_stream_kernel");
    return launch_out(B, st, yp, d_out, s_g, su, lgo, h28o, y);
}

template <int PB>
kq_status launch_stream(int64_t B, const StreamPlan& sp, cudaStream_t st, const uint32_t* packed, const float* scale,
                        const int32_t* zero, int d_out, int d_in, int ng, int grouped, const float* s_x,
                        const float* s_g, const int8_t* su, const int8_t* sv, int lgi, int h28i, int lgo, int h28o,
                        const float* x, float* yp, float* y, int* info) {
#define KQ_STREAM_CASE(NB) \
    case NB:               \
        return launch_stream_b<PB, NB>(sp, st, packed, scale, zero, d_out, d_in, ng, grouped, s_x, s_g, su, sv, lgi, h28i, lgo, h28o, x, yp, y, info);
    switch (B) {
        KQ_STREAM_CASE(1)
        KQ_STREAM_CASE(2)
        KQ_STREAM_CASE(3)
        KQ_STREAM_CASE(4)
        KQ_STREAM_CASE(5)
        KQ_STREAM_CASE(6)
        KQ_STREAM_CASE(7)
        KQ_STREAM_CASE(8)
        default:
            return KQ_ERR_INVALID_ARG;
    }
#undef KQ_STREAM_CASE
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

KQ_DEBUG_UNIT(infer)
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
                              int* info, void* ws, size_t ws_bytes, kq_stream_t stream_) {
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
    const int pb = lane_bits(bits);
    int lgi = 0, h28i = 0, lgo = 0, h28o = 0;
    if (!rht_plan(d_in, &lgi, &h28i) || !rht_plan(d_out, &lgo, &h28o)) {
        set_error("kq_infer: d_in=%lld or d_out=%lld has no Hadamard construction", (long long)d_in, (long long)d_out);
        return KQ_ERR_UNSUPPORTED;
    }
    const int ng = group ? static_cast<int>(d_in / group) : 1;
    StreamPlan sp;
    if ((reinterpret_cast<uintptr_t>(scale) & 15u) == 0 && (reinterpret_cast<uintptr_t>(zero) & 15u) == 0 &&
        d_out <= 65536 && stream_plan(B, d_out, d_in, pb, ng, &sp)) {
        const int di = static_cast<int>(d_in), dn = static_cast<int>(d_out), gr = group ? 1 : 0;
        if (pb == 2)
            return launch_stream<2>(B, sp, stream, packed, scale, zero, dn, di, ng, gr, s_x, s_g, sign_u, sign_v, lgi, h28i,
                                    lgo, h28o, x, yp, y, info);
        if (pb == 4)
            return launch_stream<4>(B, sp, stream, packed, scale, zero, dn, di, ng, gr, s_x, s_g, sign_u, sign_v, lgi, h28i,
                                    lgo, h28o, x, yp, y, info);
        return launch_stream<8>(B, sp, stream, packed, scale, zero, dn, di, ng, gr, s_x, s_g, sign_u, sign_v, lgi, h28i,
                                lgo, h28o, x, yp, y, info);
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
