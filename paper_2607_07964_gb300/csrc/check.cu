// Check-only calls: Algorithm 2's revert (dequantize, undo U, V, S_G, S_X) and the
// Kronecker-factored proxy loss of Sec. 3.1 Eq. (kron_obj), tr(H_G dW H_X dW^T). They are
// used to compare the whole pipeline against the oracle, not in the timed path.
#include "kq_common.cuh"

namespace kq {
kq_status rotate_rows_inv(float* M, int64_t rows, int64_t n, const float* s, const int8_t* sign,
                          cudaStream_t stream);
kq_status rotate_cols_inv(float* M, int64_t n, int64_t ncols, const float* s, const int8_t* sign,
                          cudaStream_t stream);

namespace {

__global__ void dequant_kernel(const uint8_t* __restrict__ codes, const float* __restrict__ scale,
                               const int32_t* __restrict__ zero, int64_t d_out, int64_t d_in, int group,
                               float* __restrict__ out) {
    const int64_t total = d_out * d_in;
    const int64_t ng = group ? (d_in + group - 1) / group : 1;
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t r = e / d_in, c = e % d_in;
        const int64_t g = r * ng + (group ? c / group : 0);
        out[e] = __fmul_rn(scale[g], static_cast<float>(static_cast<int32_t>(codes[e]) - zero[g]));
    }
}

__global__ void sub_kernel(const float* __restrict__ a, const float* __restrict__ b, int64_t n,
                           float* __restrict__ out) {
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x)
        out[e] = a[e] - b[e];
}

// C [M x N] = A [M x K] B [K x N], row-major fp32. 64 x 64 tiles, 16 x 16 threads, 4 x 4 each.
__global__ void __launch_bounds__(256) gemm_nn_kernel(const float* __restrict__ A, const float* __restrict__ B,
                                                      float* __restrict__ C, int64_t M, int64_t N, int64_t K) {
    __shared__ float as[16][65];
    __shared__ float bs[16][65];
    const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
    const int64_t m0 = static_cast<int64_t>(blockIdx.y) * 64, n0 = static_cast<int64_t>(blockIdx.x) * 64;
    float acc[4][4] = {};
    for (int64_t k0 = 0; k0 < K; k0 += 16) {
        for (int e = threadIdx.x; e < 16 * 64; e += 256) {
            const int kk = e / 64, x = e % 64;
            const int64_t ar = m0 + x, ak = k0 + kk;
            // as[kk][x] = A[m0 + x][k0 + kk]
            as[kk][x] = (ar < M && ak < K) ? A[ar * K + ak] : 0.0f;
            const int64_t bk = k0 + kk, bc = n0 + x;
            bs[kk][x] = (bk < K && bc < N) ? B[bk * N + bc] : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = as[kk][ty + 16 * i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = bs[kk][tx + 16 * j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t r = m0 + ty + 16 * i, c = n0 + tx + 16 * j;
            if (r < M && c < N) C[r * N + c] = acc[i][j];
        }
}

// partial[b] = sum over this block's grid-stride share of x * y (fp64).
__global__ void dot_partial_kernel(const float* __restrict__ x, const float* __restrict__ y, int64_t n,
                                   double* __restrict__ partial) {
    __shared__ double part[32];
    double s = 0.0;
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x)
        s += static_cast<double>(x[e]) * static_cast<double>(y[e]);
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x < 32) {
        s = threadIdx.x < blockDim.x / 32 ? part[threadIdx.x] : 0.0;
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (threadIdx.x == 0) partial[blockIdx.x] = s;
    }
}

__global__ void sum_kernel(const double* __restrict__ partial, int n, double* out) {
    if (threadIdx.x == 0 && blockIdx.x == 0) {
        double s = 0.0;
        for (int i = 0; i < n; ++i) s += partial[i];
        *out = s;
    }
}

constexpr int DOT_BLOCKS = 256;

}  // namespace

KQ_DEBUG_UNIT(check)
}  // namespace kq

using namespace kq;

extern "C" kq_status kq_dequant_revert(const uint8_t* codes, const float* scale, const int32_t* zero,
                                       int64_t d_out, int64_t d_in, int group, const float* s_x,
                                       const float* s_g, const int8_t* sign_u, const int8_t* sign_v,
                                       float* W_hat, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!codes || !scale || !zero || !sign_u || !sign_v || !W_hat || d_out < 1 || d_in < 1 || group < 0) {
        set_error("kq_dequant_revert: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    const int64_t total = d_out * d_in;
    dequant_kernel<<<static_cast<unsigned>(std::min<int64_t>(cdiv(total, 256), 65535)), 256, 0, stream>>>(
        codes, scale, zero, d_out, d_in, group, W_hat);
    KQ_LAUNCH_CHECK("dequant_kernel");
    kq_status st = rotate_cols_inv(W_hat, d_out, d_in, s_g, sign_u, stream);   // S_G^-1 U^T
    if (st != KQ_OK) {
        set_error("kq_dequant_revert: unsupported d_out=%lld", (long long)d_out);
        return st;
    }
    st = rotate_rows_inv(W_hat, d_out, d_in, s_x, sign_v, stream);             // V S_X^-1
    if (st != KQ_OK) set_error("kq_dequant_revert: unsupported d_in=%lld", (long long)d_in);
    return st;
}

extern "C" size_t kq_proxy_loss_workspace(int64_t d_out, int64_t d_in) {
    if (d_out < 1 || d_in < 1) return 0;
    return 3 * static_cast<size_t>(d_out) * d_in * sizeof(float) + DOT_BLOCKS * sizeof(double) + 256;
}

extern "C" kq_status kq_proxy_loss(const float* W, const float* W_hat, int64_t d_out, int64_t d_in,
                                   const float* H_X, const float* H_G, double* loss, void* ws,
                                   size_t ws_bytes, kq_stream_t stream_) {
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (!W || !W_hat || !H_X || !loss || d_out < 1 || d_in < 1) {
        set_error("kq_proxy_loss: invalid arguments");
        return KQ_ERR_INVALID_ARG;
    }
    if (!ws || ws_bytes < kq_proxy_loss_workspace(d_out, d_in) || (reinterpret_cast<uintptr_t>(ws) & 15u)) {
        set_error("kq_proxy_loss: workspace too small");
        return KQ_ERR_WORKSPACE;
    }
    const int64_t total = d_out * d_in;
    float* D = static_cast<float*>(ws);
    float* P = D + total;
    float* Q = P + total;
    double* partial = reinterpret_cast<double*>(Q + total);
    const unsigned eg = static_cast<unsigned>(std::min<int64_t>(cdiv(total, 256), 65535));
    sub_kernel<<<eg, 256, 0, stream>>>(W, W_hat, total, D);
    KQ_LAUNCH_CHECK("sub_kernel");
    gemm_nn_kernel<<<dim3(static_cast<unsigned>(cdiv(d_in, 64)), static_cast<unsigned>(cdiv(d_out, 64))), 256, 0,
                     stream>>>(D, H_X, P, d_out, d_in, d_in);   // P = dW H_X
    KQ_LAUNCH_CHECK("gemm_nn_kernel");
    const float* lhs = D;
    if (H_G) {
        gemm_nn_kernel<<<dim3(static_cast<unsigned>(cdiv(d_in, 64)), static_cast<unsigned>(cdiv(d_out, 64))), 256,
                         0, stream>>>(H_G, D, Q, d_out, d_in, d_out);   // Q = H_G dW
        KQ_LAUNCH_CHECK("gemm_nn_kernel");
        lhs = Q;
    }
    dot_partial_kernel<<<DOT_BLOCKS, 256, 0, stream>>>(lhs, P, total, partial);
    KQ_LAUNCH_CHECK("dot_partial_kernel");
    sum_kernel<<<1, 32, 0, stream>>>(partial, DOT_BLOCKS, loss);
    KQ_LAUNCH_CHECK("sum_kernel");
    return KQ_OK;
}
