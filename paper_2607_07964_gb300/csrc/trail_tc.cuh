// Tensor-core (3xTF32) trailing update of the OBS sweep; see trail_tc.cu.
#pragma once

#include "kq_common.cuh"

namespace kq {

// x rounded to tf32 (nearest, ties away from zero), as an fp32 value with 13 zero low bits.
__device__ __forceinline__ float tf32_hi(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return __uint_as_float(r);
}

// Tensor maps over the split error block and the split L, encoded once per sweep.
struct TrailMaps {
    CUtensorMap eh, el;                  // E_hi, E_lo [d_out x d_in], 128-row boxes
    CUtensorMap rh_narrow, rl_narrow;    // Lt_hi, Lt_lo [d_in x d_in], 128-row boxes
    CUtensorMap w;                       // W [d_out x d_in], 128-row boxes (read and written)
    kq_status init(const float* E_hi, const float* E_lo, const float* Lt_hi, const float* Lt_lo, int64_t d_out,
                   int64_t d_in);
    kq_status set_w(float* W, int64_t d_out, int64_t d_in);
};

// hi = src rounded to tf32, lo = src - hi (n elements).
kq_status split_tf32(const float* src, int64_t n, float* hi, float* lo, cudaStream_t stream);

// W[:, cb:ce] -= E[:, i0:i0+128] R[i0:i0+128, cb:ce] (R[k][c] = Lt[c][k]) on tensor cores;
// [cb, ce) must be whole 128-column tiles or end at d_in. W is the one set_w was given.
kq_status trail_tc(const TrailMaps& m, float* W, int64_t d_out, int64_t d_in, int64_t i0, int64_t cb, int64_t ce,
                   int* info, cudaStream_t stream);

}  // namespace kq
