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

// D (+)= A B for one m16n8k8 tf32 tile: A 16 x 8 (a0 (g, t), a1 (g + 8, t), a2 (g, t + 4),
// a3 (g + 8, t + 4)), B 8 x 8 (b0 (t, g), b1 (t + 4, g)), D 16 x 8 (d0 (g, 2t), d1 (g, 2t + 1),
// d2 (g + 8, 2t), d3 (g + 8, 2t + 1)); g = lane / 4, t = lane % 4. Operands are fp32 bit
// patterns (the tensor core reads their tf32 part).
__device__ __forceinline__ void mma_tf32(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile("mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
                 "{%0, %1, %2, %3};"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* m, const void* src, int x, int y) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                     reinterpret_cast<uint64_t>(m)),
                 "r"(smem_u32(src)), "r"(x), "r"(y)
                 : "memory");
}
// W[y:y+128, x:x+32] += the box in shared memory (element type and swizzle from the map;
// rows and columns outside the matrix are skipped).
__device__ __forceinline__ void tma_reduce_add_2d(const CUtensorMap* m, const void* src, int x, int y) {
    asm volatile("cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                     reinterpret_cast<uint64_t>(m)),
                 "r"(smem_u32(src)), "r"(x), "r"(y)
                 : "memory");
}
// Wait until at most N of this thread's bulk groups are still pending (their writes done).
template <int N>
__device__ __forceinline__ void bulk_wait_le() { asm volatile("cp.async.bulk.wait_group %0;" ::"n"(N) : "memory"); }
// Barrier `id` over n threads (whole warps; the non-.aligned form, so a warp may reach it
// after a branch taken by some of its lanes).
__device__ __forceinline__ void named_bar_sync(int id, int n) {
    asm volatile("barrier.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
// The same barrier, returning whether p held in every participating thread.
__device__ __forceinline__ bool named_bar_all(int id, int n, bool p) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred a, b;\n\t"
        "setp.ne.u32 a, %1, 0;\n\t"
        "barrier.red.and.pred b, %2, %3, a;\n\t"
        "selp.u32 %0, 1, 0, b;\n\t}"
        : "=r"(r)
        : "r"(static_cast<uint32_t>(p)), "r"(id), "r"(n)
        : "memory");
    return r != 0;
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Instruction descriptor, kind::tf32: fp32 accumulator, tf32 A and B, both K-major.
__host__ __device__ constexpr uint32_t idesc_tf32_k_major(int M, int N) {
    return (1u << 4)                                // D format: f32
           | (2u << 7)                              // A format: tf32
           | (2u << 10)                             // B format: tf32
           | (static_cast<uint32_t>(N >> 3) << 17)  // N / 8
           | (static_cast<uint32_t>(M >> 4) << 24); // M / 16
}

__device__ __forceinline__ void tc_mma_tf32(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// 2-D fp32 tensor map over a row-major [rows x cols] matrix: box = box_rows x 32 columns,
// 128-byte swizzle (a 32-float row is one swizzle atom), zero fill outside the matrix.
kq_status make_f32_map(CUtensorMap* m, const float* base, int64_t rows, int64_t cols, int box_rows);
// The same over a [rows x cols] block of a row-major matrix with leading dimension ld.
kq_status make_f32_map_ld(CUtensorMap* m, const float* base, int64_t rows, int64_t cols, int64_t ld, int box_rows);

// Tensor maps over the split error block and the split L, encoded once per sweep.
struct TrailMaps {
    CUtensorMap eh, el;                  // E_hi, E_lo [d_out x d_in], 128-row boxes
    CUtensorMap rh_narrow, rl_narrow;    // Lt_hi, Lt_lo [d_in x d_in], 128-row boxes
    CUtensorMap rh64, rl64;              // the same with 64-row boxes (64-column tiles)
    CUtensorMap w;                       // W [d_out x d_in], 128-row boxes (read and written)
    CUtensorMap qh, ql, ph, pl;          // with P: (-Wpre)_hi, _lo [d_out x d_in], Pt_hi, Pt_lo [d_in x d_in]
    kq_status init(const float* E_hi, const float* E_lo, const float* Lt_hi, const float* Lt_lo, int64_t d_out,
                   int64_t d_in);
    kq_status init_p(const float* Q_hi, const float* Q_lo, const float* Pt_hi, const float* Pt_lo, int64_t d_out,
                     int64_t d_in);
    kq_status set_w(float* W, int64_t d_out, int64_t d_in);
};

// Tensor maps of one inverse-Cholesky call (chol.cu): the padded A (-> C) and Z, and per
// split set the tf32 hi / lo of a block column panel of C and of the matching block rows of
// Z transposed ([npad x width] each). split[] lists Ch, Cl, Zh, Zl of set 0, then set 1.
struct CholTcMaps {
    CUtensorMap a, z;
    CUtensorMap ch[2], cl[2], zh[2], zl[2];
    kq_status init(float* A, float* Z, int64_t npad, int width, int nsets, float* const* split);
};

// A Cholesky update on the tensor cores (3xTF32): A_ij -= C_i. C_j.^T for the lower tiles with
// j in [a_j0, a_j1) and max(j, a_r0) <= i < a_r1 (a_r1 < 0: nbk), and Z_ij -= C_i. Z_.j for
// i in [b_i0, b_i1), j < b_j1, where the dot runs over the nslab * 32 split columns starting
// at kx of split set `set`: 256 x 256 tiles of 128 x 128 blocks on pairs of CTAs, on all
// resident clusters but free_sms / 2.
kq_status chol_update_tc(const CholTcMaps& m, int set, int nbk, int a_j0, int a_j1, int b_i0, int b_i1, int b_j1,
                         int kx, int nslab, int* info, cudaStream_t stream, int free_sms = 0, int a_r0 = 0,
                         int a_r1 = -1);

// out[r][c] -= sum over x < k of a[r][x] b[c][x] for r < rows, c < cols (3xTF32 from the
// tf32 hi / lo of a and b, row-major with leading dimension ld_ab; out with ld_out), on
// 256 x 256 tiles over pairs of CTAs. cols a multiple of 256, k of 32. ktri = 1: b is lower
// triangular (b[c][x] = 0 for x > c), so a tile of columns [c0, c0 + 256) runs K up to
// c0 + 256; ktri = 2: a is (a[r][x] = 0 for x > r), K up to the tile's last row + 1.
kq_status chol_gemm_tc(float* out, int64_t ld_out, int64_t rows, int64_t cols, const float* a_hi, const float* a_lo,
                       const float* b_hi, const float* b_lo, int64_t ld_ab, int k, int ktri, int* info,
                       cudaStream_t stream);

// hi = src rounded to tf32, lo = src - hi (n elements).
kq_status split_tf32(const float* src, int64_t n, float* hi, float* lo, cudaStream_t stream);

// W[:, cb:ce] -= E[:, i0:i0+kb] R[i0:i0+kb, cb:ce] (R[k][c] = Lt[c][k]) on tensor cores,
// and with_p: also -= Q[:, i0:i0+kb] P[i0:i0+kb, cb:ce] (P[k][c] = Pt[c][k]). kb = 128, or
// 256 in GPTQ mode (two blocks' updates in one launch, still applied 128 of K at a time).
// Tiles are 128 x 64 when narrow (GPTQ mode only; 129 KB of shared memory per CTA), else
// 128 x 128 (193 KB); [cb, ce) must be whole tiles or end at d_in. W is the one set_w was given.
kq_status trail_tc(const TrailMaps& m, float* W, int64_t d_out, int64_t d_in, int64_t i0, int64_t cb, int64_t ce,
                   bool with_p, bool narrow, int kb, int* info, cudaStream_t stream);

// The same update for K = kb <= 1024 (the blocks of one super-panel, GPTQ mode), applied to
// W two blocks' K at a time in block order (the accumulator drained every 256 of K), through
// TMA reduce-adds instead of a shared-memory copy of the W tile, on 256 x 256 tiles spread
// over pairs of CTAs (cta_group::2, a three-stage ring per CTA). [cb, ce) whole 256-column
// tiles or ending at d_in; kb whole blocks unless the super-panel ends at d_in.
kq_status trail_tc_long(const TrailMaps& m, int64_t d_out, int64_t d_in, int64_t i0, int kb, int64_t cb, int64_t ce,
                        int* info, cudaStream_t stream);

}  // namespace kq
