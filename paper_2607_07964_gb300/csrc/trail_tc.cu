// Stage 4, tensor-core variant of the OBS sweep's lazy trailing update (Algorithm 2):
//   W[:, cols] -= E_blk R_blk,   E_blk = E[:, i0:i0+128], R_blk[k][c] = Lt[c][i0 + k],
// and with the GPTAQ correction also -= Q_blk P_blk (Q = -Wpre, P_blk[k][c] = Pt[c][i0 + k]),
// i.e. K = 256 over [E | Q] and [R ; P],
// on the 5th-generation tensor cores with fp32-accurate products from the 3xTF32 split
// (Markidis et al. 2018; Ootomo & Yokota 2022): with x_hi = x rounded to tf32 and
// x_lo = x - x_hi (exact in fp32),  E R ~= E_hi R_hi + E_hi R_lo + E_lo R_hi, accumulated in
// fp32 in TMEM. The dropped E_lo R_lo term and the tf32 truncation of the lo parts are
// ~2^-22 of each product.
//
// Persistent CTAs (one per SM) walk 128 x BN output tiles, K = 128 in four 32-wide slabs
// through a 2-stage ring, with two TMEM accumulators so a tile's epilogue overlaps the next
// tile's loads and MMAs:
//   warp 0: TMA loads of E_hi, E_lo (128 rows x 32 k) and Lt_hi, Lt_lo (BN rows x 32 k),
//           K-major with 128-byte swizzle (a 32-float row is one swizzle atom);
//   warp 1: allocates 2 BN TMEM columns, issues tcgen05.mma kind::tf32 (M 128, N BN, K 8),
//           three per k step, into the accumulator the epilogue has released;
//   warps 2..9: two per TMEM lane quadrant, each thread one row and BN / 2 columns: they
//           load their slice of W into registers before the tile's MMAs finish (the loads
//           overlap the TMA/MMA pipeline), then subtract the accumulator and store, for the
//           rows < d_out and columns in [cb, ce).
// Every mbarrier wait is bounded; a timeout sets -KQ_ERR_TIMEOUT in *info and the CTA
// drains its copies and MMAs before it exits.
#include <algorithm>
#include <cstdlib>
#include <cstring>

#include "trail_tc.cuh"

namespace kq {
namespace {

constexpr int TBM = 128;                 // rows per tile (MMA M, TMEM lanes)
constexpr int TBK = 32;                  // k per slab (one 128-byte swizzle row)
constexpr int TK = 128;                  // block size: the K of every trailing update
constexpr int TNSLAB = TK / TBK;         // 4
constexpr int T_THREADS = 320;           // 10 warps: TMA, MMA, 8 epilogue
constexpr int A_SLAB = TBM * TBK * 4;    // 16 KB

// One-CTA tiles: the tile of W comes in by TMA, the epilogue subtracts the accumulator
// from it in shared memory and a TMA store writes it back.
template <int BN, int STAGES>
struct TrailCfg {
    static constexpr int B_SLAB = BN * TBK * 4;                    // 16 KB for BN = 128
    static constexpr int STAGE = 2 * A_SLAB + 2 * B_SLAB;          // hi + lo of both
    static constexpr int WBOX = TBM * 32 * 4;                      // one 128 x 32 box of W (16 KB)
    static constexpr int WTILE = TBM * BN * 4;                     // the tile of W
    static constexpr int SMEM = STAGES * STAGE + WTILE + 1024 + 256;
    static_assert(2 * BN <= 512, "two accumulators must fit in TMEM");
    static_assert(BN % 64 == 0, "W moves in 32-column boxes, two column halves");
    static_assert(SMEM <= 232448, "dynamic shared memory above the per-CTA limit");
};

__device__ __forceinline__ bool wait_quiet(uint64_t* bar, uint32_t parity) {
    int dummy = 0;
    return mbar_wait(bar, parity, &dummy);
}

// Which output tiles a launch updates, and from which operand maps.
//   mode 0 (the sweep; the Cholesky's products on CTA pairs): a row x column grid over
//     W[:, cb:], K slabs at columns i0 + 32 s of the first pair (E with R) and, for slabs
//     >= pslab (one-CTA kernel), at i0 + 32 (s - pslab) of the second pair (-Wpre with P).
//   mode 1 (a Cholesky update on CTA pairs, see chol.cu): first the A region -- lower tiles
//     (i, j) with j in [a_j0, a_j1) and max(j, a_r0) <= i < a_r1, output A, B operand from
//     the split C rows j -- then the B region -- tiles (i, j) with i in [b_i0, b_i1),
//     j < b_j1, output Z, B operand from the split transposed Z rows j. The A operand is the
//     split C rows i; K slabs at columns kx + 32 s of the split buffers.
struct TileSet {
    int mode;
    int n_tiles;
    int n_col_tiles, cb, i0, pslab, ce, rows;         // mode 0 (ce: end of the column range; rows of W)
    int nbk, a_j0, a_j1, n_a, b_i0, b_i1, b_j1, kx;   // mode 1
    int a_r0, a_r1;   // pair kernel, mode 1: A-region rows [max(j, a_r0), a_r1) of column block j
    int ktri;   // pair kernel, mode 0: 0, or a triangular operand bounds K per tile (see below)
};

// Tile t of the one-CTA kernel (mode 0): top-left corner (row r0, column c0).
__device__ __forceinline__ void tile_at(const TileSet& ts, int t, int bn, int* r0, int* c0) {
    *r0 = (t / ts.n_col_tiles) * TBM;
    *c0 = ts.cb + (t % ts.n_col_tiles) * bn;
}

template <int BN, int TSTAGES>
__global__ void __launch_bounds__(T_THREADS, 1)
trail_tc_kernel(const __grid_constant__ CUtensorMap mEh, const __grid_constant__ CUtensorMap mEl,
                const __grid_constant__ CUtensorMap mRh, const __grid_constant__ CUtensorMap mRl,
                const __grid_constant__ CUtensorMap mQh, const __grid_constant__ CUtensorMap mQl,
                const __grid_constant__ CUtensorMap mPh, const __grid_constant__ CUtensorMap mPl,
                const __grid_constant__ CUtensorMap mW, TileSet ts, int nslab, int drain, int* info) {
    const int n_tiles = ts.n_tiles;
    const int xk = ts.i0;
    using C = TrailCfg<BN, TSTAGES>;
    constexpr int WBOX = C::WBOX;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* wtile = smem + TSTAGES * C::STAGE;                   // BN / 32 boxes, 128-byte swizzled
    uint64_t* full = reinterpret_cast<uint64_t*>(wtile + C::WTILE);
    uint64_t* empty = full + TSTAGES;
    uint64_t* tfull = empty + TSTAGES;     // accumulator b holds a finished tile
    uint64_t* tempty = tfull + 2;          // the epilogue has read accumulator b
    uint64_t* wfull = tempty + 2;          // the W tile has arrived
    uint64_t* wfree = wfull + 1;           // the W tile has been stored (buffer reusable)
    uint64_t* wdone = wfree + 1;           // all 8 epilogue warps have updated the W tile
    uint64_t* mma_done = wdone + 1;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < TSTAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&tfull[b], 1);
            mbar_init(&tempty[b], 8);
        }
        mbar_init(wfull, 1);
        mbar_init(wfree, 1);
        mbar_init(wdone, 8);
        mbar_init(mma_done, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, 2 * BN);
        tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&mEh);
        tma_prefetch_desc(&mEl);
        tma_prefetch_desc(&mRh);
        tma_prefetch_desc(&mRl);
        tma_prefetch_desc(&mW);
        if (nslab > TNSLAB) {
            tma_prefetch_desc(&mQh);
            tma_prefetch_desc(&mQl);
            tma_prefetch_desc(&mPh);
            tma_prefetch_desc(&mPl);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int k = 0, li = 0, w_issued = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++li) {
                int r0, c0;
                tile_at(ts, t, BN, &r0, &c0);
                // the tile of W, once the previous tile has been stored from the buffer
                if (!mbar_wait(wfree, (static_cast<uint32_t>(li) & 1u) ^ 1u, abort_flag)) break;
                mbar_arrive_expect_tx(wfull, C::WTILE);
#pragma unroll
                for (int j = 0; j < BN / 32; ++j) tma_load_2d(wtile + j * WBOX, &mW, wfull, c0 + 32 * j, r0);
                w_issued = li + 1;
                for (int s = 0; s < nslab; ++s, ++k) {
                    const int st = k % TSTAGES;
                    const uint32_t u = static_cast<uint32_t>(k / TSTAGES);
                    if (!mbar_wait(&empty[st], (u & 1u) ^ 1u, abort_flag)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&full[st], C::STAGE);
                    uint8_t* base = smem + st * C::STAGE;
                    // slabs 0..3: E and R; slabs 4..7 (with P): -Wpre and P
                    const bool second = s >= ts.pslab;
                    const int x = xk + (second ? s - ts.pslab : s) * TBK;
                    tma_load_2d(base, second ? &mQh : &mEh, &full[st], x, r0);
                    tma_load_2d(base + A_SLAB, second ? &mQl : &mEl, &full[st], x, r0);
                    tma_load_2d(base + 2 * A_SLAB, second ? &mPh : &mRh, &full[st], x, c0);
                    tma_load_2d(base + 2 * A_SLAB + C::B_SLAB, second ? &mPl : &mRl, &full[st], x, c0);
                }
            }
            // every issued load must land before the CTA exits
            for (int j = (k > TSTAGES ? k - TSTAGES : 0); j < k; ++j)
                wait_quiet(&full[j % TSTAGES], static_cast<uint32_t>(j / TSTAGES) & 1u);
            if (w_issued > 0) wait_quiet(wfull, static_cast<uint32_t>(w_issued - 1) & 1u);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_tf32_k_major(TBM, BN);
            int k = 0, cc = 0;   // cc: accumulator chunks issued (the two buffers alternate per chunk)
            bool ok = true;
            for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
                for (int s0 = 0; s0 < nslab && ok; s0 += drain, ++cc) {
                    const int buf = cc & 1;
                    if (!mbar_wait(&tempty[buf], ((static_cast<uint32_t>(cc) >> 1) & 1u) ^ 1u, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t dt = tmem + static_cast<uint32_t>(buf * BN);
                    const int s1 = min(nslab, s0 + drain);
                    for (int s = s0; s < s1; ++s, ++k) {
                        const int st = k % TSTAGES;
                        if (!mbar_wait(&full[st], static_cast<uint32_t>(k / TSTAGES) & 1u, abort_flag)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t a_hi = smem_u32(smem + st * C::STAGE);
                        const uint32_t a_lo = a_hi + A_SLAB;
                        const uint32_t b_hi = a_hi + 2 * A_SLAB;
                        const uint32_t b_lo = b_hi + C::B_SLAB;
#pragma unroll
                        for (int kk = 0; kk < TBK / 8; ++kk) {   // 8 tf32 = 32 bytes per MMA
                            const uint32_t ko = static_cast<uint32_t>(kk * 32);
                            const uint64_t dah = smem_desc_sw128(a_hi + ko, 16, 1024);
                            const uint64_t dal = smem_desc_sw128(a_lo + ko, 16, 1024);
                            const uint64_t dbh = smem_desc_sw128(b_hi + ko, 16, 1024);
                            const uint64_t dbl = smem_desc_sw128(b_lo + ko, 16, 1024);
                            tc_mma_tf32(dt, dal, dbh, idesc, (s > s0 || kk > 0) ? 1u : 0u);
                            tc_mma_tf32(dt, dah, dbl, idesc, 1u);
                            tc_mma_tf32(dt, dah, dbh, idesc, 1u);
                        }
                        tc_commit(&empty[st]);
                    }
                    if (ok) tc_commit(&tfull[buf]);
                }
            }
            tc_commit(mma_done);
            wait_quiet(mma_done, 0);
        }
    } else {
        // ------------------------------------------------------------ epilogue (8 warps)
        // Thread = one row of the tile (TMEM lane) and BN / 2 columns. W sits in shared
        // memory as 128-byte swizzled rows (16-byte chunk c of row r at c ^ (r & 7)), so the
        // float4 accesses of 8 consecutive rows hit distinct banks.
        constexpr int HALF = BN / 2;
        const int q = warp & 3;                 // TMEM lane quadrant this warp may access
        const int h = (warp - 2) >> 2;          // which half of the columns
        const int r = q * 32 + lane;            // row within the tile
        int li = 0, cc = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++li) {
            ok = mbar_wait(wfull, static_cast<uint32_t>(li) & 1u, abort_flag);
            ok = __all_sync(0xffffffffu, ok) && !*abort_flag;
            if (!ok) break;
            // W -= each accumulator chunk in turn (K = drain * 32 per chunk)
            for (int s0 = 0; s0 < nslab; s0 += drain, ++cc) {
                const int buf = cc & 1;
                ok = mbar_wait(&tfull[buf], (static_cast<uint32_t>(cc) >> 1) & 1u, abort_flag);
                ok = __all_sync(0xffffffffu, ok) && !*abort_flag;
                if (!ok) break;
                tc_fence_after();
                const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) +
                                       static_cast<uint32_t>(buf * BN + h * HALF);
#pragma unroll
                for (int p = 0; p < HALF / 32; ++p) {
                    float v[32];
                    tmem_ld32(taddr + static_cast<uint32_t>(p * 32), v);
                    tc_wait_ld();
                    float4* rowp = reinterpret_cast<float4*>(wtile + (h * (HALF / 32) + p) * WBOX + r * 128);
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        float4* cp = rowp + (c ^ (r & 7));
                        const float4 o = *cp;
                        *cp = make_float4(o.x - v[4 * c], o.y - v[4 * c + 1], o.z - v[4 * c + 2], o.w - v[4 * c + 3]);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&tempty[buf]);   // the accumulator may be reused
            }
            if (!ok) break;
            fence_proxy_async();                        // this thread's W updates -> TMA
            __syncwarp();
            if (lane == 0) mbar_arrive(wdone);
            if (warp == 2 && lane == 0) {
                // store the tile once every warp has updated it, then free the buffer
                if (mbar_wait(wdone, static_cast<uint32_t>(li) & 1u, abort_flag)) {
                    int r0, c0;
                    tile_at(ts, t, BN, &r0, &c0);
#pragma unroll
                    for (int j = 0; j < BN / 32; ++j) tma_store_2d(&mW, wtile + j * WBOX, c0 + 32 * j, r0);
                    bulk_commit();
                    bulk_wait_read0();
                    mbar_arrive(wfree);
                }
            }
        }
        if (warp == 2 && lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
    }

    tc_fence_before();
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) record_error(info, -KQ_ERR_TIMEOUT);
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 2 * BN);
    }
}

// ------------------------------------------------------------ two-CTA tiles (cta_group::2)
// A cluster of two CTAs on two SMs computes one 256 x 256 tile. CTA r holds rows
// [128 r, 128 r + 128) of the tile's A operand and rows [128 r, 128 r + 128) of its B
// operand (the tile's columns 128 r ..); one tcgen05.mma with M = 256, issued by CTA 0,
// reads both CTAs' operand slabs and writes each CTA's 128 rows of the accumulator into
// that CTA's tensor memory. Each SM then stages and reads 128 x k of B per k slab instead
// of 256 x k: per 32-k slab and SM 64 KB of TMA writes and 96 KB of operand reads for
// 1536 MMA cycles, against 96 + 144 KB for the same cycles in a one-CTA 128 x 256 tile,
// whose loop is bound by the 128 bytes per cycle of shared memory. W never enters shared
// memory: the epilogue stages -accumulator one 128 x 32 box at a time (one staging box per
// column half) and a TMA reduce-add applies it to W in global memory.
//
// Synchronization: every CTA loads its own slabs with TMA, the transaction bytes of both
// landing on CTA 0's `full` barrier (the cta_group::2 form of the copy may signal the peer's
// barrier); CTA 0's MMA commits arrive on `empty`, `tfull` and `mma_done` of both CTAs
// (multicast); both CTAs' epilogue warps arrive on CTA 0's `tempty` (16 arrivals). Every
// wait is bounded as in the one-CTA kernel; both CTAs leave through one cluster barrier.
constexpr int PBN = 256;                        // tile columns (N of the pair's MMA)
constexpr int PSTAGES = 3;
constexpr int P_SLAB = TBM * TBK * 4;           // 16 KB: 128 rows x 32 k
constexpr int P_STAGE = 4 * P_SLAB;             // A hi, A lo, B hi, B lo of this CTA
constexpr int P_WBOX = TBM * 32 * 4;            // one 128 x 32 staging box
constexpr int P_SMEM = PSTAGES * P_STAGE + 2 * P_WBOX + 1024 + 256;
static_assert(P_SMEM <= 232448, "dynamic shared memory above the per-CTA limit");

__device__ __forceinline__ void tc_mma_tf32_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                                 uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Pair tile t as seen by CTA `rank`: the rows of the A operand it loads (ra; also the rows
// it writes), the rows of the B operand it loads (rb), the tile's first column (co), whether
// B and the output come from the second pair of maps, and which of its two 128-column
// halves it writes.
//   mode 0: tiles of 256 rows x 256 columns over W[:, cb:ce], column tiles inner.
//   mode 1: the A region in column-block pairs (a_j0 + 2 p, + 1), each with its row-block
//     pairs from the diagonal down (the strictly upper block of a diagonal tile is not
//     written), then the B region in (row pair, column pair) order.
struct PairTile {
    int ra, rb, co;
    bool alt;
    bool wr0, wr1;
};

// Tile of cluster `pair` in round rd of the persistent walk: the rounds alternate direction
// (boustrophedon), so a cluster that took one of the first tiles of a round takes one of the
// last of the next. Tiles whose cost grows along the order (the K bound of ktri) then even
// out per cluster, which the plain stride (with the cluster count a multiple of the column
// tiles, every tile of a cluster in one column) does not.
__device__ __forceinline__ int round_tile(int rd, int pair, int npairs) {
    return rd * npairs + ((rd & 1) ? npairs - 1 - pair : pair);
}

// K slabs of pair tile t: nslab, or in mode 0 with ktri set, only the slabs up to the end
// of the tile's 256 columns (ktri = 1: B rows c vanish beyond column c of K) or of its 256
// rows (ktri = 2: A rows r vanish beyond column r of K). The same for both CTAs of a pair.
__device__ __forceinline__ int pair_tile_nslab(const TileSet& ts, int t, int nslab) {
    if (ts.mode != 0 || ts.ktri == 0) return nslab;
    const int key = ts.ktri == 1 ? ts.cb + (t % ts.n_col_tiles) * PBN : (t / ts.n_col_tiles) * 2 * TBM;
    return min(nslab, (key + PBN) / TBK);
}

__device__ __forceinline__ PairTile pair_tile_at(const TileSet& ts, int t, int rank) {
    PairTile p;
    if (ts.mode == 0) {
        const int r0 = (t / ts.n_col_tiles) * 2 * TBM;
        const int c0 = ts.cb + (t % ts.n_col_tiles) * PBN;
        p.ra = r0 + TBM * rank;
        p.rb = c0 + TBM * rank;
        p.co = c0;
        p.alt = false;
        p.wr0 = p.ra < ts.rows && c0 < ts.ce;
        p.wr1 = p.ra < ts.rows && c0 + TBM < ts.ce;
        return p;
    }
    if (t < ts.n_a) {
        int jp = ts.a_j0;
        while (t >= (ts.a_r1 - max(jp, ts.a_r0) + 1) / 2) {
            t -= (ts.a_r1 - max(jp, ts.a_r0) + 1) / 2;
            jp += 2;
        }
        const int i = max(jp, ts.a_r0) + 2 * t + rank;
        p.ra = i * TBM;
        p.rb = (jp + rank) * TBM;
        p.co = jp * TBM;
        p.alt = false;
        p.wr0 = i < ts.a_r1;
        p.wr1 = i < ts.a_r1 && jp + 1 < ts.a_j1 && jp + 1 <= i;
        return p;
    }
    t -= ts.n_a;
    const int ncp = (ts.b_j1 + 1) / 2;
    const int i = ts.b_i0 + 2 * (t / ncp) + rank;
    const int j0 = 2 * (t % ncp);
    p.ra = i * TBM;
    p.rb = (j0 + rank) * TBM;
    p.co = j0 * TBM;
    p.alt = true;
    p.wr0 = i < ts.b_i1;
    p.wr1 = i < ts.b_i1 && j0 + 1 < ts.b_j1;
    return p;
}

// mA*: the A operand (E, or the split C panel), K slabs at columns xk + 32 s; mB*: the B
// operand (R, or the split C panel); mB2*: the second B operand (mode 1: the split Z^T
// rows); mW / mW2: the output for B / B2. Grid: two CTAs per cluster, the clusters walking
// the tiles (persistent).
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(T_THREADS, 1)
trail_pair_kernel(const __grid_constant__ CUtensorMap mAh, const __grid_constant__ CUtensorMap mAl,
                  const __grid_constant__ CUtensorMap mBh, const __grid_constant__ CUtensorMap mBl,
                  const __grid_constant__ CUtensorMap mB2h, const __grid_constant__ CUtensorMap mB2l,
                  const __grid_constant__ CUtensorMap mW, const __grid_constant__ CUtensorMap mW2, TileSet ts,
                  int nslab, int drain, int* info) {
    const int n_tiles = ts.n_tiles;
    const int xk = ts.mode == 0 ? ts.i0 : ts.kx;
    const uint32_t rank = cluster_ctarank();
    const int pair = static_cast<int>(blockIdx.x >> 1);
    const int npairs = static_cast<int>(gridDim.x >> 1);
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* wtile = smem + PSTAGES * P_STAGE;    // two staging boxes (one per column half)
    uint64_t* full = reinterpret_cast<uint64_t*>(wtile + 2 * P_WBOX);
    uint64_t* empty = full + PSTAGES;
    uint64_t* tfull = empty + PSTAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* mma_done = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < PSTAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&tfull[b], 1);
            mbar_init(&tempty[b], 16);   // 8 epilogue warps in each CTA
        }
        mbar_init(mma_done, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc_pair(tmem_slot, 2 * PBN);
        tmem_relinquish_pair();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&mAh);
        tma_prefetch_desc(&mAl);
        tma_prefetch_desc(&mBh);
        tma_prefetch_desc(&mBl);
        if (ts.mode == 1) {
            tma_prefetch_desc(&mB2h);
            tma_prefetch_desc(&mB2l);
        }
    }
    tc_fence_before();
    __syncthreads();
    cluster_barrier();   // both CTAs' barriers initialized before any remote arrival
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t full0 = mapa_shared(smem_u32(full), 0);       // CTA 0's full[0]
    const uint32_t tempty0 = mapa_shared(smem_u32(tempty), 0);   // CTA 0's tempty[0]

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer (both CTAs)
        if (lane == 0) {
            int k = 0;
            bool ok = true;
            for (int rd = 0; rd * npairs < n_tiles && ok; ++rd) {
                const int t = round_tile(rd, pair, npairs);
                if (t >= n_tiles) continue;
                const PairTile pt = pair_tile_at(ts, t, static_cast<int>(rank));
                const CUtensorMap* bh = pt.alt ? &mB2h : &mBh;
                const CUtensorMap* bl = pt.alt ? &mB2l : &mBl;
                const int ns = pair_tile_nslab(ts, t, nslab);
                for (int s = 0; s < ns; ++s, ++k) {
                    const int st = k % PSTAGES;
                    const uint32_t u = static_cast<uint32_t>(k / PSTAGES);
                    if (!mbar_wait(&empty[st], (u & 1u) ^ 1u, abort_flag)) {
                        ok = false;
                        break;
                    }
                    if (rank == 0) mbar_arrive_expect_tx(&full[st], 2 * P_STAGE);
                    uint8_t* base = smem + st * P_STAGE;
                    const uint32_t bar = full0 + static_cast<uint32_t>(st * 8);
                    const int x = xk + s * TBK;
                    tma_load_2d_pair(base, &mAh, bar, x, pt.ra);
                    tma_load_2d_pair(base + P_SLAB, &mAl, bar, x, pt.ra);
                    tma_load_2d_pair(base + 2 * P_SLAB, bh, bar, x, pt.rb);
                    tma_load_2d_pair(base + 3 * P_SLAB, bl, bar, x, pt.rb);
                }
            }
            // the last slabs consumed by the pair's MMAs (so this CTA's loads have landed)
            for (int j = (k > PSTAGES ? k - PSTAGES : 0); j < k; ++j)
                wait_quiet(&empty[j % PSTAGES], static_cast<uint32_t>(j / PSTAGES) & 1u);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (CTA 0)
        if (lane == 0) {
            if (rank == 0) {
                constexpr uint32_t idesc = idesc_tf32_k_major(2 * TBM, PBN);
                int k = 0, cc = 0;
                bool ok = true;
                for (int rd = 0; rd * npairs < n_tiles && ok; ++rd) {
                    const int t = round_tile(rd, pair, npairs);
                    if (t >= n_tiles) continue;
                    const int ns = pair_tile_nslab(ts, t, nslab);
                    for (int s0 = 0; s0 < ns && ok; s0 += drain, ++cc) {
                        const int buf = cc & 1;
                        if (!mbar_wait_cl(&tempty[buf], ((static_cast<uint32_t>(cc) >> 1) & 1u) ^ 1u, abort_flag)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t dt = tmem + static_cast<uint32_t>(buf * PBN);
                        const int s1 = min(ns, s0 + drain);
                        for (int s = s0; s < s1; ++s, ++k) {
                            const int st = k % PSTAGES;
                            if (!mbar_wait(&full[st], static_cast<uint32_t>(k / PSTAGES) & 1u, abort_flag)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            const uint32_t a_hi = smem_u32(smem + st * P_STAGE);
                            const uint32_t a_lo = a_hi + P_SLAB;
                            const uint32_t b_hi = a_hi + 2 * P_SLAB;
                            const uint32_t b_lo = a_hi + 3 * P_SLAB;
#pragma unroll
                            for (int kk = 0; kk < TBK / 8; ++kk) {
                                const uint32_t ko = static_cast<uint32_t>(kk * 32);
                                const uint64_t dah = smem_desc_sw128(a_hi + ko, 16, 1024);
                                const uint64_t dal = smem_desc_sw128(a_lo + ko, 16, 1024);
                                const uint64_t dbh = smem_desc_sw128(b_hi + ko, 16, 1024);
                                const uint64_t dbl = smem_desc_sw128(b_lo + ko, 16, 1024);
                                tc_mma_tf32_pair(dt, dal, dbh, idesc, (s > s0 || kk > 0) ? 1u : 0u);
                                tc_mma_tf32_pair(dt, dah, dbl, idesc, 1u);
                                tc_mma_tf32_pair(dt, dah, dbh, idesc, 1u);
                            }
                            tc_commit_pair(&empty[st]);
                        }
                        if (ok) tc_commit_pair(&tfull[buf]);
                    }
                }
                tc_commit_pair(mma_done);
            }
            wait_quiet(mma_done, 0);
        }
    } else {
        // ------------------------------------------------------------ epilogue (8 warps, both CTAs)
        // Thread = one row of this CTA's 128 rows (TMEM lane); warps 2-5 take columns
        // [0, 128) of the tile, warps 6-9 columns [128, 256). Each drained chunk goes to W
        // box by box, the same box of the previous chunk landing first (block order per
        // element).
        constexpr int HALF = PBN / 2;
        constexpr int PIECES = HALF / 32;
        const int q = warp & 3;
        const int h = (warp - 2) >> 2;
        const int r = q * 32 + lane;
        const bool issuer = (warp == 2 + 4 * h) && lane == 0;
        uint8_t* stg = wtile + h * P_WBOX;
        int cc = 0;
        bool ok = true;
        for (int rd = 0; rd * npairs < n_tiles && ok; ++rd) {
            const int t = round_tile(rd, pair, npairs);
            if (t >= n_tiles) continue;
            const PairTile pt = pair_tile_at(ts, t, static_cast<int>(rank));
            const CUtensorMap* wm = pt.alt ? &mW2 : &mW;
            const int xh = pt.co + h * HALF;
            const bool wrh = h ? pt.wr1 : pt.wr0;
            const bool whole = wrh && (ts.mode == 1 || xh + HALF <= ts.ce);
            const int ns = pair_tile_nslab(ts, t, nslab);
            for (int s0 = 0; s0 < ns; s0 += drain, ++cc) {
                const int buf = cc & 1;
                ok = mbar_wait(&tfull[buf], (static_cast<uint32_t>(cc) >> 1) & 1u, abort_flag);
                ok = __all_sync(0xffffffffu, ok) && !*abort_flag;
                ok = named_bar_all(1 + h, 128, ok);
                if (!ok) break;
                tc_fence_after();
                const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) +
                                       static_cast<uint32_t>(buf * PBN + h * HALF);
#pragma unroll 1
                for (int p = 0; p < PIECES; ++p) {
                    const int x = xh + 32 * p;
                    float v[32];
                    tmem_ld32(taddr + static_cast<uint32_t>(p * 32), v);
                    tc_wait_ld();
                    if (p == PIECES - 1) {   // the accumulator may be reused
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive_remote(tempty0 + static_cast<uint32_t>(buf * 8));
                    }
                    if (!wrh || (ts.mode == 0 && x >= ts.ce)) continue;   // same for the whole half
                    float4* rowp = reinterpret_cast<float4*>(stg + r * 128);
#pragma unroll
                    for (int c = 0; c < 8; ++c)
                        rowp[c ^ (r & 7)] = make_float4(-v[4 * c], -v[4 * c + 1], -v[4 * c + 2], -v[4 * c + 3]);
                    fence_proxy_async();
                    named_bar_sync(1 + h, 128);
                    if (issuer) {
                        // the same box of the previous chunk lands first (block order per element)
                        if (whole)
                            bulk_wait_le<PIECES - 1>();
                        else
                            bulk_wait_le<0>();
                        tma_reduce_add_2d(wm, stg, x, pt.ra);
                        bulk_commit();
                        bulk_wait_read0();
                    }
                    named_bar_sync(1 + h, 128);
                }
            }
        }
        if ((warp == 2 || warp == 6) && lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
    }

    tc_fence_before();
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) {
        record_error(info, -KQ_ERR_TIMEOUT);
        // copies this CTA issued toward the peer's barriers have had time to land
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 1000000ull) {
        }
    }
    cluster_barrier();   // neither CTA leaves while the other may still signal it
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, 2 * PBN);
    }
}

__global__ void split_tf32_kernel(const float* __restrict__ src, int64_t n, float* __restrict__ hi,
                                  float* __restrict__ lo) {
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const float x = src[i];
        const float h = tf32_hi(x);
        if (!KQ_IN_RANGE(i, n)) continue;
        hi[i] = h;
        lo[i] = x - h;
    }
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

}  // namespace

kq_status make_f32_map(CUtensorMap* m, const float* base, int64_t rows, int64_t cols, int box_rows) {
    return make_f32_map_ld(m, base, rows, cols, cols, box_rows);
}

kq_status make_f32_map_ld(CUtensorMap* m, const float* base, int64_t rows, int64_t cols, int64_t ld, int box_rows) {
    EncodeTiledFn enc = encode_tiled();
    if (!enc) {
        set_error("trailing update: cuTensorMapEncodeTiled is unavailable");
        return KQ_ERR_CUDA;
    }
    std::memset(m, 0, sizeof(*m));
    cuuint64_t gdim[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    cuuint64_t gstride[1] = {static_cast<cuuint64_t>(ld) * 4};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(TBK), static_cast<cuuint32_t>(box_rows)};
    cuuint32_t estride[2] = {1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(base), gdim, gstride, box, estride,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("trailing update: cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
        return KQ_ERR_CUDA;
    }
    return KQ_OK;
}

kq_status split_tf32(const float* src, int64_t n, float* hi, float* lo, cudaStream_t stream) {
    const int64_t grid = std::min<int64_t>(cdiv(n, 256), static_cast<int64_t>(num_sms()) * 16);
    split_tf32_kernel<<<static_cast<unsigned>(std::max<int64_t>(grid, 1)), 256, 0, stream>>>(src, n, hi, lo);
    KQ_LAUNCH_CHECK("split_tf32_kernel");
    return KQ_OK;
}

kq_status TrailMaps::init(const float* E_hi, const float* E_lo, const float* Lt_hi, const float* Lt_lo,
                          int64_t d_out, int64_t d_in) {
    kq_status st;
    if ((st = make_f32_map(&eh, E_hi, d_out, d_in, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&el, E_lo, d_out, d_in, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&rh_narrow, Lt_hi, d_in, d_in, 128)) != KQ_OK) return st;
    if ((st = make_f32_map(&rl_narrow, Lt_lo, d_in, d_in, 128)) != KQ_OK) return st;
    if ((st = make_f32_map(&rh64, Lt_hi, d_in, d_in, 64)) != KQ_OK) return st;
    if ((st = make_f32_map(&rl64, Lt_lo, d_in, d_in, 64)) != KQ_OK) return st;
    return KQ_OK;
}

kq_status TrailMaps::init_p(const float* Q_hi, const float* Q_lo, const float* Pt_hi, const float* Pt_lo,
                            int64_t d_out, int64_t d_in) {
    kq_status st;
    if ((st = make_f32_map(&qh, Q_hi, d_out, d_in, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&ql, Q_lo, d_out, d_in, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&ph, Pt_hi, d_in, d_in, 128)) != KQ_OK) return st;
    if ((st = make_f32_map(&pl, Pt_lo, d_in, d_in, 128)) != KQ_OK) return st;
    return KQ_OK;
}

kq_status TrailMaps::set_w(float* W, int64_t d_out, int64_t d_in) {
    return make_f32_map(&w, W, d_out, d_in, TBM);
}

namespace {
template <int BN>
kq_status launch_trail(const TrailMaps& m, const CUtensorMap& rh, const CUtensorMap& rl, int64_t d_out, int64_t i0,
                       int64_t cb, int64_t ce, bool with_p, int kslabs, int* info, cudaStream_t stream) {
    using Cfg = TrailCfg<BN, 2>;
    static std::atomic<uint64_t> attr{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(trail_tc_kernel<BN, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM));
        KQ_CUDA(cudaFuncSetAttribute(trail_tc_kernel<BN, 2>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                     cudaSharedmemCarveoutMaxShared));
        return KQ_OK;
    }));
    const int n_row = static_cast<int>(cdiv(d_out, TBM));
    const int n_col = static_cast<int>(cdiv(ce - cb, BN));
    TileSet ts{};
    ts.mode = 0;
    ts.n_tiles = n_row * n_col;
    ts.n_col_tiles = n_col;
    ts.cb = static_cast<int>(cb);
    ts.i0 = static_cast<int>(i0);
    ts.pslab = with_p ? kslabs : 1 << 30;
    ts.ce = static_cast<int>(ce);
    // the accumulator goes into W every 128 of K (one block's update at a time, as the
    // per-block schedule does); with P after the E and P halves of one block together
    trail_tc_kernel<BN, 2><<<static_cast<unsigned>(std::min(ts.n_tiles, num_sms())), T_THREADS, Cfg::SMEM, stream>>>(
        m.eh, m.el, rh, rl, with_p ? m.qh : m.eh, with_p ? m.ql : m.el, with_p ? m.ph : rh, with_p ? m.pl : rl, m.w, ts,
        with_p ? 2 * kslabs : kslabs, with_p ? 2 * kslabs : TNSLAB, info);
    KQ_LAUNCH_CHECK("trail_tc_kernel");
    return KQ_OK;
}
}  // namespace

kq_status trail_tc(const TrailMaps& m, float* W, int64_t d_out, int64_t d_in, int64_t i0, int64_t cb, int64_t ce,
                   bool with_p, bool narrow, int kb, int* info, cudaStream_t stream) {
    // Persistent: at most one CTA per SM, each walking the tiles t, t + grid, ... (column
    // tile fastest, so the CTAs running together share row and column operands in L2). A
    // range either is a whole number of tiles or ends at d_in (the TMA copies clip the last
    // tile there).
    (void)W;
    narrow = narrow && !with_p;
    const int bn = narrow ? 64 : 128;
    if ((ce - cb) % bn != 0 && ce != d_in) {
        set_error("trailing update: column range [%lld, %lld) is not whole tiles", (long long)cb, (long long)ce);
        return KQ_ERR_INVALID_ARG;
    }
    if ((kb != 128 && kb != 256) || (with_p && kb != 128)) {
        set_error("trailing update: K must be 128 or (GPTQ mode) 256, got %d", kb);
        return KQ_ERR_INVALID_ARG;
    }
    if (narrow) return launch_trail<64>(m, m.rh64, m.rl64, d_out, i0, cb, ce, false, kb / TBK, info, stream);
    return launch_trail<128>(m, m.rh_narrow, m.rl_narrow, d_out, i0, cb, ce, with_p, kb / TBK, info, stream);
}

namespace {
// Slabs of 32 K between two drains of the accumulator into W in the long updates (K up to
// 1024): 8, i.e. two blocks' updates summed in TMEM before each reduce-add into W (half the
// epilogue traffic of one drain per block: the 70B down_proj layer 297 against 309 ms; the
// inverse Cholesky's relative error at n = 4096 and 8192 grows from 5.6e-7 and 6.4e-7 to
// 9.2e-7 and 1.1e-6, against a 1e-5 bar), or 4 (one block at a time) when the environment
// variable KQ_TRAIL_DRAIN_SLABS says 4 (a tuning switch).
int long_drain_slabs() {
    static const int n = [] {
        const char* e = std::getenv("KQ_TRAIL_DRAIN_SLABS");
        return (e && std::atoi(e) == 4) ? 4 : 8;
    }();
    return n;
}

// Persistent: as many clusters as can be resident at once walk the tiles, less free_sms / 2
// (SMs left to kernels that run beside the launch, such as the next super-panel's steps of
// the inverse Cholesky). One cluster per tile (so that finished clusters hand their SMs to
// the critical-path kernels of the higher-priority stream) measured slower on the 70B
// down_proj layer: Cholesky 84.5 against 74.6 ms, sweep 37.9 against 34.2 ms.
kq_status launch_pair(const CUtensorMap& ah, const CUtensorMap& al, const CUtensorMap& bh, const CUtensorMap& bl,
                      const CUtensorMap& b2h, const CUtensorMap& b2l, const CUtensorMap& w, const CUtensorMap& w2,
                      const TileSet& ts, int nslab, int drain, int* info, cudaStream_t stream, int free_sms = 0) {
    static std::atomic<uint64_t> attr{0};
    static std::atomic<int> clusters{0};
    KQ_TRY(once_per_device(attr, [&]() -> kq_status {
        KQ_CUDA(cudaFuncSetAttribute(trail_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, P_SMEM));
        KQ_CUDA(cudaFuncSetAttribute(trail_pair_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                     cudaSharedmemCarveoutMaxShared));
        // clusters resident at once (pairs of SMs that can both take a CTA)
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(2 * num_sms()));
        cfg.blockDim = dim3(T_THREADS);
        cfg.dynamicSmemBytes = P_SMEM;
        int c = 0;
        KQ_CUDA(cudaOccupancyMaxActiveClusters(&c, trail_pair_kernel, &cfg));
        clusters.store(c > 0 ? c : num_sms() / 2);
        return KQ_OK;
    }));
    if (ts.n_tiles == 0) return KQ_OK;
    const int nc = std::min(ts.n_tiles, std::max(1, clusters.load() - free_sms / 2));
    trail_pair_kernel<<<static_cast<unsigned>(2 * nc), T_THREADS, P_SMEM, stream>>>(ah, al, bh, bl, b2h, b2l, w, w2,
                                                                                    ts, nslab, drain, info);
    KQ_LAUNCH_CHECK("trail_pair_kernel");
    return KQ_OK;
}

}  // namespace

kq_status trail_tc_long(const TrailMaps& m, int64_t d_out, int64_t d_in, int64_t i0, int kb, int64_t cb, int64_t ce,
                        int* info, cudaStream_t stream) {
    if (kb < 1 || kb > 1024 || i0 + kb > d_in || (kb % TK != 0 && i0 + kb != d_in)) {
        set_error("trailing update: K = %d from column %lld is not whole blocks of the super-panel", kb, (long long)i0);
        return KQ_ERR_INVALID_ARG;
    }
    if ((ce - cb) % PBN != 0 && ce != d_in) {
        set_error("trailing update: column range [%lld, %lld) is not whole %d-column tiles", (long long)cb,
                  (long long)ce, PBN);
        return KQ_ERR_INVALID_ARG;
    }
    if (ce <= cb) return KQ_OK;
    TileSet ts{};
    ts.mode = 0;
    ts.n_col_tiles = static_cast<int>(cdiv(ce - cb, PBN));
    ts.n_tiles = static_cast<int>(cdiv(d_out, 2 * TBM)) * ts.n_col_tiles;
    ts.cb = static_cast<int>(cb);
    ts.i0 = static_cast<int>(i0);
    ts.pslab = 1 << 30;
    ts.ce = static_cast<int>(ce);
    ts.rows = static_cast<int>(d_out);
    return launch_pair(m.eh, m.el, m.rh_narrow, m.rl_narrow, m.rh_narrow, m.rl_narrow, m.w, m.w, ts,
                       static_cast<int>(cdiv(kb, TBK)), long_drain_slabs(), info, stream);
}

// ------------------------------------------------------------ Cholesky step updates
kq_status CholTcMaps::init(float* A, float* Z, int64_t npad, int width, int nsets, float* const* split) {
    kq_status st;
    if ((st = make_f32_map(&a, A, npad, npad, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map(&z, Z, npad, npad, TBM)) != KQ_OK) return st;
    for (int q = 0; q < nsets; ++q) {
        if ((st = make_f32_map(&ch[q], split[4 * q + 0], npad, width, TBM)) != KQ_OK) return st;
        if ((st = make_f32_map(&cl[q], split[4 * q + 1], npad, width, TBM)) != KQ_OK) return st;
        if ((st = make_f32_map(&zh[q], split[4 * q + 2], npad, width, TBM)) != KQ_OK) return st;
        if ((st = make_f32_map(&zl[q], split[4 * q + 3], npad, width, TBM)) != KQ_OK) return st;
    }
    return KQ_OK;
}

kq_status chol_gemm_tc(float* out, int64_t ld_out, int64_t rows, int64_t cols, const float* a_hi, const float* a_lo,
                       const float* b_hi, const float* b_lo, int64_t ld_ab, int k, int ktri, int* info,
                       cudaStream_t stream) {
    if (rows < 1 || cols < 1) return KQ_OK;
    if (k < TBK || k % TBK != 0 || k > ld_ab || cols % PBN != 0 || ktri < 0 || ktri > 2) {
        set_error("Cholesky GEMM: K = %d, %lld columns (whole %d-column tiles, K in 32-column slabs)", k,
                  (long long)cols, PBN);
        return KQ_ERR_INVALID_ARG;
    }
    CUtensorMap ah, al, bh, bl, w;
    kq_status st;
    if ((st = make_f32_map_ld(&ah, a_hi, rows, k, ld_ab, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map_ld(&al, a_lo, rows, k, ld_ab, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map_ld(&bh, b_hi, cols, k, ld_ab, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map_ld(&bl, b_lo, cols, k, ld_ab, TBM)) != KQ_OK) return st;
    if ((st = make_f32_map_ld(&w, out, rows, cols, ld_out, TBM)) != KQ_OK) return st;
    TileSet ts{};
    ts.mode = 0;
    ts.n_col_tiles = static_cast<int>(cols / PBN);
    ts.n_tiles = static_cast<int>(cdiv(rows, 2 * TBM)) * ts.n_col_tiles;
    ts.cb = 0;
    ts.i0 = 0;
    ts.pslab = 1 << 30;
    ts.ce = static_cast<int>(cols);
    ts.rows = static_cast<int>(rows);
    ts.ktri = ktri;
    return launch_pair(ah, al, bh, bl, bh, bl, w, w, ts, k / TBK, long_drain_slabs(), info, stream);
}

kq_status chol_update_tc(const CholTcMaps& m, int set, int nbk, int a_j0, int a_j1, int b_i0, int b_i1, int b_j1,
                         int kx, int nslab, int* info, cudaStream_t stream, int free_sms, int a_r0, int a_r1) {
    // 256 x 256 tiles on CTA pairs
    if (a_r1 < 0) a_r1 = nbk;
    TileSet ts{};
    ts.mode = 1;
    ts.nbk = nbk;
    ts.a_j0 = a_j0;
    ts.a_j1 = a_j1;
    ts.a_r0 = a_r0;
    ts.a_r1 = a_r1;
    for (int jp = a_j0; jp < a_j1; jp += 2) ts.n_a += std::max(0, (a_r1 - std::max(jp, a_r0) + 1) / 2);
    ts.b_i0 = b_i0;
    ts.b_i1 = b_i1;
    ts.b_j1 = b_j1;
    ts.kx = kx;
    ts.ce = 1 << 30;
    ts.n_tiles = ts.n_a + ((b_i1 > b_i0 && b_j1 > 0) ? ((b_i1 - b_i0 + 1) / 2) * ((b_j1 + 1) / 2) : 0);
    return launch_pair(m.ch[set], m.cl[set], m.ch[set], m.cl[set], m.zh[set], m.zl[set], m.a, m.z, ts, nslab,
                       long_drain_slabs(), info, stream, free_sms);
}


KQ_DEBUG_UNIT(trail_tc)
}  // namespace kq
