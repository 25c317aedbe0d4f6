// gs_gemm_tc.cu -- general tcgen05 GEMM for the matrix-space operators:
//
//     C = alpha * A B^T            (optionally divided by rownorm[i] * colnorm[j])
//
//   A  m x K row-major, in one of three modes:
//        kAF16     fp32, rounded to fp16 (RN) on the fly   D  = A16 B0^T
//        kABF16X2  fp32, hi = bf16(A), lo = bf16(A - hi)   D  = Ah B0^T + Al B0^T + Ah B1^T
//        kAF16T    fp16 already (rounded once by the caller) D = A16 B0^T
//      In the first two, TMA streams fp32 tiles into a staging ring and two groups
//      of converter warps write the 128-byte-swizzled K-major operand layout (the
//      split keeps ~16 significant bits and fp32's exponent range, for products
//      whose terms do not average out, e.g. with the dominant diagonal of R).  In
//      kAF16T, TMA writes that layout itself, straight into the A stages: for an A
//      that every N tile re-reads (reconstruct: T against 40 column tiles of Q),
//      rounding it once halves its L2 traffic and frees the converters and the
//      staging ring's shared memory for deeper A and B rings.
//   B0, B1  16-bit (fp16 with kAF16 / kAF16T, bf16 with kABF16X2), n x K row-major
//      (K-major), by TMA; these are the basis' operand copies, L2-resident.
//   C  fp32 or bf16, m x n, leading dimension ldc.
//
// Uses (paper Sec. 3.1 / 3.3): reconstruction Xhat = T Q (kAF16T, B0 = fp16 Q^T), the
// projection Y = X Q^T for bases too wide for the fused kernel (B0 = fp16 Q),
// scores S = Y R^T (split, B0 / B1 = bf16 hi / lo of R) and probability
// vectorization V = P R (split, B0 / B1 = bf16 hi / lo of R^T).
//
// Tiles are 128 x nt (nt <= 256) with the fp32 accumulator double-buffered in
// TMEM (2 x 256 columns), or, for a long K with A rounded to fp16 and n > 256, 128 x 2 nt (nt <= 256)
// (two 256-column accumulators filling TMEM, single-buffered: each converted A K-block
// feeds both); one persistent CTA per SM walks the tiles with the n index fastest (rotated
// each wave so that no CTA keeps one column tile), so
// CTAs running at the same time share A rows in L2.
// Warp roles (608 threads): 0-3 and 15-18 epilogue (warp w reads TMEM lanes
// 32 (w % 4)..+31; the two warps of a lane quadrant take alternate 32-column chunks,
// so output-heavy products like reconstruct are not held up by the stores),
// 4 TMA producer of A, 5 TMEM allocator + MMA issuer, 6 TMA producer of B,
// 7-14 converters in two groups taking alternate K-blocks (with A loaded by TMA they
// join the epilogue: four warps per lane quadrant).  Every mbarrier wait
// is bounded (see gs_tc_ptx.cuh); on expiry the CTA records GS_DEV_ERR_TIMEOUT,
// unwinds, waits for its own copies and MMAs, frees TMEM and returns.

#include <float.h>

#include <algorithm>

#include "gs_internal.h"
#include "gs_tc_ptx.cuh"

namespace gs {
namespace {

using namespace ptx;

__device__ unsigned g_err_gemm = 0;

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kEpiWarps = 4;
constexpr int kAWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kBWarp = 6;
constexpr int kCvt0 = 7;
constexpr int kCvtGroups = 2;
constexpr int kCvtGroupWarps = 4;
constexpr int kCvtWarps = kCvtGroups * kCvtGroupWarps;
constexpr int kEpi2 = kCvt0 + kCvtWarps;               // second epilogue group: warps 15-18
constexpr int kEpiWarpsTotal = 2 * kEpiWarps;
constexpr int kThreads = (kEpi2 + kEpiWarps) * 32;       // 608
// 19 warps: one sub-partition holds 5, so a thread may use at most 65536 / 4 / (5 * 32) = 102
// registers (allocated in steps of 8: 96)
constexpr int kCvtRowStep = kCvtGroupWarps * 32 / 16;  // 8
constexpr int kCvtRows = kBM / kCvtRowStep;            // 16
constexpr int kXStageBytes = kBM * kBK * 4;            // 32 KB
constexpr int kAPartBytes = kBM * kBK * 2;             // 16 KB
constexpr int kBStageBytes = 256 * kBK * 2;            // 32 KB
constexpr int kMaxSX = 4, kMaxSA = 4, kMaxSB = 4;
constexpr int kTmemCols = 512;
constexpr int kMaxTilesN = 64;  // column tiles whose K-block range can be trimmed

// A operand modes: fp32 rounded to fp16 by the converters; fp32 split into bf16 hi / lo by
// the converters (three products with B hi / lo); fp16 already, loaded by TMA straight into
// the A stages (no staging ring, no converters).
enum { kAF16 = 0, kABF16X2 = 1, kAF16T = 2 };

struct GemmParams {
    long long m;
    int n, K, nkb, nt, tiles_n;
    long long tiles;
    int amode, nb, parts;   // nb: B matrices per K-block; parts: A operand tiles per K-block
    int sx, sa, sb;
    void* C;
    long long ldc;
    int c_bf16, c_vec;      // c_vec: rows aligned for two-element stores
    float alpha;
    const float* rownorm;
    const float* colnorm;
    // K-blocks [kb_lo[tn], kb_hi[tn]) of column tile tn (krange = 1); outside them B's rows of the
    // tile are zero (R's echelon structure), so skipping them changes no sum
    int krange;
    int kb_lo[kMaxTilesN], kb_hi[kMaxTilesN];
    int rotate;             // the grid is a multiple of tiles_n: column tiles rotate by one each wave
    float* xn2;             // kAF16 (optional): per converter group, the rows' partial ||a||^2 (2 x m)
    const float* rowmul;    // optional: outputs of row i multiplied by rowmul[i]
};

struct Ctl {
    uint64_t x_full[kMaxSX], x_empty[kMaxSX];
    uint64_t a_full[kMaxSA], a_empty[kMaxSA];
    uint64_t b_full[kMaxSB], b_empty[kMaxSB];
    uint64_t d_full[2], d_empty[2];
    uint64_t mma_done;
    uint32_t tmem_base;
    int abort_flag;
};

// AMODE: kAF16, kABF16X2 or kAF16T; HALVES = 2: 128 x 2 nt tiles (two accumulators, fp16 A, one
// B).  Template parameters, so that each kernel carries only its own mode's control flow.
template <int AMODE, int HALVES>
__global__ void __maxnreg__(96)  // 608 threads: at most 96 registers each (see kThreads)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b0,
              const __grid_constant__ CUtensorMap tmap_b1, const __grid_constant__ GemmParams p) {
    // A loaded by TMA leaves the converter warps idle: they store output tiles instead
    constexpr bool kCvtEpi = AMODE == kAF16T;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    uint8_t* Xs = base;
    uint8_t* As = Xs + (size_t)p.sx * kXStageBytes;
    uint8_t* Bs = As + (size_t)p.sa * p.parts * kAPartBytes;
    Ctl& c = *reinterpret_cast<Ctl*>(Bs + (size_t)p.sb * kBStageBytes);
    volatile int* abort_flag = &c.abort_flag;
    unsigned* err = &g_err_gemm;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // this CTA's tiles: blockIdx.x, blockIdx.x + gridDim.x, ...
    const int ntiles = p.tiles > blockIdx.x ? (int)((p.tiles - 1 - blockIdx.x) / gridDim.x + 1) : 0;
    auto krange = [&](int tn, int& lo, int& hi) {
        lo = p.krange ? p.kb_lo[tn] : 0;
        hi = p.krange ? p.kb_hi[tn] : p.nkb;
    };
    // Tile lt of this CTA is tile index tg = blockIdx.x + lt gridDim.x: row block tg / tiles_n and
    // column tile tg mod tiles_n, rotated by one each wave (lt) when the grid is a multiple of
    // tiles_n (p.rotate).  CTAs working at the same time share A row blocks in L2, and no CTA keeps
    // one column tile: with trimmed K ranges (R's echelon structure) column tiles differ in length,
    // and the CTAs fixed to the longest would set the kernel's time.  (A wave then covers whole row
    // blocks, so the rotation permutes each block's column tiles; with any other grid the plain
    // order already moves every CTA through the column tiles.)
    auto tile_mn = [&](int lt, long long& tm, int& tn) {
        const long long tg = blockIdx.x + (long long)lt * gridDim.x;
        tm = tg / p.tiles_n;
        tn = (int)((tg + (p.rotate ? lt : 0)) % p.tiles_n);
    };
    int total_it = 0;  // K-blocks over this CTA's tiles
    for (int lt = 0; lt < ntiles; ++lt) {
        long long tm;
        int tn, lo, hi;
        tile_mn(lt, tm, tn);
        krange(tn, lo, hi);
        total_it += hi - lo;
    }

    if (threadIdx.x == 0) {
        for (int s = 0; s < p.sx; ++s) {
            mbar_init(&c.x_full[s], 1);
            mbar_init(&c.x_empty[s], kCvtGroupWarps);
        }
        for (int s = 0; s < p.sa; ++s) {
            mbar_init(&c.a_full[s], AMODE == kAF16T ? 1 : kCvtGroupWarps);
            mbar_init(&c.a_empty[s], 1);
        }
        for (int s = 0; s < p.sb; ++s) {
            mbar_init(&c.b_full[s], 1);
            mbar_init(&c.b_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&c.d_full[b], 1);
            mbar_init(&c.d_empty[b], kCvtEpi ? kEpiWarpsTotal + kCvtWarps : kEpiWarpsTotal);
        }
        mbar_init(&c.mma_done, 1);
        c.abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(&c.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = c.tmem_base;

    if (warp == kAWarp && AMODE == kAF16T) {
        // ------------------------------------------------------------- A tiles (fp16) via TMA
        // straight into the swizzled A stages the MMA reads
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_last();  // each row block is read once per N tile
            int it = 0;
            RingPos as;
            bool ok = true;
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                long long tm;
                int tn, lo, hi;
                tile_mn(lt, tm, tn);
                krange(tn, lo, hi);
                for (int kb = lo; kb < hi; ++kb, ++it, as.next(p.sa)) {
                    const int s = as.idx;
                    if (!mbar_wait_1t(&c.a_empty[s], as.phase ^ 1u, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&c.a_full[s], kAPartBytes);
                    tma_load_2d(As + (size_t)s * kAPartBytes, &tmap_a, &c.a_full[s], kb * kBK, (int)(tm * kBM),
                                pol);
                }
            }
            for (int j = std::max(0, it - p.sa); j < it; ++j) mbar_drain(&c.a_full[j % p.sa], (uint32_t)(j / p.sa) & 1u, err);
        }
    } else if (warp == kAWarp) {
        // ------------------------------------------------------------- A tiles (fp32) via TMA
        if (lane == 0) {
            // A row block read by one column tile: first to go from L2.  Read by several (the CTAs
            // of a wave take a row block's column tiles side by side): the normal class, so the
            // lines one CTA brings in stay for its neighbours, behind the B operands (evict_last)
            // but ahead of nothing (evict_first had them evicted before the neighbour's read:
            // 1.48 bytes read from DRAM per byte of A over a 10,000-deep projection)
            const uint64_t pol = p.tiles_n > 1 ? l2_policy_evict_normal() : l2_policy_evict_first();
            int it = 0;
            RingPos xs;
            bool ok = true;
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                long long tm;
                int tn, lo, hi;
                tile_mn(lt, tm, tn);
                krange(tn, lo, hi);
                for (int kb = lo; kb < hi; ++kb, ++it, xs.next(p.sx)) {
                    const int s = xs.idx;
                    if (!mbar_wait_1t(&c.x_empty[s], xs.phase ^ 1u, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&c.x_full[s], kXStageBytes);
                    tma_load_2d(Xs + (size_t)s * kXStageBytes, &tmap_a, &c.x_full[s], kb * kBK, (int)(tm * kBM),
                                pol);
                }
            }
            for (int j = std::max(0, it - p.sx); j < it; ++j) mbar_drain(&c.x_full[j % p.sx], (uint32_t)(j / p.sx) & 1u, err);
        }
    } else if (warp == kBWarp) {
        // ------------------------------------------------------------- B tiles via TMA (nb per K-block)
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_last();
            const uint32_t bytes = (uint32_t)p.nt * kBK * 2;
            int ib = 0;
            RingPos bs;
            bool ok = true;
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                long long tm;
                int tn, lo, hi;
                tile_mn(lt, tm, tn);
                krange(tn, lo, hi);
                for (int kb = lo; kb < hi && ok; ++kb)
                    for (int hf = 0; hf < HALVES && ok; ++hf)
                        for (int which = 0; which < p.nb; ++which, ++ib, bs.next(p.sb)) {
                            const int s = bs.idx;
                            if (!mbar_wait_1t(&c.b_empty[s], bs.phase ^ 1u, abort_flag, err)) {
                                ok = false;
                                break;
                            }
                            mbar_arrive_expect_tx(&c.b_full[s], bytes);
                            tma_load_2d(Bs + (size_t)s * kBStageBytes, which ? &tmap_b1 : &tmap_b0, &c.b_full[s],
                                        kb * kBK, (tn * HALVES + hf) * p.nt, pol);
                        }
            }
            for (int j = std::max(0, ib - p.sb); j < ib; ++j) mbar_drain(&c.b_full[j % p.sb], (uint32_t)(j / p.sb) & 1u, err);
        }
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc = AMODE == kABF16X2 ? idesc_bf16_f32(p.nt) : idesc_f16_f32(p.nt);
            RingPos ra, rb;
            bool ok = true;
            const int nbuf = HALVES == 2 ? 1 : 2;  // a tile of two halves fills TMEM
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                const int buf = lt % nbuf;
                if (!mbar_wait_1t(&c.d_empty[buf], ((uint32_t)(lt / nbuf) & 1u) ^ 1u, abort_flag, err)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * 256);
                long long tm;
                int tn, lo, hi;
                tile_mn(lt, tm, tn);
                krange(tn, lo, hi);
                for (int kb = lo; kb < hi; ++kb, ra.next(p.sa)) {
                    const int sa = ra.idx;
                    if (!mbar_wait_1t(&c.a_full[sa], ra.phase, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    const uint8_t* At = As + (size_t)sa * p.parts * kAPartBytes;
                    const uint64_t ah = sdesc_sw128(smem_u32(At));
                    if (HALVES == 1) {
                        const int sb0 = rb.idx;
                        if (!mbar_wait_1t(&c.b_full[sb0], rb.phase, abort_flag, err)) {
                            ok = false;
                            break;
                        }
                        rb.next(p.sb);
                        tc_fence_after();
                        const uint64_t b0 = sdesc_sw128(smem_u32(Bs + (size_t)sb0 * kBStageBytes));
                        if (AMODE != kABF16X2) {
#pragma unroll
                            for (int k = 0; k < kBK / 16; ++k)
                                mma_f16_ss(d_tmem, ah + (uint64_t)(2 * k), b0 + (uint64_t)(2 * k), idesc,
                                           (kb != lo || k != 0) ? 1u : 0u);
                            mma_commit(&c.a_empty[sa]);
                            mma_commit(&c.b_empty[sb0]);
                            continue;
                        }
                        // split operands: the two products with B hi (Ah Bh + Al Bh) go first and
                        // release B hi's stage, so B lo, one stage behind in the ring, has that long
                        // to land before Ah Bl needs it
                        const uint64_t al = sdesc_sw128(smem_u32(At + kAPartBytes));
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            mma_f16_ss(d_tmem, ah + (uint64_t)(2 * k), b0 + (uint64_t)(2 * k), idesc,
                                       (kb != lo || k != 0) ? 1u : 0u);
                            mma_f16_ss(d_tmem, al + (uint64_t)(2 * k), b0 + (uint64_t)(2 * k), idesc, 1u);
                        }
                        mma_commit(&c.b_empty[sb0]);
                        const int sb1 = rb.idx;
                        if (!mbar_wait_1t(&c.b_full[sb1], rb.phase, abort_flag, err)) {
                            ok = false;
                            break;
                        }
                        rb.next(p.sb);
                        tc_fence_after();
                        const uint64_t b1 = sdesc_sw128(smem_u32(Bs + (size_t)sb1 * kBStageBytes));
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k)
                            mma_f16_ss(d_tmem, ah + (uint64_t)(2 * k), b1 + (uint64_t)(2 * k), idesc, 1u);
                        mma_commit(&c.a_empty[sa]);
                        mma_commit(&c.b_empty[sb1]);
                        continue;
                    }
                    // wide tile (fp16 A, one B per half): the A K-block feeds both halves
                    for (int hf = 0; hf < 2 && ok; ++hf) {
                        const int sb0 = rb.idx;
                        if (!mbar_wait_1t(&c.b_full[sb0], rb.phase, abort_flag, err)) {
                            ok = false;
                            break;
                        }
                        rb.next(p.sb);
                        tc_fence_after();
                        const uint32_t dh = d_tmem + (uint32_t)(hf * p.nt);  // the halves side by side
                        const uint64_t b0 = sdesc_sw128(smem_u32(Bs + (size_t)sb0 * kBStageBytes));
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k)
                            mma_f16_ss(dh, ah + (uint64_t)(2 * k), b0 + (uint64_t)(2 * k), idesc,
                                       (kb != lo || k != 0) ? 1u : 0u);
                        mma_commit(&c.b_empty[sb0]);
                    }
                    if (!ok) break;
                    mma_commit(&c.a_empty[sa]);
                }
                if (ok) mma_commit(&c.d_full[buf]);
            }
            mma_commit(&c.mma_done);
            mbar_drain(&c.mma_done, 0, err);
        }
    } else if (!kCvtEpi && warp >= kCvt0 && warp < kEpi2) {
        // ------------------------------------------------------------- converters
        const int g = (warp - kCvt0) / kCvtGroupWarps;
        const int l = threadIdx.x - (kCvt0 + g * kCvtGroupWarps) * 32;  // 0..127
        const int c4 = l & 15, rbase = l >> 4;
        float amax = 0.f;
        // kAF16 with xn2: this group's part of each row's ||a||^2 over the current tile.  The 16
        // lanes that share rows (one row phase, c4 = lane & 15) fold their 16 per-row K-block sums
        // together in a butterfly after each K-block, so that lane c4 keeps the sum of row
        // rbase + 8 c4 in one register; it is written out (for column tile 0, which every row
        // block has) when the group moves to the next tile.
        const bool want_xn2 = AMODE == kAF16 && p.xn2 != nullptr;
        float nacc = 0.f;
        int lt = 0, tile_end = 0;  // tile of the K-blocks being converted, and its end in `it`
        if (ntiles > 0) {
            long long tm;
            int tn, lo, hi;
            tile_mn(0, tm, tn);
            krange(tn, lo, hi);
            tile_end = hi - lo;
        }
        auto flush_xn2 = [&]() {
            long long tm;
            int tn;
            tile_mn(lt, tm, tn);
            const long long row = tm * kBM + rbase + kCvtRowStep * c4;
            if (tn == 0 && row < p.m) p.xn2[(long long)g * p.m + row] = nacc;
            nacc = 0.f;
        };
        // ring positions of K-block g, then advanced by the two groups' K-blocks each step
        RingPos rx, ra;
        for (int j = 0; j < g; ++j) {
            rx.next(p.sx);
            ra.next(p.sa);
        }
        for (int it = g; AMODE != kAF16T && it < total_it; it += kCvtGroups) {
            if (want_xn2) {
                while (it >= tile_end) {  // this group is done with tile lt
                    flush_xn2();
                    ++lt;
                    long long tm;
                    int tn, lo, hi;
                    tile_mn(lt, tm, tn);
                    krange(tn, lo, hi);
                    tile_end += hi - lo;
                }
            }
            const int sx = rx.idx, sa = ra.idx;
            if (!mbar_wait_warp(&c.x_full[sx], rx.phase, abort_flag, err) ||
                !mbar_wait_warp(&c.a_empty[sa], ra.phase ^ 1u, abort_flag, err))
                break;
            for (int j = 0; j < kCvtGroups; ++j) {
                rx.next(p.sx);
                ra.next(p.sa);
            }
            const uint8_t* Xt = Xs + (size_t)sx * kXStageBytes;
            uint8_t* At = As + (size_t)sa * p.parts * kAPartBytes;
            // fp16 A: the whole K-block into registers first, so the staging stage goes back to
            // the A producer before the conversion rather than after it (the split mode, with
            // twice the stores per element, keeps the loads inside the loop: its registers are
            // spoken for).  Every loaded value is used (range, norm) before the stage is released:
            // an arrive issued while loads were still outstanding let the TMA refill overwrite
            // the stage under them
            constexpr bool kEarlyX = AMODE == kAF16;
            float4 xv[kCvtRows];
            float nrm[kCvtRows];  // this K-block's part of ||a||^2 of each of the thread's rows
            if (kEarlyX) {
#pragma unroll
                for (int u = 0; u < kCvtRows; ++u)
                    xv[u] = *reinterpret_cast<const float4*>(Xt + (rbase + kCvtRowStep * u) * (kBK * 4) + c4 * 16);
#pragma unroll
                for (int u = 0; u < kCvtRows; ++u) {
                    const float4 x = xv[u];
                    amax = fmaxf(amax, fmaxf(fmaxf(fabsf(x.x), fabsf(x.y)), fmaxf(fabsf(x.z), fabsf(x.w))));
                    nrm[u] = fmaf(x.x, x.x, fmaf(x.y, x.y, fmaf(x.z, x.z, x.w * x.w)));
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&c.x_empty[sx]);
            }
#pragma unroll
            for (int u = 0; u < kCvtRows; ++u) {
                const int row = rbase + kCvtRowStep * u;
                const float4 x = kEarlyX ? xv[u] : *reinterpret_cast<const float4*>(Xt + row * (kBK * 4) + c4 * 16);
                const int off = row * 128 + (((c4 >> 1) ^ (row & 7)) * 16) + (c4 & 1) * 8;
                uint2 hi;
                if (AMODE == kAF16) {
                    const __half2 h0 = __floats2half2_rn(x.x, x.y), h1 = __floats2half2_rn(x.z, x.w);
                    hi.x = *reinterpret_cast<const uint32_t*>(&h0);
                    hi.y = *reinterpret_cast<const uint32_t*>(&h1);
                } else {
                    const __nv_bfloat162 b0 = __floats2bfloat162_rn(x.x, x.y), b1 = __floats2bfloat162_rn(x.z, x.w);
                    hi.x = *reinterpret_cast<const uint32_t*>(&b0);
                    hi.y = *reinterpret_cast<const uint32_t*>(&b1);
                    const float2 f0 = __bfloat1622float2(b0), f1 = __bfloat1622float2(b1);
                    uint2 lo;
                    lo.x = pack_bf16(x.x - f0.x, x.y - f0.y);
                    lo.y = pack_bf16(x.z - f1.x, x.w - f1.y);
                    *reinterpret_cast<uint2*>(At + kAPartBytes + off) = lo;
                }
                *reinterpret_cast<uint2*>(At + off) = hi;
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&c.a_full[sa]);
                if (!kEarlyX) mbar_arrive(&c.x_empty[sx]);
            }
            if (want_xn2) {
                // butterfly over the 16 lanes of a row phase: after the step with lane bit b, a
                // lane holds half as many rows, those whose index u has bit b equal to its own
#pragma unroll
                for (int w = kCvtRows / 2; w >= 1; w >>= 1) {
                    const bool up = (lane & w) != 0;
#pragma unroll
                    for (int j = 0; j < w; ++j) {
                        const float send = up ? nrm[j] : nrm[j + w];
                        const float keep = up ? nrm[j + w] : nrm[j];
                        nrm[j] = keep + __shfl_xor_sync(0xffffffffu, send, w);
                    }
                }
                nacc += nrm[0];  // the K-block's sum for row rbase + 8 c4
            }
        }
        if (want_xn2) {
            while (lt < ntiles) {  // the last tile (and any tile with no K-block of this group)
                flush_xn2();
                ++lt;
            }
        }
        // with xn2 the caller recomputes the rows outside fp16's range; otherwise they are an error
        if (!want_xn2 && amax > 65504.f) atomicOr(err, GS_DEV_ERR_RANGE);
    } else {
        // ------------------------------------------------------------- epilogue (warps 0-3, 15-18,
        // and with A loaded by TMA the idle converter warps 7-14 as well)
        // TMEM is read in the 16x256b pattern so that each store writes whole sectors:
        // thread t holds rows (t/4) and (t/4 + 8) of a 16-lane half, 8 columns per quad.
        // The warps of a lane quadrant take alternate 32-column chunks: two per quadrant, or
        // four when the converter warps join.
        const int quad = warp & 3;  // lane quadrant
        const int chunk = warp < kCvt0 ? 0 : warp >= kEpi2 ? 1 : 2 + (warp - kCvt0) / kCvtGroupWarps;
        constexpr int nchunks = kCvtEpi ? 4 : 2;
        const int nbuf = HALVES == 2 ? 1 : 2;
        const int tw = p.nt * HALVES;  // tile width
        for (int lt = 0; lt < ntiles; ++lt) {
            const int buf = lt % nbuf;
            if (!mbar_wait_warp(&c.d_full[buf], (uint32_t)(lt / nbuf) & 1u, abort_flag, err)) break;
            tc_fence_after();
            long long tm;
            int tn;
            tile_mn(lt, tm, tn);
            for (int half = 0; half < 2; ++half) {
                const int lrow = quad * 32 + half * 16;
                const uint32_t tb = tmem + ((uint32_t)lrow << 16) + (uint32_t)(buf * 256);
                const long long row[2] = {tm * kBM + lrow + (lane >> 2), tm * kBM + lrow + (lane >> 2) + 8};
                float rn[2], rm[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    rn[h] = (p.rownorm && row[h] < p.m) ? p.rownorm[row[h]] : 1.f;
                    rm[h] = (p.rowmul && row[h] < p.m) ? p.rowmul[row[h]] * p.alpha : p.alpha;
                }
                for (int jc = 32 * chunk; jc < tw; jc += 32 * nchunks) {
                    float v[16];
                    tmem_ld16x256b_x4(tb + (uint32_t)jc, v);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int col = tn * tw + jc + 8 * j + 2 * (lane & 3);
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            if (row[h] >= p.m || col >= p.n) continue;
                            float g0 = rm[h] * v[4 * j + 2 * h], g1 = rm[h] * v[4 * j + 2 * h + 1];
                            if (p.colnorm) {
                                const float d0 = rn[h] * p.colnorm[col];
                                const float d1 = col + 1 < p.n ? rn[h] * p.colnorm[col + 1] : 0.f;
                                g0 = d0 > 0.f ? g0 / d0 : 0.f;
                                g1 = d1 > 0.f ? g1 / d1 : 0.f;
                            }
                            const size_t off = (size_t)row[h] * p.ldc + col;
                            if (p.c_bf16) {
                                __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(p.C) + off;
                                if (p.c_vec && col + 1 < p.n) {
                                    *reinterpret_cast<uint32_t*>(dst) = pack_bf16(g0, g1);
                                } else {
                                    dst[0] = __float2bfloat16_rn(g0);
                                    if (col + 1 < p.n) dst[1] = __float2bfloat16_rn(g1);
                                }
                            } else {
                                float* dst = reinterpret_cast<float*>(p.C) + off;
                                if (p.c_vec && col + 1 < p.n) {
                                    __stcs(reinterpret_cast<float2*>(dst), make_float2(g0, g1));
                                } else {
                                    dst[0] = g0;
                                    if (col + 1 < p.n) dst[1] = g1;
                                }
                            }
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.d_empty[buf]);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ----------------------------------------------------------------- CTA-pair GEMM, fp16 A by TMA
// k_gemm_tc2: C = alpha A B^T (x rowmul[i]) with A already fp16 (reconstruct: the rounded T) on
// pairs of CTAs (clusters of two): one pair MMA (tcgen05 cta_group::2, M = 256) computes a
// 256 x nt tile, each CTA staging its own 128 rows of A and half of the tile's nt rows of B, so an
// SM stages half the B bytes the single-CTA kernel does for the same outputs (B dominated the
// shared-memory traffic that held reconstruct's MMAs at half rate).  The even CTA's A and B
// producers expect both CTAs' bytes on its own full barriers, the odd CTA's TMA loads complete on
// them; the even CTA's MMA thread commits stage releases and accumulator hand-offs to both CTAs;
// each CTA's epilogue reads its own TMEM rows and releases the accumulator on the even CTA's
// barrier.  Warp roles (640 threads): 0 A producer, 1 TMEM allocator + MMA issuer (even CTA),
// 2 B producer, 3 idle, 4-19 epilogue (warp w reads TMEM lanes 32 (w % 4)..+31; the four warps of a
// lane quadrant take alternate 32-column chunks, one TMEM row per thread, and write them through
// two 2 KB staging buffers each (32 rows x 16 floats, 64-byte swizzle) as TMA tensor stores, so the
// output bytes leave through the TMA unit rather than as per-thread stores through L1).  Every wait
// is bounded.
constexpr int kP2EpiWarps = 16;
constexpr int kP2Threads = (4 + kP2EpiWarps) * 32;
constexpr int kP2StageBytes = 128 * kBK * 2;  // 16 KB: 128 rows of one fp16 K-block (A, or half of B)
constexpr int kP2MaxS = 5;
constexpr int kP2ZCols = 16;                  // an output box: 32 rows x 64 bytes
constexpr int kP2ZStage = 32 * kP2ZCols * 4;  // 2 KB

struct Gemm2Params {
    long long m;
    int n, nkb, nt, tiles_n;
    long long tiles;  // pair tiles (256 rows x nt columns)
    int sa, sb, rotate;
    float* C;
    long long ldc;
    float alpha;
    const float* rowmul;
};

struct Ctl2 {
    uint64_t a_full[kP2MaxS], a_empty[kP2MaxS];
    uint64_t b_full[kP2MaxS], b_empty[kP2MaxS];
    uint64_t d_full[2], d_empty[2];
    uint64_t mma_done;
    uint32_t tmem_base;
    int abort_flag;
};

__global__ void __launch_bounds__(kP2Threads, 1)
    k_gemm_tc2(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
               const __grid_constant__ CUtensorMap tmap_c, const __grid_constant__ Gemm2Params p) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    uint8_t* As = base;
    uint8_t* Bs = As + (size_t)p.sa * kP2StageBytes;
    uint8_t* Cs = Bs + (size_t)p.sb * kP2StageBytes;
    Ctl2& c = *reinterpret_cast<Ctl2*>(Cs + (size_t)kP2EpiWarps * 2 * kP2ZStage);
    volatile int* abort_flag = &c.abort_flag;
    unsigned* err = &g_err_gemm;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool lead = rank == 0;
    const long long pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
    const int ntiles = p.tiles > pair ? (int)((p.tiles - 1 - pair) / npairs + 1) : 0;
    auto tile_mn = [&](int lt, long long& tm, int& tn) {
        const long long tg = pair + (long long)lt * npairs;
        tm = tg / p.tiles_n;
        tn = (int)((tg + (p.rotate ? lt : 0)) % p.tiles_n);
    };
    if (threadIdx.x == 0) {
        for (int s = 0; s < p.sa; ++s) {
            mbar_init(&c.a_full[s], 1);
            mbar_init(&c.a_empty[s], 1);
        }
        for (int s = 0; s < p.sb; ++s) {
            mbar_init(&c.b_full[s], 1);
            mbar_init(&c.b_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&c.d_full[b], 1);
            mbar_init(&c.d_empty[b], 2 * kP2EpiWarps);  // the epilogue warps of both CTAs
        }
        mbar_init(&c.mma_done, 1);
        c.abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc2(&c.tmem_base, kTmemCols);
        tmem_relinquish2();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();  // the even CTA's barriers exist before the odd CTA signals them
    tc_fence_after();
    const uint32_t tmem = c.tmem_base;
    const uint32_t bbytes = (uint32_t)(p.nt / 2) * kBK * 2;  // one CTA's half of a B K-block

    if (warp == 0 || warp == 2) {
        // ------------------------------------------------------------- A (warp 0) / B (warp 2) tiles
        if (lane == 0) {
            const bool isa = warp == 0;
            const int depth = isa ? p.sa : p.sb;
            uint64_t* full = isa ? c.a_full : c.b_full;
            uint64_t* empty = isa ? c.a_empty : c.b_empty;
            uint8_t* stages = isa ? As : Bs;
            const uint32_t bytes = isa ? (uint32_t)kP2StageBytes : bbytes;
            const CUtensorMap* map = isa ? &tmap_a : &tmap_b;
            const uint64_t pol = l2_policy_evict_last();
            int it = 0;
            RingPos rp;
            bool ok = true;
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                long long tm;
                int tn;
                tile_mn(lt, tm, tn);
                const int y = isa ? (int)(tm * 256 + 128 * rank) : tn * p.nt + (int)rank * (p.nt / 2);
                for (int kb = 0; kb < p.nkb; ++kb, ++it, rp.next(depth)) {
                    if (!mbar_wait_1t(&empty[rp.idx], rp.phase ^ 1u, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    if (lead) mbar_arrive_expect_tx(&full[rp.idx], 2u * bytes);
                    tma_load_2d_pair(stages + (size_t)rp.idx * kP2StageBytes, map,
                                     mapa_shared(smem_u32(&full[rp.idx]), 0), kb * kBK, y, pol);
                }
            }
            // the even CTA waits until every stage it expected (both CTAs' loads) has landed; the
            // odd CTA's loads land on those barriers, and it leaves only after the closing cluster
            // barrier, which the even CTA reaches after this drain
            if (lead)
                for (int j = std::max(0, it - depth); j < it; ++j)
                    mbar_drain(&full[j % depth], (uint32_t)(j / depth) & 1u, err);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------- pair MMA issue (even CTA)
        if (lane == 0 && lead) {
            const uint32_t idesc = idesc2_f16_f32(p.nt);
            RingPos ra, rb;
            bool ok = true;
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                const int buf = lt & 1;
                // both CTAs' epilogues have read this accumulator (arrivals at cluster scope)
                if (!mbar_wait_cluster(&c.d_empty[buf], ((uint32_t)(lt >> 1) & 1u) ^ 1u, abort_flag, err)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * 256);
                // a narrow last column tile (w <= nt / 2 valid columns) takes all of them from the even
                // CTA's half of B, so an MMA of N = 2 ceil(w / 8) 8 covers them; the odd CTA's half
                // (rows beyond n, zero) and the accumulator columns it leaves stale map to output
                // columns at or beyond n, which the tensor stores clip
                long long tm;
                int tn;
                tile_mn(lt, tm, tn);
                const int w = p.n - tn * p.nt;
                const uint32_t idesc_t = w <= p.nt / 2 ? idesc2_f16_f32(std::max(32, 2 * ((w + 7) / 8 * 8))) : idesc;
                for (int kb = 0; kb < p.nkb; ++kb, ra.next(p.sa), rb.next(p.sb)) {
                    if (!mbar_wait_1t(&c.a_full[ra.idx], ra.phase, abort_flag, err) ||
                        !mbar_wait_1t(&c.b_full[rb.idx], rb.phase, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = sdesc_sw128(smem_u32(As + (size_t)ra.idx * kP2StageBytes));
                    const uint64_t bd = sdesc_sw128(smem_u32(Bs + (size_t)rb.idx * kP2StageBytes));
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k)
                        mma2_f16_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc_t, (kb | k) != 0 ? 1u : 0u);
                    mma2_commit(&c.a_empty[ra.idx], 3);
                    mma2_commit(&c.b_empty[rb.idx], 3);
                }
                if (ok) mma2_commit(&c.d_full[buf], 3);
            }
            mma2_commit(&c.mma_done, 1);
            mbar_drain(&c.mma_done, 0, err);
        }
    } else if (warp >= 4) {
        // ------------------------------------------------------------- epilogue: this CTA's 128 rows
        const int quad = warp & 3, chunk = (warp - 4) >> 2;
        const uint32_t lanes = (uint32_t)(32 * quad) << 16;
        uint8_t* zst = Cs + (size_t)(warp - 4) * 2 * kP2ZStage;
        int zb = 0;
        for (int lt = 0; lt < ntiles; ++lt) {
            const int buf = lt & 1;
            if (!mbar_wait_warp(&c.d_full[buf], (uint32_t)(lt >> 1) & 1u, abort_flag, err)) break;
            tc_fence_after();
            long long tm;
            int tn;
            tile_mn(lt, tm, tn);
            const long long row0 = tm * 256 + 128 * rank;
            const long long row = row0 + 32 * quad + lane, y = row0 + 32 * quad;
            const float rm = (p.rowmul && row < p.m) ? p.rowmul[row] * p.alpha : p.alpha;
            for (int jc = 32 * chunk; jc < p.nt; jc += 32 * 4) {
                uint32_t v[32];
                tmem_ld32_issue(tmem + lanes + (uint32_t)(buf * 256 + jc), v);
                tmem_wait_ld32(v);
                if (jc + 32 * 4 >= p.nt) {  // this warp's last read of the accumulator: back to the MMA
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        if (lead)
                            mbar_arrive(&c.d_empty[buf]);
                        else
                            mbar_arrive_cluster(mapa_shared(smem_u32(&c.d_empty[buf]), 0));
                    }
                }
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    const int x = tn * p.nt + jc + kP2ZCols * hh;
                    if (lane == 0) bulk_wait_read_1();  // the store two boxes back has read this buffer
                    __syncwarp();
                    uint8_t* sb = zst + (size_t)zb * kP2ZStage;
                    zb ^= 1;
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const uint32_t* w = v + 16 * hh + 4 * u;
                        *reinterpret_cast<float4*>(sb + lane * 64 + ((u ^ ((lane >> 1) & 3)) << 4)) =
                            make_float4(rm * __uint_as_float(w[0]), rm * __uint_as_float(w[1]),
                                        rm * __uint_as_float(w[2]), rm * __uint_as_float(w[3]));
                    }
                    fence_proxy_async();
                    __syncwarp();
                    if (lane == 0) {
                        if (x < p.n && y < p.m) tma_store_2d(&tmap_c, sb, x, (int)y);
                        bulk_commit();
                    }
                }
            }
        }
        if (lane == 0) bulk_wait_all();
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync_all();  // neither CTA leaves while the other may still signal its barriers
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc2(tmem, kTmemCols);
    }
}

size_t gemm_smem_bytes(int sx, int sa, int parts, int sb) {
    return 1024 + (size_t)sx * kXStageBytes + (size_t)sa * parts * kAPartBytes + (size_t)sb * kBStageBytes +
           sizeof(Ctl);
}

bool g_attr_set[64];

// fp32 rows -> fp16 (RN), one warp per row: the row's largest magnitude a sets an exact scale 2^s
// with 2^14 <= a 2^s < 2^15, so every scaled value is inside fp16's range and the row's mass far
// above its subnormals; rowmul[row] = 2^-s undoes it in the GEMM's fp32 epilogue.  A zero row, or
// one holding a non-finite value, keeps s = 0; rows whose largest magnitude is below 2^-112 take
// the largest exact scale, 2^126.  Rows of up to 32 x 4 x kRoundRegs columns are read once into
// registers; longer rows are read twice.  (X 16-byte aligned, ldx % 4 == 0; out rows 8-byte
// aligned.)
constexpr int kRoundRegs = 8;

__device__ __forceinline__ float amax4(float a, float4 v) {
    return fmaxf(a, fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w))));
}

__device__ __forceinline__ void store_h4(__half* dst, float4 v, float sc) {
    const __half2 h0 = __floats2half2_rn(v.x * sc, v.y * sc), h1 = __floats2half2_rn(v.z * sc, v.w * sc);
    uint2 pk;
    pk.x = *reinterpret_cast<const uint32_t*>(&h0);
    pk.y = *reinterpret_cast<const uint32_t*>(&h1);
    *reinterpret_cast<uint2*>(dst) = pk;
}

__global__ void __launch_bounds__(256) k_round_f16(const float* __restrict__ X, long long ldx, long long rows,
                                                   int cols, __half* __restrict__ out, long long ldo,
                                                   float* __restrict__ rowmul) {
    const int lane = threadIdx.x & 31;
    const long long nw = (long long)gridDim.x * (blockDim.x >> 5);
    const int c4n = cols / 4;
    const bool in_regs = c4n <= 32 * kRoundRegs;
    for (long long row = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); row < rows; row += nw) {
        const float* src = X + row * ldx;
        __half* dst = out + row * ldo;
        float4 v[kRoundRegs];
        float amax = 0.f;
        if (in_regs) {
#pragma unroll
            for (int j = 0; j < kRoundRegs; ++j) {
                const int c = lane + 32 * j;
                v[j] = c < c4n ? *reinterpret_cast<const float4*>(src + 4 * c) : make_float4(0.f, 0.f, 0.f, 0.f);
                amax = amax4(amax, v[j]);
            }
        } else {
            for (int c = lane; c < c4n; c += 32) amax = amax4(amax, *reinterpret_cast<const float4*>(src + 4 * c));
        }
        const float tail = 4 * c4n + lane < cols ? src[4 * c4n + lane] : 0.f;  // cols % 4 elements
        amax = fmaxf(amax, fabsf(tail));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        int e = 0;  // 2^14 <= amax 2^e < 2^15
        if (amax > 0.f && amax <= FLT_MAX) e = min(14 - ilogbf(amax), 126);
        const float sc = __int_as_float((127 + e) << 23);
        if (in_regs) {
#pragma unroll
            for (int j = 0; j < kRoundRegs; ++j) {
                const int c = lane + 32 * j;
                if (c < c4n) store_h4(dst + 4 * c, v[j], sc);
            }
        } else {
            for (int c = lane; c < c4n; c += 32) store_h4(dst + 4 * c, *reinterpret_cast<const float4*>(src + 4 * c), sc);
        }
        if (4 * c4n + lane < cols) dst[4 * c4n + lane] = __float2half_rn(tail * sc);
        if (lane == 0) rowmul[row] = __int_as_float((127 - e) << 23);
    }
}

}  // namespace

unsigned take_device_error_gemm() {
    unsigned v = 0, z = 0;
    cudaMemcpyFromSymbol(&v, g_err_gemm, sizeof(v));
    if (v) cudaMemcpyToSymbol(g_err_gemm, &z, sizeof(z));
    return v;
}

// C = alpha A B^T (x rowmul) with fp16 A on CTA pairs (k_gemm_tc2); fp32 C, no norms, no K trimming.
static cudaError_t launch_gemm_tc2(const GemmTcArgs& a, int device, cudaStream_t s) {
    Gemm2Params q;
    q.m = a.m;
    q.n = a.n;
    q.nkb = (a.K + kBK - 1) / kBK;
    q.nt = 256;  // the pair MMA's N (each CTA stages nt / 2 rows of B; the launcher requires n >= 256)
    q.tiles_n = (a.n + q.nt - 1) / q.nt;
    q.tiles = ((a.m + 255) / 256) * (long long)q.tiles_n;
    q.sa = q.sb = kP2MaxS;
    q.C = static_cast<float*>(a.C);
    q.ldc = a.ldc;
    q.alpha = a.alpha;
    q.rowmul = a.rowmul;
    const size_t smem = 1024 + (size_t)(q.sa + q.sb) * kP2StageBytes + (size_t)kP2EpiWarps * 2 * kP2ZStage +
                        sizeof(Ctl2);
    CUtensorMap ta, tb, tc;
    if (!make_tmap_2d(&ta, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, a.A, a.m, a.K, a.lda, kBK, 128,
                      CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&tb, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, a.B0, a.n, a.K, a.ldb, kBK, q.nt / 2,
                      CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&tc, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, a.C, a.m, a.n, a.ldc, kP2ZCols, 32,
                      CU_TENSOR_MAP_SWIZZLE_64B))
        return cudaErrorInvalidValue;
    static bool attr[64];
    if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
    if (!attr[device]) {
        cudaError_t e = cudaFuncSetAttribute(k_gemm_tc2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr[device] = true;
    }
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    const long long pairs = std::min<long long>(std::max(sms / 2, 1), q.tiles);
    q.rotate = pairs % q.tiles_n == 0 ? 1 : 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(2 * pairs));
    cfg.blockDim = dim3(kP2Threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_gemm_tc2, ta, tb, tc, q);
}

cudaError_t launch_gemm_tc(const GemmTcArgs& a, int device, cudaStream_t s) {
    if (a.m <= 0 || a.n <= 0) return cudaSuccess;
    // fp16 A (T rounded once, the reconstruction): the CTA-pair kernel, whose SMs stage half of B each,
    // for products of at least one full pair tile (256 rows, 256 columns: the pair MMA is run at
    // N = 256 only, the only width its tests cover; the reconstruction needs D >= 1024 anyway)
    if (a.a_half && !a.split && !a.c_bf16 && !a.rownorm && !a.colnorm && !a.b_klo && a.m >= 256 && a.n >= 256 &&
        (uintptr_t)a.C % 16 == 0 && a.ldc % 4 == 0)  // the output's tensor map: 16-byte rows
        return launch_gemm_tc2(a, device, s);
    GemmParams p;
    p.m = a.m;
    p.n = a.n;
    p.K = a.K;
    p.nkb = (a.K + kBK - 1) / kBK;
    p.nt = a.n >= 256 ? 256 : (a.n + 31) / 32 * 32;
    // a long K with fp32 A rounded to fp16 and more than 256 columns: tiles of two column halves
    // (up to 512 columns), so each converted A K-block feeds two MMAs (half the A loads and
    // conversions per output; the single TMEM accumulator costs one epilogue per tile, small
    // against the K loop)
    const int halves = (!a.a_half && !a.split && a.n > 256 && p.nkb >= 32) ? 2 : 1;
    if (halves == 2) {
        // the columns split evenly over the wide tiles, each half rounded up to 16 (r = 922: two
        // tiles of 2 x 240 columns rather than of 2 x 256, whose last 102 columns would be padding)
        const int nw = (a.n + 511) / 512;
        p.nt = std::min(256, ((a.n + nw - 1) / nw + 31) / 32 * 16);
    }
    p.tiles_n = (a.n + p.nt * halves - 1) / (p.nt * halves);
    p.tiles = ((a.m + kBM - 1) / kBM) * (long long)p.tiles_n;
    p.amode = a.a_half ? kAF16T : a.split ? kABF16X2 : kAF16;
    p.nb = a.split ? 2 : 1;
    p.parts = a.split ? 2 : 1;
    if (a.a_half && a.split) return cudaErrorInvalidValue;
    // deepest staging that fits: two A stages, B stages for at least one K-block (+1).
    // The X depth stays even: the two converter groups take alternate K-blocks, and with
    // an even depth each X stage belongs to one group, which waits on its phases in order
    // (on an odd-depth ring a group could pass a parity test on a stage's older phase).
    const size_t cap = 227 * 1024;
    p.sa = 2;
    p.sx = 2;
    p.sb = 2 * p.nb;
    for (int sx = kMaxSX / 2 * 2; sx >= 2; sx -= 2) {
        bool done = false;
        for (int sb = kMaxSB; sb >= p.nb + 1; --sb)
            if (gemm_smem_bytes(sx, p.sa, p.parts, sb) <= cap) {
                p.sx = sx;
                p.sb = sb;
                done = true;
                break;
            }
        if (done) break;
    }
    if (p.amode == kAF16T) {  // no staging ring: the deepest A and B rings that fit
        p.sx = 0;
        p.sa = kMaxSA;
        p.sb = kMaxSB;
    }
    if (halves == 2) {  // two B boxes per K-block: B stages for two K-blocks
        p.sx = 2;
        p.sb = kMaxSB;
    }
    if (gemm_smem_bytes(p.sx, p.sa, p.parts, p.sb) > cap) return cudaErrorInvalidConfiguration;
    p.C = a.C;
    p.ldc = a.ldc;
    p.c_bf16 = a.c_bf16 ? 1 : 0;
    p.c_vec = ((uintptr_t)a.C % (a.c_bf16 ? 4 : 8) == 0) && (a.ldc % 2 == 0);
    p.alpha = a.alpha;
    p.rownorm = a.rownorm;
    p.colnorm = a.colnorm;
    p.xn2 = p.amode == kAF16 ? a.xn2_out : nullptr;
    p.rowmul = a.rowmul;
    p.krange = 0;
    if (a.b_klo && a.b_khi && p.tiles_n <= kMaxTilesN) {
        // per column tile: the K-blocks holding the tile's nonzero B entries
        p.krange = 1;
        for (int tn = 0; tn < p.tiles_n; ++tn) {
            int lo = a.K, hi = 0;
            for (int j = tn * p.nt * halves; j < std::min(a.n, (tn + 1) * p.nt * halves); ++j) {
                lo = std::min(lo, a.b_klo[j]);
                hi = std::max(hi, a.b_khi[j]);
            }
            const int kl = std::min(std::max(lo, 0), a.K) / kBK;
            p.kb_lo[tn] = std::min(kl, p.nkb - 1);
            p.kb_hi[tn] = std::min(p.nkb, std::max(p.kb_lo[tn] + 1, (hi + kBK - 1) / kBK));
        }
    }
    CUtensorMap ta, tb0, tb1;
    const CUtensorMapDataType bt = a.split ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
    const bool ta_ok = a.a_half ? make_tmap_2d(&ta, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, a.A, a.m, a.K, a.lda, kBK,
                                               kBM, CU_TENSOR_MAP_SWIZZLE_128B)
                                : make_tmap_2d(&ta, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, a.A, a.m, a.K, a.lda, kBK,
                                               kBM, CU_TENSOR_MAP_SWIZZLE_NONE);
    if (!ta_ok ||
        !make_tmap_2d(&tb0, bt, 2, a.B0, a.n, a.K, a.ldb, kBK, p.nt, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&tb1, bt, 2, a.split ? a.B1 : a.B0, a.n, a.K, a.ldb, kBK, p.nt, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    const size_t smem = gemm_smem_bytes(p.sx, p.sa, p.parts, p.sb);
    if (device >= 0 && device < 64 && !g_attr_set[device]) {
        for (auto fn : {k_gemm_tc<kAF16, 1>, k_gemm_tc<kAF16, 2>, k_gemm_tc<kABF16X2, 1>, k_gemm_tc<kAF16T, 1>}) {
            cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cap);
            if (e != cudaSuccess) return e;
        }
        g_attr_set[device] = true;
    }
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    const int grid = (int)std::min<long long>(sms > 0 ? sms : 1, p.tiles);
    p.rotate = grid % p.tiles_n == 0 ? 1 : 0;
    if (halves == 2)
        k_gemm_tc<kAF16, 2><<<grid, kThreads, smem, s>>>(ta, tb0, tb1, p);
    else if (p.amode == kAF16)
        k_gemm_tc<kAF16, 1><<<grid, kThreads, smem, s>>>(ta, tb0, tb1, p);
    else if (p.amode == kABF16X2)
        k_gemm_tc<kABF16X2, 1><<<grid, kThreads, smem, s>>>(ta, tb0, tb1, p);
    else
        k_gemm_tc<kAF16T, 1><<<grid, kThreads, smem, s>>>(ta, tb0, tb1, p);
    return cudaGetLastError();
}

}  // namespace gs

namespace gs {

cudaError_t launch_round_f16(const float* X, long long ldx, long long rows, int cols, void* out, long long ldo,
                             float* rowmul, cudaStream_t s) {
    if (rows <= 0 || cols <= 0) return cudaSuccess;
    const int grid = (int)std::min<long long>((rows + 7) / 8, 152LL * 8);  // 8 rows (warps) per block
    k_round_f16<<<grid, 256, 0, s>>>(X, ldx, rows, cols, static_cast<__half*>(out), ldo, rowmul);
    return cudaGetLastError();
}

}  // namespace gs
