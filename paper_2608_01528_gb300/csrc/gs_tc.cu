// gs_tc.cu -- tcgen05 (5th-generation tensor core) kernels for sm_103a.
//
// k_ps_tc: fused project + similarity for large query batches (paper Sec. 3.1
// t = U^T x, Sec. 2.2 scaled dot-product similarity, Sec. 3.2 Eq. 2-3), for
// bases with r <= 256 and codebooks with M <= 256.
//
//   GEMM1  Y = X Q^T   tcgen05.mma kind::f16, M = 128 queries, N = r,
//                      fp32 accumulator in TMEM columns [0, 256).
//                      A = X: fp32 tiles streamed from HBM by TMA into a staging
//                      ring (several 32 KB tiles in flight per SM), rounded to
//                      fp16 (RN) by converter warps into the 128-byte-swizzled
//                      K-major layout the MMA reads.
//                      B = Q: the basis' fixed fp16 copy (dithered rounding, see
//                      gs_build.cu), fetched per K-block by TMA (L2-resident).
//   GEMM2  S = Y R^T   tcgen05.mma kind::f16 with bf16 operands split in two,
//                      Y = Yh + Yl and R = Rh + Rl, S = Yh Rh + Yl Rh + Yh Rl
//                      (relative error ~2^-16, fp32's exponent range), fp32
//                      accumulator in TMEM columns [256, 512).  The epilogue
//                      splits Y in place in TMEM (each 16-column fp32 chunk
//                      becomes 8 columns of packed Yh and 8 of packed Yl), and
//                      the MMA reads that A operand straight from TMEM.  S runs
//                      in halves of up to 128 codewords; one B-ring slot holds
//                      one K-block of both Rh and Rl of a half, so each slot is
//                      consumed on its own and the next one loads meanwhile.
//                      Gram-Schmidt leaves R lower echelon (codeword i has no
//                      component past the basis vectors built before it), so a
//                      half stops at the K-block holding its last nonzero.
//                      A single fp16/tf32 rounding would not do here: the
//                      dominant terms of S are single products Y_i R_ii.
//   epilogue           scale / cosine (full-D ||x|| accumulated by the
//                      converters from the fp32 input) / online softmax, argmax
//                      (lowest index on ties), maxval, optional Y and S stores.
//
// Why the X tiles go through TMA rather than through registers: a thread that
// signals "A stage full" with an mbarrier arrive (a release) cannot complete
// that arrive while its own prefetched global loads are still in flight, so a
// register-prefetch loader serialises on one memory round trip per K-block.
// With TMA the bytes in flight are the hardware's, and the converters' release
// only orders shared-memory traffic.
//
// Work split: one persistent CTA per SM; each CTA takes a contiguous, balanced
// range of rows and cuts it into tiles of at most 128 rows, so every CTA moves
// the same number of bytes.  Warp roles (480 threads):
//   warps 0-3    epilogue: warp w owns TMEM lanes 32w..32w+31 (rows of the tile)
//   warp  4      TMA producer of the X tiles
//   warp  5      TMEM allocator and MMA issuer (one elected lane)
//   warp  6      TMA producer of the B operand tiles (Q per K-block, then Rh / Rl)
//   warps 7-14   converters (fp32 -> fp16, row norms, range check), two groups of
//                four warps taking alternate K-blocks so two blocks convert at once
// Every wait on an mbarrier is bounded (wall-clock limit): on expiry the CTA
// records GS_DEV_ERR_TIMEOUT, raises a CTA-wide abort flag so the other roles
// leave their loops, waits (bounded) for its own TMA copies and MMAs to land,
// frees TMEM and returns.

#include <float.h>

#include <algorithm>
#include <vector>

#include "gs_internal.h"
#include "gs_tc_ptx.cuh"

namespace gs {
namespace {

using namespace ptx;

__device__ unsigned g_err_tc = 0;

constexpr int kBM = 128;             // queries per tile (MMA M)
constexpr int kBK = 64;              // K elements per block (fp16 A row = 128 B, fp32 staging row = 256 B)
constexpr int kEpiWarps = 4;
constexpr int kXWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kBWarp = 6;
constexpr int kCvt0 = 7;
constexpr int kCvtGroups = 2;        // converter groups take alternate K-blocks
constexpr int kCvtGroupWarps = 4;
constexpr int kCvtWarps = kCvtGroups * kCvtGroupWarps;
constexpr int kThreads = (kCvt0 + kCvtWarps) * 32;  // 480
constexpr int kCvtThreads = kCvtGroupWarps * 32;     // 128 per group
constexpr int kCvtRowStep = kCvtThreads / 16;        // 8 rows per sweep of the 16 float4 columns
constexpr int kCvtRows = kBM / kCvtRowStep;          // 16 rows per converter thread
constexpr int kAStageBytes = kBM * kBK * 2;          // 16 KB fp16 operand tile
constexpr int kBStageBytes = 256 * kBK * 2;          // 32 KB: up to 256 rows of one B operand K-block
constexpr int kMaxSX = 6, kMaxSA = 2, kMaxSB = 4;
constexpr int kTmemCols = 512;
constexpr int kMaxKR = 4;            // K-blocks of 64 in r <= 256
constexpr int kSCol = 256;           // first TMEM column of the score accumulator

// ----------------------------------------------------------------- work split
struct TileRange {
    long long row0;
    int nrows;
};

// Balanced contiguous row range of CTA c, cut into tiles of at most 128 rows.
struct CtaRows {
    long long rb;
    long long rows;
    int ntiles;
    int tsize;
    __host__ __device__ CtaRows(long long N, int G, int c) {
        const long long base = N / G, rem = N % G;
        rows = base + (c < rem ? 1 : 0);
        rb = (long long)c * base + (c < rem ? c : rem);
        ntiles = (int)((rows + kBM - 1) / kBM);
        tsize = ntiles ? (int)((rows + ntiles - 1) / ntiles) : 0;
    }
    __host__ __device__ TileRange tile(int t) const {
        TileRange tr;
        tr.row0 = rb + (long long)t * tsize;
        const long long left = rb + rows - tr.row0;
        tr.nrows = (int)(left < tsize ? left : tsize);
        return tr;
    }
};

struct PsParams {
    long long N;
    int D, r, npad, M, mpad, nkb;
    int nh, half_rows, nkr_h[2];  // GEMM2: halves of codewords, K-blocks of R each half needs
    int sx, sa, sb;         // ring depths: fp32 X staging, fp16 A, B operand tiles
    int box_rows;           // rows of each X TMA box (>= every tile's rows)
    int xstage;             // bytes between X staging tiles (box_rows x 256, 1 KB aligned)
    float xn2_lo, xn2_hi;   // rows with ||x||^2 outside [lo, hi] (and > 0) are redone scaled
    const float* cnorm;     // M
    int mode;
    float scale;
    float* Y;
    int ldy;
    float* S;
    int lds;
    int* argmax;
    float* maxval;
};

struct Ctl {
    uint64_t x_full[kMaxSX], x_empty[kMaxSX];
    uint64_t a_full[kMaxSA], a_empty[kMaxSA];
    uint64_t b_full[kMaxSB], b_empty[kMaxSB];
    uint64_t y_full, s_full, s_empty, gemm2_done;
    uint64_t ysplit[kMaxKR];  // Y columns [64 k, 64 k + 64) split in TMEM (GEMM2 K-block k may start)
    uint64_t xn_full[2], xn_empty[2];
    uint64_t dec_full[2];     // redo decision of regular tile t published in slot t % 2
    uint64_t mma_done;
    float xn[2][kBM];  // ||x||^2 per row, both converter groups add into it
    int8_t rsc[2][kBM];      // per-row exponent s of the redo's scale 2^s, for the tile in that slot
    int redo[2][kEpiWarps];  // per epilogue warp: some row of its lane quadrant needs the redo
    uint32_t tmem_base;
    int abort_flag;
};

// Exact power of two 2^k (|k| <= 126).
__device__ __forceinline__ float pow2f(int k) { return __int_as_float((127 + k) << 23); }

// The exponent s that brings a row of squared norm xn2 to 2^14 <= ||x|| 2^s < 2^15: every
// element then lies below 2^15 (inside fp16's range) and the row's mass far above fp16's
// subnormals.  s lies in [-49, 89] for any finite positive fp32 xn2; rows whose squared norm is
// not a finite positive number keep s = 0.
__device__ __forceinline__ int row_scale_exp(float xn2) {
    if (!(xn2 > 0.f) || !(xn2 <= FLT_MAX)) return 0;
    return 14 - (ilogbf(xn2) >> 1);  // ilogbf(xn2) >> 1 = floor(log2 ||x||)
}

// Processing order of a CTA's tiles: regular tile t, and once tile t + 1 has been handed on, the
// redo of tile t when its epilogue asked for one (the decision is published in slot t % 2, so it
// is always known by then and nobody waits on it in the common case).  body(t, redo, q) runs one
// tile; q counts processed tiles (the per-tile barrier phases and the norm buffers follow it).
// wait(bar, parity) is the role's bounded wait.  Returns false when a wait or the body gave up.
template <class Wait, class Body>
__device__ __forceinline__ bool walk_tiles(const CtaRows& cr, Ctl& c, Wait wait, Body body) {
    int q = 0;
    for (int t = 0; t <= cr.ntiles; ++t) {
        if (t < cr.ntiles && !body(t, false, q++)) return false;
        if (t >= 1) {
            const int d = t - 1, slot = d & 1;
            if (!wait(&c.dec_full[slot], (uint32_t)(d >> 1) & 1u)) return false;
            const volatile int* rd = c.redo[slot];
            bool again = false;
#pragma unroll
            for (int w = 0; w < kEpiWarps; ++w) again |= rd[w] != 0;
            if (again && !body(d, true, q++)) return false;
        }
    }
    return true;
}

// FULL = false: raw scores with only argmax / maxval out (the large-batch lookup); true: every
// mode and output.  A template parameter, so the lookup kernel carries none of the other paths.
template <bool FULL>
__global__ void __launch_bounds__(kThreads, 1)
    k_ps_tc(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ CUtensorMap tmap_q,
            const __grid_constant__ CUtensorMap tmap_rh, const __grid_constant__ CUtensorMap tmap_rl,
            const PsParams p) {
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte aligned operand area (SW128 atoms), control block after it
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    uint8_t* Xs = base;
    uint8_t* As = Xs + (size_t)p.sx * p.xstage;
    uint8_t* Bs = As + (size_t)p.sa * kAStageBytes;
    Ctl& c = *reinterpret_cast<Ctl*>(Bs + (size_t)p.sb * kBStageBytes);
    volatile int* abort_flag = &c.abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const CtaRows cr(p.N, gridDim.x, blockIdx.x);

    if (threadIdx.x == 0) {
        for (int s = 0; s < p.sx; ++s) {
            mbar_init(&c.x_full[s], 1);
            mbar_init(&c.x_empty[s], kCvtGroupWarps);
        }
        for (int s = 0; s < p.sa; ++s) {
            mbar_init(&c.a_full[s], kCvtGroupWarps);
            mbar_init(&c.a_empty[s], 1);
        }
        for (int s = 0; s < p.sb; ++s) {
            mbar_init(&c.b_full[s], 1);
            mbar_init(&c.b_empty[s], 1);
        }
        mbar_init(&c.y_full, 1);
        for (int k = 0; k < kMaxKR; ++k) mbar_init(&c.ysplit[k], kEpiWarps);
        mbar_init(&c.s_full, 1);
        mbar_init(&c.s_empty, kEpiWarps);
        mbar_init(&c.gemm2_done, 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(&c.xn_full[b], kCvtWarps);
            mbar_init(&c.xn_empty[b], kEpiWarps);
            mbar_init(&c.dec_full[b], kEpiWarps);
        }
        mbar_init(&c.mma_done, 1);
        c.abort_flag = 0;
        for (int j = 0; j < 2 * kBM; ++j) (&c.xn[0][0])[j] = 0.f;
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
    auto wait_1t = [&](uint64_t* bar, uint32_t par) { return mbar_wait_1t(bar, par, abort_flag, &g_err_tc); };
    auto wait_warp = [&](uint64_t* bar, uint32_t par) { return mbar_wait_warp(bar, par, abort_flag, &g_err_tc); };

    if (warp == kXWarp) {
        // ------------------------------------------------------------- X tiles via TMA
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_first();
            const uint32_t bytes = (uint32_t)p.box_rows * kBK * 4;
            int it = 0;
            RingPos xs;
            walk_tiles(cr, c, wait_1t, [&](int t, bool, int) {
                const TileRange tr = cr.tile(t);
                for (int kb = 0; kb < p.nkb; ++kb, ++it, xs.next(p.sx)) {
                    if (!wait_1t(&c.x_empty[xs.idx], xs.phase ^ 1u)) return false;
                    mbar_arrive_expect_tx(&c.x_full[xs.idx], bytes);
                    tma_load_2d(Xs + (size_t)xs.idx * p.xstage, &tmap_x, &c.x_full[xs.idx], kb * kBK, (int)tr.row0,
                                pol);
                }
                return true;
            });
            // every copy this thread started lands before the CTA can exit
            for (int j = std::max(0, it - p.sx); j < it; ++j) mbar_drain(&c.x_full[j % p.sx], (uint32_t)(j / p.sx) & 1u, &g_err_tc);
        }
    } else if (warp == kBWarp) {
        // ------------------------------------------------------------- B operand tiles via TMA:
        // per tile, nkb Q tiles (GEMM1), then per half of the codewords its K-blocks of
        // Rh and Rl, both in one slot (GEMM2)
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_last();
            const uint32_t qbytes = (uint32_t)p.npad * kBK * 2, rbytes = 2u * (uint32_t)p.half_rows * kBK * 2;
            const uint32_t rl_off = (uint32_t)p.half_rows * kBK * 2;  // Rl after Rh in the slot
            const int per_tile = p.nkb + p.nkr_h[0] + p.nkr_h[1];
            int it = 0;
            RingPos bs;
            walk_tiles(cr, c, wait_1t, [&](int, bool, int) {
                for (int k = 0; k < per_tile; ++k, ++it, bs.next(p.sb)) {
                    const int s = bs.idx;
                    if (!wait_1t(&c.b_empty[s], bs.phase ^ 1u)) return false;
                    uint8_t* dst = Bs + (size_t)s * kBStageBytes;
                    if (k < p.nkb) {
                        mbar_arrive_expect_tx(&c.b_full[s], qbytes);
                        tma_load_2d(dst, &tmap_q, &c.b_full[s], k * kBK, 0, pol);
                    } else {
                        const int j = k - p.nkb;
                        const int h = j < p.nkr_h[0] ? 0 : 1;
                        const int kr = h ? j - p.nkr_h[0] : j;
                        mbar_arrive_expect_tx(&c.b_full[s], rbytes);
                        tma_load_2d(dst, &tmap_rh, &c.b_full[s], kr * kBK, h * p.half_rows, pol);
                        tma_load_2d(dst + rl_off, &tmap_rl, &c.b_full[s], kr * kBK, h * p.half_rows, pol);
                    }
                }
                return true;
            });
            for (int j = std::max(0, it - p.sb); j < it; ++j) mbar_drain(&c.b_full[j % p.sb], (uint32_t)(j / p.sb) & 1u, &g_err_tc);
        }
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc1 = idesc_f16_f32(p.npad);
            const uint32_t idesc2 = idesc_bf16_f32(p.half_rows);
            const uint32_t y_tmem = tmem, s_tmem = tmem + kSCol;
            RingPos ra, rb;
            walk_tiles(cr, c, wait_1t, [&](int, bool, int q) {
                const uint32_t pt = (uint32_t)q & 1u;
                // GEMM1: Y = X Q^T into columns [0, npad)
                for (int kb = 0; kb < p.nkb; ++kb, ra.next(p.sa), rb.next(p.sb)) {
                    const int sa = ra.idx, sb = rb.idx;
                    if (!wait_1t(&c.a_full[sa], ra.phase) || !wait_1t(&c.b_full[sb], rb.phase)) return false;
                    tc_fence_after();
                    const uint64_t ad = sdesc_sw128(smem_u32(As + (size_t)sa * kAStageBytes));
                    const uint64_t bd = sdesc_sw128(smem_u32(Bs + (size_t)sb * kBStageBytes));
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k)
                        mma_f16_ss(y_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc1,
                                   (kb | k) != 0 ? 1u : 0u);
                    mma_commit(&c.a_empty[sa]);
                    mma_commit(&c.b_empty[sb]);
                }
                mma_commit(&c.y_full);
                // GEMM2: S = Yh Rh + Yl Rh + Yh Rl into columns [256, 256 + mpad), once the
                // epilogue has split Y in place and released the previous tile's S
                if (!wait_1t(&c.s_empty, pt ^ 1u)) return false;
                int nsplit = 0;  // K-blocks of Y known to be split; the epilogue signals each one
                for (int h = 0; h < p.nh; ++h) {
                    const uint32_t s_half = s_tmem + (uint32_t)(h * p.half_rows);
                    for (int kr = 0; kr < p.nkr_h[h]; ++kr, rb.next(p.sb)) {
                        for (; nsplit <= kr; ++nsplit)
                            if (!wait_1t(&c.ysplit[nsplit], pt)) return false;
                        const int sr = rb.idx;
                        if (!wait_1t(&c.b_full[sr], rb.phase)) return false;
                        tc_fence_after();
                        const uint32_t rs = smem_u32(Bs + (size_t)sr * kBStageBytes);
                        const uint64_t rh = sdesc_sw128(rs);
                        const uint64_t rl = sdesc_sw128(rs + (uint32_t)p.half_rows * kBK * 2);
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            // r columns [64 kr + 16 k, +16) were split into TMEM columns
                            // [16 kk, 16 kk + 8) (Yh) and [16 kk + 8, 16 kk + 16) (Yl), kk = 4 kr + k
                            const int kk = 4 * kr + k;
                            if (16 * kk >= p.npad) break;  // past r: no split columns there
                            const uint32_t a_hi = y_tmem + (uint32_t)(16 * kk);
                            const uint32_t a_lo = a_hi + 8;
                            mma_bf16_ts(s_half, a_hi, rh + (uint64_t)(2 * k), idesc2, (kr | k) != 0 ? 1u : 0u);
                            mma_bf16_ts(s_half, a_lo, rh + (uint64_t)(2 * k), idesc2, 1u);
                            mma_bf16_ts(s_half, a_hi, rl + (uint64_t)(2 * k), idesc2, 1u);
                        }
                        mma_commit(&c.b_empty[sr]);
                    }
                }
                mma_commit(&c.s_full);
                // the next tile's GEMM1 overwrites the columns GEMM2 reads: wait for it to finish
                mma_commit(&c.gemm2_done);
                if (!wait_1t(&c.gemm2_done, pt)) return false;
                tc_fence_after();
                return true;
            });
            // all MMAs issued by this thread complete before TMEM is released
            mma_commit(&c.mma_done);
            mbar_drain(&c.mma_done, 0, &g_err_tc);
        }
    } else if (warp >= kCvt0) {
        // ------------------------------------------------------------- converters
        const int g = (warp - kCvt0) / kCvtGroupWarps;           // group: K-blocks with it % 2 == g
        const int l = threadIdx.x - (kCvt0 + g * kCvtGroupWarps) * 32;  // 0..127 within the group
        const int c4 = l & 15;                   // float4 column of the 64-wide K-block
        const int rbase = l >> 4;                // rows rbase + 8u, u < 16
        float nrm[kCvtRows];
#pragma unroll
        for (int u = 0; u < kCvtRows; ++u) nrm[u] = 0.f;
        float amax = 0.f;
        int it = 0;
        RingPos rx, ra;  // every K-block advances both rings; this group takes those with it % 2 == g
        walk_tiles(cr, c, wait_warp, [&](int t, bool redo, int q) {
            const TileRange tr = cr.tile(t);
            const int b = q & 1;
            const int8_t* rs = c.rsc[t & 1];  // the rows' scale exponents (redo only)
            for (int kb = 0; kb < p.nkb; ++kb, ++it, rx.next(p.sx), ra.next(p.sa)) {
                if ((it & 1) != g) continue;
                const int sx = rx.idx, sa = ra.idx;
                if (!wait_warp(&c.x_full[sx], rx.phase) || !wait_warp(&c.a_empty[sa], ra.phase ^ 1u)) return false;
                const uint8_t* Xt = Xs + (size_t)sx * p.xstage;
                uint8_t* At = As + (size_t)sa * kAStageBytes;
#pragma unroll
                for (int u = 0; u < kCvtRows; ++u) {
                    const int row = rbase + kCvtRowStep * u;
                    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (row < tr.nrows) x = *reinterpret_cast<const float4*>(Xt + row * (kBK * 4) + c4 * 16);
                    if (redo) {  // exact power-of-two scale: the fp16 rounding below loses nothing to range
                        const float sc = pow2f(rs[row]);
                        x.x *= sc;
                        x.y *= sc;
                        x.z *= sc;
                        x.w *= sc;
                        amax = fmaxf(amax, fmaxf(fmaxf(fabsf(x.x), fabsf(x.y)), fmaxf(fabsf(x.z), fabsf(x.w))));
                    }
                    nrm[u] = fmaf(x.x, x.x, fmaf(x.y, x.y, fmaf(x.z, x.z, fmaf(x.w, x.w, nrm[u]))));
                    const __half2 h0 = __floats2half2_rn(x.x, x.y);
                    const __half2 h1 = __floats2half2_rn(x.z, x.w);
                    uint2 pk;
                    pk.x = *reinterpret_cast<const uint32_t*>(&h0);
                    pk.y = *reinterpret_cast<const uint32_t*>(&h1);
                    const int chunk = (c4 >> 1) ^ (row & 7);
                    *reinterpret_cast<uint2*>(At + row * 128 + chunk * 16 + (c4 & 1) * 8) = pk;
                }
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&c.a_full[sa]);
                    mbar_arrive(&c.x_empty[sx]);
                }
            }
            // tile finished: this group's part of ||x||^2 of each row is added into shared memory
#pragma unroll
            for (int u = 0; u < kCvtRows; ++u) {
                float v = nrm[u];
                v += __shfl_xor_sync(0xffffffffu, v, 8);
                v += __shfl_xor_sync(0xffffffffu, v, 4);
                v += __shfl_xor_sync(0xffffffffu, v, 2);
                v += __shfl_xor_sync(0xffffffffu, v, 1);
                nrm[u] = v;
            }
            if (!wait_warp(&c.xn_empty[b], ((uint32_t)(q >> 1) & 1u) ^ 1u)) return false;
            if ((lane & 15) == 0) {
#pragma unroll
                for (int u = 0; u < kCvtRows; ++u) atomicAdd(&c.xn[b][rbase + kCvtRowStep * u], nrm[u]);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.xn_full[b]);
#pragma unroll
            for (int u = 0; u < kCvtRows; ++u) nrm[u] = 0.f;
            return true;
        });
        // only a redone row can still leave fp16's range (a norm that is not a finite fp32 number)
        if (amax > 65504.f) atomicOr(&g_err_tc, GS_DEV_ERR_RANGE);
    } else {
        // ------------------------------------------------------------- epilogue (warps 0-3)
        const int i = threadIdx.x;  // row within the tile = TMEM lane
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        const uint32_t ty = tmem + lane_base, ts = tmem + lane_base + kSCol;
        walk_tiles(cr, c, wait_warp, [&](int t, bool redo, int q) {
            const uint32_t pt = (uint32_t)q & 1u;
            const int b = q & 1;
            if (!wait_warp(&c.y_full, pt)) return false;
            tc_fence_after();
            const TileRange tr = cr.tile(t);
            const bool valid = i < tr.nrows;
            const long long row = tr.row0 + i;
            // a redone tile ran on x 2^s: Y and ||x|| come back multiplied by 2^s
            const float unscale = redo ? pow2f(-c.rsc[t & 1][i]) : 1.f;
            // split Y in place: chunk of 16 fp32 columns -> 8 columns bf16(Y) + 8 columns
            // bf16(Y - bf16(Y)), read 32 columns per TMEM load wait.  Each finished K-block
            // of 64 columns is signalled on its own, so GEMM2 starts on it while the rest
            // of Y is still being split.
            for (int jc = 0; jc < p.npad; jc += 32) {
                const int w = p.npad - jc >= 32 ? 32 : 16;
                float y[32];
                if (w == 32)
                    tmem_ld32(ty + (uint32_t)jc, y);
                else
                    tmem_ld16(ty + (uint32_t)jc, y);
                if (redo) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) y[j] *= unscale;
                }
                if (FULL && p.Y && valid) {
                    float* dst = p.Y + (size_t)row * p.ldy + jc;
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < w && jc + j < p.r) dst[j] = y[j];
                }
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    if (h * 16 >= w) break;
                    uint32_t hl[16];  // 8 columns of packed hi, then 8 of packed lo
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const float a = y[16 * h + 2 * j], bb = y[16 * h + 2 * j + 1];
                        const float ah = __bfloat162float(__float2bfloat16_rn(a));
                        const float bh = __bfloat162float(__float2bfloat16_rn(bb));
                        hl[j] = pack_bf16(ah, bh);
                        hl[8 + j] = pack_bf16(a - ah, bb - bh);
                    }
                    tmem_st16(ty + (uint32_t)(jc + 16 * h), hl);
                }
                if (((jc + 32) & 63) == 0 || jc + 32 >= p.npad) {  // K-block jc / 64 is split
                    tmem_wait_st();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&c.ysplit[jc >> 6]);
                }
            }
            if (!wait_warp(&c.xn_full[b], (uint32_t)(q >> 1) & 1u)) return false;
            const float xn2 = c.xn[b][i];
            c.xn[b][i] = 0.f;  // ready for the tile after next (both groups add into it)
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.xn_empty[b]);
            const float xnorm = sqrtf(xn2) * unscale;
            if (!redo) {
                // one fp16 rounding of x is accurate when every element is inside fp16's range
                // (||x|| <= 2^15) and the row's mass is far above its subnormals (||x|| >= 2^-8
                // sqrt(D): the subnormals' absolute errors, at most 2^-25 each, then add at most
                // 2^-19 ||x|| to the error of <x, q_j>); any other nonzero row has its tile redone
                // with an exact power-of-two scale (a norm that is not a number keeps scale 1)
                const bool bad = xn2 > 0.f && !(xn2 >= p.xn2_lo && xn2 <= p.xn2_hi);
                const int slot = t & 1;
                c.rsc[slot][i] = (int8_t)row_scale_exp(xn2);
                const unsigned any = __ballot_sync(0xffffffffu, bad);
                if (lane == 0) c.redo[slot][warp] = any != 0u;
                __syncwarp();
                if (lane == 0) mbar_arrive(&c.dec_full[slot]);
            }
            if (!wait_warp(&c.s_full, pt)) return false;
            tc_fence_after();
            float best = -FLT_MAX, run_max = -FLT_MAX, run_sum = 0.f;
            int besti = 0;
            for (int ic = 0; ic < p.mpad; ic += 16) {
                float sv[16];
                tmem_ld16(ts + (uint32_t)ic, sv);
                if (p.nkr_h[ic >= p.half_rows ? 1 : 0] == 0) {  // a half with no nonzero R: S = 0
#pragma unroll
                    for (int j = 0; j < 16; ++j) sv[j] = 0.f;
                }
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int ci = ic + j;
                    if (ci >= p.M) break;
                    float g = p.scale * sv[j];
                    if (FULL && p.mode == GS_SCORE_COSINE) {
                        const float den = xnorm * p.cnorm[ci];
                        g = den > 0.f ? g / den : 0.f;
                    }
                    if (g > best) {
                        best = g;
                        besti = ci;
                    }
                    if (FULL && p.mode == GS_SCORE_SOFTMAX) {
                        const float nm = fmaxf(run_max, g);
                        run_sum = run_sum * __expf(run_max - nm) + __expf(g - nm);
                        run_max = nm;
                    }
                    if (FULL && p.S && valid) p.S[(size_t)row * p.lds + ci] = g;
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.s_empty);
            if (!valid) return true;
            float outmax = best;
            if (FULL && p.mode == GS_SCORE_SOFTMAX) {
                const float inv = 1.f / run_sum;
                outmax = __expf(best - run_max) * inv;
                if (p.S) {
                    float* sr = p.S + (size_t)row * p.lds;
                    for (int ci = 0; ci < p.M; ++ci) sr[ci] = __expf(sr[ci] - run_max) * inv;
                }
            }
            if (p.argmax) p.argmax[row] = besti;
            if (p.maxval) p.maxval[row] = outmax;
            return true;
        });
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ----------------------------------------------------------------- host side
// R (M x r fp32) -> Rh = bf16(R), Rl = bf16(R - Rh) (mpad x npad) and the same
// split of R^T (npad x mpad), all zero padded.
__global__ void k_split_r(const float* __restrict__ R, int M, int r, int ldr, __nv_bfloat16* __restrict__ Rh,
                          __nv_bfloat16* __restrict__ Rl, __nv_bfloat16* __restrict__ Rth,
                          __nv_bfloat16* __restrict__ Rtl, int mpad, int npad) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)mpad * npad) return;
    const int i = (int)(idx / npad), j = (int)(idx % npad);
    const float v = (i < M && j < r) ? R[(size_t)i * ldr + j] : 0.f;
    const __nv_bfloat16 hv = __float2bfloat16_rn(v);
    const __nv_bfloat16 lv = __float2bfloat16_rn(v - __bfloat162float(hv));
    Rh[idx] = hv;
    Rl[idx] = lv;
    Rth[(size_t)j * mpad + i] = hv;
    Rtl[(size_t)j * mpad + i] = lv;
}

// Q (r x D fp32, ld = D) -> Qh = bf16(Q), Ql = bf16(Q - Qh), both r x ldq, zero padded.
__global__ void k_split_q(const float* __restrict__ Q, int r, int D, int ldq, __nv_bfloat16* __restrict__ Qh,
                          __nv_bfloat16* __restrict__ Ql) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)r * ldq) return;
    const int j = (int)(idx / ldq), d = (int)(idx % ldq);
    const float v = d < D ? Q[(size_t)j * D + d] : 0.f;
    const __nv_bfloat16 hv = __float2bfloat16_rn(v);
    Qh[idx] = hv;
    Ql[idx] = __float2bfloat16_rn(v - __bfloat162float(hv));
}

int num_sms(int dev) {
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

struct Rings {
    int sx, sa, sb;
};

constexpr size_t kSmemCap = 227 * 1024;

// bytes between fp32 X staging tiles of `box_rows` rows (SW128 operand areas follow: 1 KB aligned)
int ps_xstage(int box_rows) { return (box_rows * kBK * 4 + 1023) / 1024 * 1024; }

size_t ps_smem_bytes(Rings g, int xstage) {
    return 1024 + (size_t)g.sx * xstage + (size_t)g.sa * kAStageBytes + (size_t)g.sb * kBStageBytes + sizeof(Ctl);
}

// Ring depths for X boxes of `box_rows` rows: the deepest X ring that fits, then the
// deepest B ring.  The X depth must be even.  The two converter groups take alternate
// K-blocks, so with an even depth every X stage belongs to one group, which waits on its
// phases in order.  With an odd depth a stage alternates between the groups: one group
// can reach the stage two phases on while the other group's load into it is still in
// flight (TMA loads may land out of order), and the parity test would then pass on the
// stage's older, completed phase and hand over stale data.
Rings ps_rings(int box_rows) {
    const int xs = ps_xstage(box_rows);
    for (int sx = kMaxSX; sx >= 2; sx -= 2)
        for (int sb = kMaxSB; sb >= 2; --sb) {
            Rings g{sx, kMaxSA, sb};
            if (ps_smem_bytes(g, xs) <= kSmemCap) return g;
        }
    return Rings{2, kMaxSA, 2};
}

}  // namespace

namespace {
// Self-test of the bounded waits: one thread waits, through the same mbar_wait the
// tensor-core kernels use, on an mbarrier that nothing ever arrives on.  The wait gives up
// after its limit, records GS_DEV_ERR_TIMEOUT in this file's device word and returns.
__global__ void k_wait_selftest() {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) mbar_wait(&bar, 0u, &abort_flag, &g_err_tc);  // phase 0 never completes
}
}  // namespace

cudaError_t launch_wait_selftest(cudaStream_t s) {
    k_wait_selftest<<<1, 32, 0, s>>>();
    return cudaGetLastError();
}

unsigned take_device_error_tc() {
    unsigned v = 0, z = 0;
    cudaMemcpyFromSymbol(&v, g_err_tc, sizeof(v));
    if (v) cudaMemcpyToSymbol(g_err_tc, &z, sizeof(z));
    return v;
}

bool tc_available(int device) {
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, device);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, device);
    return major == 10 && minor == 3 && encode_fn() != nullptr;
}

gs_status tc_prepare(gs_basis* h) {
    if (h->r < 1) return GS_OK;
    const int npad = (h->r + 15) / 16 * 16;
    const int mpad = (h->M + 15) / 16 * 16;
    const size_t n = (size_t)mpad * npad;
    // bf16 hi / lo splits of R (mpad x npad) and of R^T (npad x mpad)
    for (void** ptr : {&h->tc_Rh, &h->tc_Rl, &h->tc_Rth, &h->tc_Rtl})
        if (cudaMalloc(ptr, sizeof(__nv_bfloat16) * n) != cudaSuccess) return GS_ERR_NOMEM;
    k_split_r<<<(unsigned)((n + 255) / 256), 256>>>(h->R, h->M, h->r, h->ldr, (__nv_bfloat16*)h->tc_Rh,
                                                    (__nv_bfloat16*)h->tc_Rl, (__nv_bfloat16*)h->tc_Rth,
                                                    (__nv_bfloat16*)h->tc_Rtl, mpad, npad);
    // bf16 hi / lo split of Q (r x ldq16, zero padded)
    const size_t nq = (size_t)h->r * h->ldq16;
    for (void** ptr : {&h->tc_Qh, &h->tc_Ql})
        if (cudaMalloc(ptr, sizeof(__nv_bfloat16) * nq) != cudaSuccess) return GS_ERR_NOMEM;
    k_split_q<<<(unsigned)((nq + 255) / 256), 256>>>(h->Q, h->r, h->D, h->ldq16, (__nv_bfloat16*)h->tc_Qh,
                                                     (__nv_bfloat16*)h->tc_Ql);
    if (cudaGetLastError() != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) return GS_ERR_CUDA;
    h->tc_npad = npad;
    h->tc_mpad = mpad;
    h->has_split = true;
    // R's echelon structure on the host, for the GEMMs' K trimming
    h->rlen_host.assign((size_t)h->M, 0);
    if (cudaMemcpy(h->rlen_host.data(), h->rlen, sizeof(int) * (size_t)h->M, cudaMemcpyDeviceToHost) != cudaSuccess)
        return GS_ERR_CUDA;
    h->kzero_host.assign((size_t)h->M, 0);
    h->kM_host.assign((size_t)h->r, h->M);
    h->pivot_host.assign((size_t)h->r, h->M);
    for (int j = 0, i = 0; j < h->r; ++j) {  // first row reaching column j (nondecreasing in j)
        while (i < h->M && h->rlen_host[(size_t)i] <= j) ++i;
        h->pivot_host[(size_t)j] = i;
    }
    // the fused kernel keeps Y (r <= 256 columns) and S (M <= 256 columns) in TMEM
    if (h->r > 256 || h->M > 256) return GS_OK;
    // GEMM2 halves: up to 128 codewords each; K-blocks per half from the last nonzero of R
    h->tc_half_rows = mpad > 128 ? 128 : mpad;
    h->tc_nh = (mpad + h->tc_half_rows - 1) / h->tc_half_rows;
    {
        std::vector<int> rl((size_t)h->M);
        if (cudaMemcpy(rl.data(), h->rlen, sizeof(int) * (size_t)h->M, cudaMemcpyDeviceToHost) != cudaSuccess)
            return GS_ERR_CUDA;
        for (int hh = 0; hh < 2; ++hh) {
            int last = 0;
            for (int i = hh * h->tc_half_rows; hh < h->tc_nh && i < std::min(h->M, (hh + 1) * h->tc_half_rows); ++i)
                last = std::max(last, rl[(size_t)i]);
            h->tc_nkr_half[hh] = (last + kBK - 1) / kBK;
        }
    }
    if (!make_tmap_2d(&h->tmap_q16, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, h->Q16, h->r, h->D, h->ldq16, kBK, npad,
                      CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&h->tmap_rh, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, h->tc_Rh, mpad, npad, npad, kBK,
                      h->tc_half_rows, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&h->tmap_rl, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, h->tc_Rl, mpad, npad, npad, kBK,
                      h->tc_half_rows, CU_TENSOR_MAP_SWIZZLE_128B))
        return GS_ERR_CUDA;
    if (cudaFuncSetAttribute(k_ps_tc<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemCap) !=
            cudaSuccess ||
        cudaFuncSetAttribute(k_ps_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemCap) !=
            cudaSuccess)
        return GS_ERR_CUDA;
    // the fused kernel needs all of its threads resident in one CTA; otherwise the
    // basis simply has no fused tensor-core similarity path
    cudaFuncAttributes fa, fb;
    if (cudaFuncGetAttributes(&fa, k_ps_tc<false>) != cudaSuccess ||
        cudaFuncGetAttributes(&fb, k_ps_tc<true>) != cudaSuccess)
        return GS_ERR_CUDA;
    h->has_tmap_q16 = fa.maxThreadsPerBlock >= kThreads && fb.maxThreadsPerBlock >= kThreads;
    return GS_OK;
}

cudaError_t launch_ps_tc(const gs_basis* h, const float* X, long long N, int ldx, int mode, float scale, float* Y,
                         int ldy, float* S, int lds, int* argmax, float* maxval, cudaStream_t s) {
    if (!h->has_tmap_q16) return cudaErrorNotSupported;
    const long long tiles = (N + kBM - 1) / kBM;
    const int grid = (int)std::min<long long>(num_sms(h->device), tiles);
    // the X box must cover the largest tile of any CTA (CTAs differ by one row)
    int box_rows = 1;
    for (int cta : {0, grid - 1}) box_rows = std::max(box_rows, CtaRows(N, grid, cta).tsize);
    CUtensorMap tmx;
    if (!make_tmap_2d(&tmx, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, X, N, h->D, ldx, kBK, box_rows,
                      CU_TENSOR_MAP_SWIZZLE_NONE))
        return cudaErrorInvalidValue;
    const Rings g = ps_rings(box_rows);
    if (g.sx % kCvtGroups != 0 || g.sa % kCvtGroups != 0) return cudaErrorInvalidConfiguration;
    PsParams p;
    p.N = N;
    p.D = h->D;
    p.r = h->r;
    p.npad = h->tc_npad;
    p.M = h->M;
    p.mpad = h->tc_mpad;
    p.nkb = (h->D + kBK - 1) / kBK;
    p.nh = h->tc_nh;
    p.half_rows = h->tc_half_rows;
    p.nkr_h[0] = h->tc_nkr_half[0];
    p.nkr_h[1] = h->tc_nkr_half[1];
    p.sx = g.sx;
    p.sa = g.sa;
    p.sb = g.sb;
    p.box_rows = box_rows;
    p.xstage = ps_xstage(box_rows);
    // one fp16 rounding of a row is accurate for 2^-8 sqrt(D) <= ||x|| <= 2^15; other rows are redone
    p.xn2_lo = (float)h->D * 0x1p-16f;
    p.xn2_hi = 0x1p30f;
    p.cnorm = h->cnorm;
    p.mode = mode;
    p.scale = scale;
    p.Y = Y;
    p.ldy = ldy;
    p.S = S;
    p.lds = lds;
    p.argmax = argmax;
    p.maxval = maxval;
    if (mode == GS_SCORE_RAW && !Y && !S)
        k_ps_tc<false><<<grid, kThreads, ps_smem_bytes(g, p.xstage), s>>>(tmx, h->tmap_q16, h->tmap_rh, h->tmap_rl, p);
    else
        k_ps_tc<true><<<grid, kThreads, ps_smem_bytes(g, p.xstage), s>>>(tmx, h->tmap_q16, h->tmap_rh, h->tmap_rl, p);
    return cudaGetLastError();
}

}  // namespace gs
