// gs_attn_tc.cu -- attention scores between compressed vectors on tcgen05
// (paper Sec. 2.2 attention score; Sec. 3.2: scores that use matrix
// multiplication are preserved on Gram-loc):
//
//     A[b] = softmax_row(scale * Yq[b] Yk[b]^T)      (or the scaled logits)
//
// Yq: B x Lq x r bf16, Yk: B x Lk x r bf16 (row stride ld, r <= 512), A: fp32.
//
// One persistent CTA per SM walks work items (sequence b, 128-query tile).  The
// query tile (128 x r bf16, up to 128 KB) stays resident in shared memory for
// the whole item, in K-blocks of 64 that are released one by one, so the next
// item's tile streams in while the current item's last MMAs run.  Key tiles
// (256 keys x 64) stream through a TMA ring.  Logits accumulate in fp32 in TMEM,
// double-buffered over units of 256 keys.  The row softmax needs every key, so
// each item runs two passes over its key tiles: pass 1 keeps an online row max
// and sum of exponentials; pass 2 recomputes the logits and writes
// exp(scale s - max) / sum.  The logits never go to HBM; the price is twice the
// MMA work (the tensor pipe has the headroom: the output write bounds it).
//
// Warp roles (352 threads): 0-7 epilogue (warp w reads TMEM lanes 32 (w % 4)..+31 =
// query rows, and keys [128 (w / 4), +128) of each 256-key unit; the two warps of a
// lane quadrant merge their row statistics between the passes through shared
// memory), 8 TMA producer of query K-blocks, 9 TMEM allocator + MMA issuer, 10 TMA
// producer of key tiles.  Every mbarrier wait is bounded.

#include <float.h>

#include <algorithm>

#include "gs_internal.h"
#include "gs_tc_ptx.cuh"

namespace gs {
namespace {

using namespace ptx;

__device__ unsigned g_err_attn = 0;

constexpr int kBM = 128;          // queries per item
constexpr int kBN = 256;          // keys per unit
constexpr int kBK = 64;           // r per K-block (128 bytes of bf16)
constexpr int kMaxKB = 8;         // r <= 512
constexpr int kQBlockBytes = kBM * kBK * 2;   // 16 KB
constexpr int kKStageBytes = kBN * kBK * 2;   // 32 KB
constexpr int kKStages = 3;
constexpr int kEpiWarps = 8;        // two per TMEM lane quadrant, each half of the keys of a unit
constexpr int kQWarp = 8, kMmaWarp = 9, kKWarp = 10;
constexpr int kThreads = 11 * 32;
constexpr int kTmemCols = 512;

struct AttnParams {
    int B, Lq, Lk, r, nkb;
    int qtiles, ntiles;      // query tiles per sequence, key tiles per sequence
    int passes;              // 2 with the row softmax, 1 for plain scaled logits
    float scale;
    float* A;                // B x Lq x Lk
    int a_vec;               // rows aligned for two-element stores (Lk even, A 8-byte aligned)
};

struct Ctl {
    uint64_t q_full[kMaxKB], q_empty[kMaxKB];
    uint64_t k_full[kKStages], k_empty[kKStages];
    uint64_t d_full[2], d_empty[2];
    uint64_t st_part, st_merged;  // row statistics: second key half posted / merged result posted
    uint64_t mma_done;
    float st_m[kBM], st_l[kBM];   // per query row: max and sum of exponentials being merged
    uint32_t tmem_base;
    int abort_flag;
};

__global__ void __launch_bounds__(kThreads, 1)
    k_attn_tc(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
              const AttnParams p) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    uint8_t* Qs = base;                                 // kMaxKB x 16 KB
    uint8_t* Ks = Qs + (size_t)kMaxKB * kQBlockBytes;   // kKStages x 32 KB
    Ctl& c = *reinterpret_cast<Ctl*>(Ks + (size_t)kKStages * kKStageBytes);
    volatile int* abort_flag = &c.abort_flag;
    unsigned* err = &g_err_attn;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long items = (long long)p.B * p.qtiles;
    const int nitems = items > blockIdx.x ? (int)((items - 1 - blockIdx.x) / gridDim.x + 1) : 0;
    const int units_per_item = p.passes * p.ntiles;

    if (threadIdx.x == 0) {
        for (int k = 0; k < kMaxKB; ++k) {
            mbar_init(&c.q_full[k], 1);
            mbar_init(&c.q_empty[k], 1);
        }
        for (int s = 0; s < kKStages; ++s) {
            mbar_init(&c.k_full[s], 1);
            mbar_init(&c.k_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&c.d_full[b], 1);
            mbar_init(&c.d_empty[b], kEpiWarps);
        }
        mbar_init(&c.st_part, kEpiWarps / 2);
        mbar_init(&c.st_merged, kEpiWarps / 2);
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

    auto item_bq = [&](int li, int& b, int& qt) {
        const long long ig = blockIdx.x + (long long)li * gridDim.x;
        b = (int)(ig / p.qtiles);
        qt = (int)(ig % p.qtiles);
    };

    if (warp == kQWarp) {
        // ------------------------------------------------------------- query K-blocks via TMA
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_first();
            int li = 0;
            bool ok = true;
            for (; li < nitems && ok; ++li) {
                int b, qt;
                item_bq(li, b, qt);
                const uint32_t ph = ((uint32_t)li & 1u) ^ 1u;
                for (int k = 0; k < p.nkb; ++k) {
                    if (!mbar_wait_1t(&c.q_empty[k], ph, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&c.q_full[k], kQBlockBytes);
                    tma_load_2d(Qs + (size_t)k * kQBlockBytes, &tmap_q, &c.q_full[k], k * kBK,
                                b * p.Lq + qt * kBM, pol);
                }
            }
            // the last item's (possibly partial) loads land before the CTA exits
            if (li > 0)
                for (int k = 0; k < p.nkb; ++k) mbar_drain(&c.q_full[k], (uint32_t)(li - 1) & 1u, err);
        }
    } else if (warp == kKWarp) {
        // ------------------------------------------------------------- key tiles via TMA
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_last();
            const int total = nitems * units_per_item * p.nkb;
            int it = 0;
            RingPos ks;
            int b = 0, qt = 0;
            for (int kb = 0, unit = 0, nt = 0, li = 0; it < total; ++it, ks.next(kKStages)) {
                const int s = ks.idx;
                if (!mbar_wait_1t(&c.k_empty[s], ks.phase ^ 1u, abort_flag, err)) break;
                if (kb == 0 && unit == 0) item_bq(li, b, qt);
                mbar_arrive_expect_tx(&c.k_full[s], kKStageBytes);
                tma_load_2d(Ks + (size_t)s * kKStageBytes, &tmap_k, &c.k_full[s], kb * kBK, b * p.Lk + nt * kBN, pol);
                // next (item, unit, K-block); units run over the key tiles once per pass
                if (++kb == p.nkb) {
                    kb = 0;
                    if (++nt == p.ntiles) nt = 0;
                    if (++unit == units_per_item) {
                        unit = 0;
                        nt = 0;
                        ++li;
                    }
                }
            }
            for (int j = std::max(0, it - kKStages); j < it; ++j)
                mbar_drain(&c.k_full[j % kKStages], (uint32_t)(j / kKStages) & 1u, err);
        }
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(kBN);
            int gu = 0;
            RingPos ks;
            bool ok = true;
            for (int li = 0; li < nitems && ok; ++li) {
                const uint32_t qph = (uint32_t)li & 1u;
                for (int u = 0; u < units_per_item && ok; ++u, ++gu) {
                    const int buf = gu & 1;
                    if (!mbar_wait_1t(&c.d_empty[buf], ((uint32_t)(gu >> 1) & 1u) ^ 1u, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t d_tmem = tmem + (uint32_t)(buf * kBN);
                    for (int kb = 0; kb < p.nkb; ++kb, ks.next(kKStages)) {
                        const int s = ks.idx;
                        if ((u == 0 && !mbar_wait_1t(&c.q_full[kb], qph, abort_flag, err)) ||
                            !mbar_wait_1t(&c.k_full[s], ks.phase, abort_flag, err)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t ad = sdesc_sw128(smem_u32(Qs + (size_t)kb * kQBlockBytes));
                        const uint64_t bd = sdesc_sw128(smem_u32(Ks + (size_t)s * kKStageBytes));
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k)
                            mma_f16_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                                       (kb | k) != 0 ? 1u : 0u);
                        mma_commit(&c.k_empty[s]);
                        // the item's last unit releases each query K-block as soon as it has used it
                        if (u == units_per_item - 1) mma_commit(&c.q_empty[kb]);
                    }
                    if (ok) mma_commit(&c.d_full[buf]);
                }
            }
            mma_commit(&c.mma_done);
            mbar_drain(&c.mma_done, 0, err);
        }
    } else if (warp < kEpiWarps) {
        // ------------------------------------------------------------- epilogue
        // Statistics pass: TMEM read one row per thread (32x32b), online max / sum over
        // this warp's half of the keys; the halves are merged before the writing pass.
        // Writing pass: TMEM read in the 16x256b pattern (a quad of threads holds 8
        // consecutive keys of one row, so stores write whole sectors); each row's
        // max and sum come by shuffle from the thread that owned the row.
        const int quad = warp & 3, kh = warp >> 2;  // lane quadrant, key half of each unit
        const int i = quad * 32 + lane;             // query row within the item (statistics pass)
        const int c0 = kh * (kBN / 2);              // first column of this warp's key half
        const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
        int gu = 0;
        for (int li = 0; li < nitems; ++li) {
            int b, qt;
            item_bq(li, b, qt);
            const bool valid = qt * kBM + i < p.Lq;
            float m = -FLT_MAX, l = 0.f;
            bool ok = true;
            for (int u = 0; u < units_per_item; ++u, ++gu) {
                const int buf = gu & 1;
                if (!mbar_wait_warp(&c.d_full[buf], (uint32_t)(gu >> 1) & 1u, abort_flag, err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int nt = u % p.ntiles;
                if (p.passes == 2 && u == p.ntiles) {
                    // merge the two key halves' statistics of each row (max, rescaled sums)
                    const uint32_t ph = (uint32_t)li & 1u;
                    if (kh == 1) {
                        c.st_m[i] = m;
                        c.st_l[i] = l;
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&c.st_part);
                        if (!mbar_wait_warp(&c.st_merged, ph, abort_flag, err)) {
                            ok = false;
                            break;
                        }
                        m = c.st_m[i];
                        l = c.st_l[i];
                    } else {
                        if (!mbar_wait_warp(&c.st_part, ph, abort_flag, err)) {
                            ok = false;
                            break;
                        }
                        const float m1 = c.st_m[i], l1 = c.st_l[i];
                        const float mm = fmaxf(m, m1);
                        l = l * __expf(m - mm) + l1 * __expf(m1 - mm);
                        m = mm;
                        c.st_m[i] = m;
                        c.st_l[i] = l;
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&c.st_merged);
                    }
                }
                if (p.passes == 2 && u < p.ntiles) {
                    const uint32_t tb = tmem + lane_base + (uint32_t)(buf * kBN);
                    for (int jc = c0; jc < c0 + kBN / 2; jc += 16) {
                        float v[16];
                        tmem_ld16(tb + (uint32_t)jc, v);
                        const int k0 = nt * kBN + jc;
                        if (!valid || k0 >= p.Lk) continue;
                        const int nv = min(16, p.Lk - k0);
                        float cm = m;
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            if (j < nv) cm = fmaxf(cm, p.scale * v[j]);
                        float add = 0.f;
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            if (j < nv) add += __expf(p.scale * v[j] - cm);
                        l = l * __expf(m - cm) + add;
                        m = cm;
                    }
                } else {
                    for (int half = 0; half < 2; ++half) {
                        const int r0 = half * 16 + (lane >> 2);  // rows r0 and r0 + 8 of this warp
                        const float m0 = __shfl_sync(0xffffffffu, m, r0), l0 = __shfl_sync(0xffffffffu, l, r0);
                        const float m1 = __shfl_sync(0xffffffffu, m, r0 + 8), l1 = __shfl_sync(0xffffffffu, l, r0 + 8);
                        const float mh[2] = {m0, m1};
                        const float ih[2] = {l0 > 0.f ? 1.f / l0 : 0.f, l1 > 0.f ? 1.f / l1 : 0.f};
                        int qrow[2];
                        float* arow[2];
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            qrow[h] = qt * kBM + quad * 32 + r0 + 8 * h;
                            arow[h] = p.A + ((size_t)b * p.Lq + (qrow[h] < p.Lq ? qrow[h] : 0)) * p.Lk;
                        }
                        const uint32_t tb = tmem + ((uint32_t)(quad * 32 + half * 16) << 16) + (uint32_t)(buf * kBN);
                        for (int jc = c0; jc < c0 + kBN / 2; jc += 32) {
                            float v[16];
                            tmem_ld16x256b_x4(tb + (uint32_t)jc, v);
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                const int key = nt * kBN + jc + 8 * j + 2 * (lane & 3);
#pragma unroll
                                for (int h = 0; h < 2; ++h) {
                                    if (qrow[h] >= p.Lq || key >= p.Lk) continue;
                                    float a0 = p.scale * v[4 * j + 2 * h], a1 = p.scale * v[4 * j + 2 * h + 1];
                                    if (p.passes == 2) {
                                        a0 = __expf(a0 - mh[h]) * ih[h];
                                        a1 = __expf(a1 - mh[h]) * ih[h];
                                    }
                                    float* dst = arow[h] + key;
                                    if (p.a_vec && key + 1 < p.Lk) {
                                        __stcs(reinterpret_cast<float2*>(dst), make_float2(a0, a1));
                                    } else {
                                        dst[0] = a0;
                                        if (key + 1 < p.Lk) dst[1] = a1;
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
            if (!ok) break;
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ================================================================= one pass, key units spread over a cluster
// With the row softmax and Lk <= 4 x 256, the G = ceil(Lk / 256) CTAs of a thread-block
// cluster share each work item: CTA g computes the logits of keys [256 g, 256 g + 256)
// for the item's 128 queries, once.  The epilogue warps form two teams that take the
// items in turn (team t: items t, t + 2, ...; TMEM accumulator t), so one team's exchange
// and writes overlap the other team's statistics.  A team thread owns one query row and
// 128 of the unit's keys, read from TMEM in two 64-key passes: the statistics pass takes,
// in base-2 units, the max m of c s_j (c = scale log2 e) and l = sum 2^(c s_j - m); the two
// key halves of each row meet in shared memory, the team posts each row's CTA result to
// every CTA of the cluster with asynchronous remote stores, and with all G results the
// row's max M and sum L are known; the writing pass reads the logits again and writes
// 2^(c s_j - M) / L.  The logits never leave the chip.  Outputs go through a 64-byte-
// swizzled 32 x 16 fp32 tile per warp and TMA tensor stores over a 3-D map (B x Lq x Lk),
// which clips rows past Lq and keys past Lk.  (Multicasting the query tile across the cluster
// halved its L2 reads but tied every CTA's stage release to the slowest CTA: 2 % slower.)
//
// Warp roles (576 threads): 0-7 team 0 and 8-15 team 1 (warp w: TMEM lanes 32 (w % 4) =
// query rows, keys [128 ((w / 4) % 2), +128) of the CTA's unit; warps with (w / 4) even also
// merge and post their rows), 16 TMA producer (query and key K-blocks into one stage), 17
// TMEM allocator + MMA issuer.

constexpr int kClMaxG = 4;
constexpr int kClStageBytes = kQBlockBytes + kKStageBytes;  // 48 KB: query block, then key block
constexpr int kClStages = 3;
constexpr int kClEpiWarps = 16;
constexpr int kClCols = kBN / 4;            // keys per epilogue thread
constexpr int kClProdWarp = 16, kClMmaWarp = 17;
constexpr int kClThreads = 18 * 32;
constexpr int kClStgCols = 16;             // one output box: 32 query rows x 16 keys fp32 (64-byte rows)
constexpr int kClStgBytes = 32 * kClStgCols * 4;

struct ClCtl {
    uint64_t full[kClStages], empty[kClStages];
    uint64_t d_full[2], d_empty[2];  // TMEM accumulator t, used by team t
    uint64_t p_full[2];              // team t's two key halves of an item's rows are in part[t]
    uint64_t x_full[2][2];           // team t, slot s: every CTA's row results of an item
    uint64_t mma_done;
    float2 part[2][2][kBM];             // [team][key half][query row] = (max, sum)
    float2 xch[2][2][kClMaxG][kBM];     // [team][slot][rank][query row] = (max, sum)
    uint32_t tmem_base;
    int abort_flag;
};

// 2^x on the special-function unit (ex2.approx.ftz: 2^-inf = 0).
__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// max (MIN: min) of v[0, n), eight independent chains; MASK: n may be below the length
template <bool MIN, bool MASK>
__device__ __forceinline__ float row_extreme(const float* v, int n) {
    float e8[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) e8[k] = MIN ? INFINITY : -INFINITY;
#pragma unroll
    for (int j = 0; j < kClCols; ++j)
        if (!MASK || j < n) e8[j & 7] = MIN ? fminf(e8[j & 7], v[j]) : fmaxf(e8[j & 7], v[j]);
    if (MIN)
        return fminf(fminf(fminf(e8[0], e8[1]), fminf(e8[2], e8[3])), fminf(fminf(e8[4], e8[5]), fminf(e8[6], e8[7])));
    return fmaxf(fmaxf(fmaxf(e8[0], e8[1]), fmaxf(e8[2], e8[3])), fmaxf(fmaxf(e8[4], e8[5]), fmaxf(e8[6], e8[7])));
}

// merge of partial (max, sum) pairs taken in base 2 (empty parts are (-inf, 0))
__device__ __forceinline__ float2 merge_stats(const float2* e, int n) {
    float M = -INFINITY;
#pragma unroll
    for (int j = 0; j < kClMaxG; ++j)
        if (j < n) M = fmaxf(M, e[j].x);
    float L = 0.f;
#pragma unroll
    for (int j = 0; j < kClMaxG; ++j)
        if (j < n && e[j].y > 0.f) L += e[j].y * ex2_approx(e[j].x - M);
    return make_float2(M, L);
}

__global__ void __launch_bounds__(kClThreads, 1)
    k_attn_cl(const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
              const __grid_constant__ CUtensorMap tmap_a, const AttnParams p) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    uint8_t* St = base;                                          // kClStages x 48 KB
    uint8_t* Stg = St + (size_t)kClStages * kClStageBytes;       // 16 warps x 2 KB output box
    ClCtl& c = *reinterpret_cast<ClCtl*>(Stg + (size_t)kClEpiWarps * kClStgBytes);
    volatile int* abort_flag = &c.abort_flag;
    unsigned* err = &g_err_attn;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const int G = p.ntiles;  // CTAs per cluster = key units per row
    const long long cid = cluster_id_x(), ncl = cluster_count_x();
    const long long items = (long long)p.B * p.qtiles;
    const int nitems = items > cid ? (int)((items - 1 - cid) / ncl + 1) : 0;
    const int nkb = p.nkb;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kClStages; ++s) {
            mbar_init(&c.full[s], 1);
            mbar_init(&c.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&c.d_full[b], 1);
            mbar_init(&c.d_empty[b], kClEpiWarps / 2);
            mbar_init(&c.p_full[b], kClEpiWarps / 2);
            mbar_init(&c.x_full[b][0], 1);
            mbar_init(&c.x_full[b][1], 1);
        }
        mbar_init(&c.mma_done, 1);
        c.abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == kClMmaWarp) {
        tmem_alloc(&c.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();  // every CTA's barriers exist before any CTA arrives on them
    tc_fence_after();
    const uint32_t tmem = c.tmem_base;

    auto item_bq = [&](int li, int& b, int& qt) {
        const long long ig = cid + (long long)li * ncl;
        b = (int)(ig / p.qtiles);
        qt = (int)(ig % p.qtiles);
    };

    if (warp == kClProdWarp) {
        // ------------------------------------------------------------- query + key K-blocks via TMA
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_last();
            RingPos st;
            int it = 0;
            bool ok = true;
            for (int li = 0; li < nitems && ok; ++li) {
                int b, qt;
                item_bq(li, b, qt);
                for (int kb = 0; kb < nkb; ++kb, ++it, st.next(kClStages)) {
                    if (!mbar_wait_1t(&c.empty[st.idx], st.phase ^ 1u, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    uint8_t* dst = St + (size_t)st.idx * kClStageBytes;
                    mbar_arrive_expect_tx(&c.full[st.idx], kClStageBytes);
                    tma_load_2d(dst, &tmap_q, &c.full[st.idx], kb * kBK, b * p.Lq + qt * kBM, pol);
                    tma_load_2d(dst + kQBlockBytes, &tmap_k, &c.full[st.idx], kb * kBK,
                                b * p.Lk + (int)rank * kBN, pol);
                }
            }
            for (int j = std::max(0, it - kClStages); j < it; ++j)
                mbar_drain(&c.full[j % kClStages], (uint32_t)(j / kClStages) & 1u, err);
        }
    } else if (warp == kClMmaWarp) {
        // ------------------------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32(kBN);
            RingPos st;
            bool ok = true;
            for (int li = 0; li < nitems && ok; ++li) {
                const int buf = li & 1;
                if (!mbar_wait_1t(&c.d_empty[buf], ((uint32_t)(li >> 1) & 1u) ^ 1u, abort_flag, err)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * kBN);
                for (int kb = 0; kb < nkb; ++kb, st.next(kClStages)) {
                    if (!mbar_wait_1t(&c.full[st.idx], st.phase, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(St + (size_t)st.idx * kClStageBytes);
                    const uint64_t ad = sdesc_sw128(sa);
                    const uint64_t bd = sdesc_sw128(sa + kQBlockBytes);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k)
                        mma_f16_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                                   (kb | k) != 0 ? 1u : 0u);
                    mma_commit(&c.empty[st.idx]);
                }
                if (ok) mma_commit(&c.d_full[buf]);
            }
            mma_commit(&c.mma_done);
            mbar_drain(&c.mma_done, 0, err);
        }
    } else {
        // ------------------------------------------------------------- epilogue (two teams)
        const int team = warp >> 3, quad = warp & 3, kh = (warp >> 2) & 1;
        const int i = quad * 32 + lane;                          // query row within the item
        const int keyh = (int)rank * kBN + kh * (kBN / 2);       // first of this warp's 128 keys
        const float c2 = p.scale * 1.4426950408889634f;
        uint8_t* sb = Stg + (size_t)warp * kClStgBytes;
        const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
        const uint32_t tcol = (uint32_t)(team * kBN + kh * (kBN / 2));
        for (int li = team; li < nitems; li += 2) {
            int b, qt;
            item_bq(li, b, qt);
            const int k = li >> 1;                   // this team's k-th item
            const uint32_t ph = (uint32_t)k & 1u;    // phase of d_full[team] / p_full[team]
            const int xs = k & 1;                    // exchange slot (two per team)
            const uint32_t xph = (uint32_t)(k >> 1) & 1u;
            if (!mbar_wait_warp(&c.d_full[team], ph, abort_flag, err)) break;
            tc_fence_after();
            // statistics pass over the two 64-key chunks: max m and sum l in base 2
            float m = -INFINITY, l = 0.f;
            for (int cc = 0; cc < 2; ++cc) {
                const int nvalid = min(kClCols, max(0, p.Lk - (keyh + cc * kClCols)));
                float v[kClCols];
                {
                    uint32_t r[kClCols];
                    const uint32_t ta = tmem + lane_base + tcol + (uint32_t)(cc * kClCols);
                    tmem_ld32_issue(ta, r);
                    tmem_ld32_issue(ta + 32u, r + 32);
                    tmem_wait_ld32(r);
                    tmem_wait_ld32(r + 32);
#pragma unroll
                    for (int j = 0; j < kClCols; ++j) v[j] = __uint_as_float(r[j]);
                }
                if (nvalid == 0) continue;
                float ext;
                if (nvalid == kClCols)
                    ext = c2 >= 0.f ? row_extreme<false, false>(v, kClCols) : row_extreme<true, false>(v, kClCols);
                else
                    ext = c2 >= 0.f ? row_extreme<false, true>(v, nvalid) : row_extreme<true, true>(v, nvalid);
                const float mc = c2 * ext;
                float l8[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) l8[q] = 0.f;
#pragma unroll
                for (int j = 0; j < kClCols; ++j)
                    if (nvalid == kClCols || j < nvalid) l8[j & 7] += ex2_approx(fmaf(v[j], c2, -mc));
                const float lc = ((l8[0] + l8[1]) + (l8[2] + l8[3])) + ((l8[4] + l8[5]) + (l8[6] + l8[7]));
                const float mn = fmaxf(m, mc);
                l = (l > 0.f ? l * ex2_approx(m - mn) : 0.f) + lc * ex2_approx(mc - mn);
                m = mn;
            }
            // the row's two key halves meet in shared memory; the even-half warps merge them
            // and post the CTA's result to every CTA of the cluster
            c.part[team][kh][i] = make_float2(m, l);
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.p_full[team]);
            if (kh == 0) {
                if (!mbar_wait_warp(&c.p_full[team], ph, abort_flag, err)) break;
                float2 e[kClMaxG];
                e[0] = c.part[team][0][i];
                e[1] = c.part[team][1][i];
                const float2 rc = merge_stats(e, 2);
                const uint32_t slot = smem_u32(&c.xch[team][xs][rank][i]);
                const uint32_t bar = smem_u32(&c.x_full[team][xs]);
                // the barrier's one arrival per phase carries the byte count of every CTA's
                // posts; the posts are asynchronous stores that complete those bytes (a
                // release-arrive after plain remote stores cost microseconds per item)
                if (quad == 0 && lane == 0) mbar_arrive_expect_tx(&c.x_full[team][xs], (uint32_t)(G * kBM * 8));
                for (int g = 0; g < G; ++g)
                    st_async_f32x2(mapa_shared(slot, (uint32_t)g), rc.x, rc.y, mapa_shared(bar, (uint32_t)g));
            }
            const bool got = mbar_wait_cluster(&c.x_full[team][xs], xph, abort_flag, err);
            if (!__all_sync(0xffffffffu, got)) break;
            float M, invL;
            {
                float2 e[kClMaxG];
#pragma unroll
                for (int q = 0; q < kClMaxG; ++q) e[q] = q < G ? c.xch[team][xs][q][i] : make_float2(-INFINITY, 0.f);
                const float2 rw = merge_stats(e, G);
                M = rw.x;
                invL = rw.y > 0.f ? __fdividef(1.f, rw.y) : 0.f;
            }
            // writing pass: 2^(c s_j - M) / L through 32 x 16 tiles (16-byte chunk q of row
            // `lane` at chunk q ^ ((lane / 2) % 4), the TMA's 64-byte swizzle) and tensor stores
            const int y = qt * kBM + quad * 32;
            for (int cc = 0; cc < 2; ++cc) {
                float v[kClCols];
                {
                    uint32_t r[kClCols];
                    const uint32_t ta = tmem + lane_base + tcol + (uint32_t)(cc * kClCols);
                    tmem_ld32_issue(ta, r);
                    tmem_ld32_issue(ta + 32u, r + 32);
                    tmem_wait_ld32(r);
                    tmem_wait_ld32(r + 32);
#pragma unroll
                    for (int j = 0; j < kClCols; ++j) v[j] = __uint_as_float(r[j]);
                }
                if (cc == 1) {  // the accumulator has been read twice: back to the MMA
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&c.d_empty[team]);
                }
#pragma unroll
                for (int q = 0; q < kClCols / kClStgCols; ++q) {
                    const int x = keyh + cc * kClCols + q * kClStgCols;
                    if (lane == 0) bulk_wait_read_0();  // the previous store has read the tile
                    __syncwarp();
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const float* vv = v + q * kClStgCols + 4 * u;
                        const float4 o = make_float4(ex2_approx(fmaf(vv[0], c2, -M)) * invL,
                                                     ex2_approx(fmaf(vv[1], c2, -M)) * invL,
                                                     ex2_approx(fmaf(vv[2], c2, -M)) * invL,
                                                     ex2_approx(fmaf(vv[3], c2, -M)) * invL);
                        *reinterpret_cast<float4*>(sb + lane * 64 + ((u ^ ((lane >> 1) & 3)) << 4)) = o;
                    }
                    fence_proxy_async();
                    __syncwarp();
                    if (lane == 0) {
                        if (x < p.Lk && y < p.Lq) tma_store_3d(&tmap_a, sb, x, y, b);
                        bulk_commit();
                    }
                }
            }
        }
        if (lane == 0) bulk_wait_all();
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync_all();  // no CTA leaves while a peer may still post into its shared memory
    if (warp == kClMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

constexpr size_t kClSmemBytes =
    1024 + (size_t)kClStages * kClStageBytes + (size_t)kClEpiWarps * kClStgBytes + sizeof(ClCtl);
static_assert(kClSmemBytes <= 227 * 1024, "cluster attention kernel shared memory exceeds the per-CTA limit");

constexpr size_t kSmemBytes = 1024 + (size_t)kMaxKB * kQBlockBytes + (size_t)kKStages * kKStageBytes + sizeof(Ctl);
static_assert(kSmemBytes <= 227 * 1024, "attention kernel shared memory exceeds the per-CTA limit");

bool g_attr_set[64];
bool g_cl_attr_set[64];
int g_cl_max[64][kClMaxG + 1];  // active clusters of k_attn_cl per device and cluster size

}  // namespace

unsigned take_device_error_attn() {
    unsigned v = 0, z = 0;
    cudaMemcpyFromSymbol(&v, g_err_attn, sizeof(v));
    if (v) cudaMemcpyToSymbol(g_err_attn, &z, sizeof(z));
    return v;
}

bool attn_tc_supported(int r, long long ldy, const void* Yq, const void* Yk) {
    return r >= 1 && r <= kMaxKB * kBK && ldy % 8 == 0 && (uintptr_t)Yq % 16 == 0 && (uintptr_t)Yk % 16 == 0;
}

cudaError_t launch_attn_tc(const void* Yq, const void* Yk, int B, int Lq, int Lk, int r, long long ldy, float scale,
                           bool softmax, float* A, int device, cudaStream_t s) {
    AttnParams p;
    p.B = B;
    p.Lq = Lq;
    p.Lk = Lk;
    p.r = r;
    p.nkb = (r + kBK - 1) / kBK;
    p.qtiles = (Lq + kBM - 1) / kBM;
    p.ntiles = (Lk + kBN - 1) / kBN;
    p.passes = softmax ? 2 : 1;
    p.scale = scale;
    p.A = A;
    p.a_vec = ((uintptr_t)A % 8 == 0) && (Lk % 2 == 0);
    CUtensorMap tq, tk;
    if (!make_tmap_2d(&tq, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, Yq, (long long)B * Lq, r, ldy, kBK, kBM,
                      CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&tk, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, Yk, (long long)B * Lk, r, ldy, kBK, kBN,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    const long long items = (long long)B * p.qtiles;
    CUtensorMap ta;
    if (softmax && p.ntiles <= kClMaxG && Lk % 4 == 0 && (uintptr_t)A % 16 == 0 &&
        make_tmap_3d(&ta, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, A, Lk, Lq, B, Lk, (long long)Lq * Lk, kClStgCols, 32,
                     CU_TENSOR_MAP_SWIZZLE_64B)) {
        // one pass: the key units of a row spread over a cluster of ntiles CTAs
        const int G = p.ntiles;
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = (unsigned)G;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.blockDim = dim3(kClThreads);
        cfg.dynamicSmemBytes = kClSmemBytes;
        cfg.stream = s;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
        if (!g_cl_attr_set[device]) {
            cudaError_t e =
                cudaFuncSetAttribute(k_attn_cl, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kClSmemBytes);
            if (e != cudaSuccess) return e;
            g_cl_attr_set[device] = true;
        }
        int& ncl_max = g_cl_max[device][G];
        if (ncl_max <= 0) {
            int sms = 0;
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
            cfg.gridDim = dim3((unsigned)(std::max(sms, G) / G * G));
            cudaError_t e = cudaOccupancyMaxActiveClusters(&ncl_max, k_attn_cl, &cfg);
            if (e != cudaSuccess) return e;
            if (ncl_max <= 0) return cudaErrorInvalidConfiguration;
        }
        const long long ncl = std::min<long long>(ncl_max, items);
        cfg.gridDim = dim3((unsigned)(ncl * G));
        cudaError_t e = cudaLaunchKernelEx(&cfg, k_attn_cl, tq, tk, ta, p);
        if (e != cudaSuccess) return e;
        return cudaGetLastError();
    }
    if (device >= 0 && device < 64 && !g_attr_set[device]) {
        cudaError_t e = cudaFuncSetAttribute(k_attn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
        if (e != cudaSuccess) return e;
        g_attr_set[device] = true;
    }
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    const int grid = (int)std::min<long long>(sms > 0 ? sms : 1, items);
    k_attn_tc<<<grid, kThreads, kSmemBytes, s>>>(tq, tk, p);
    return cudaGetLastError();
}

}  // namespace gs
