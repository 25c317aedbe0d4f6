// gs_rbind_tc.cu -- reconstruction fused with binding: Z = op(T Q, Y) in one kernel, the
// reconstructed rows never leaving the SM.
//
// Sec. 3.3 reconstructs x_hat = t Q from Gram-loc coefficients and binds it with a partner row y
// block by block (Sec. 2.2: circular convolution of blocks of L; unbinding: circular
// correlation).  Here persistent pairs of CTAs (clusters of two) compute 256-row x 256-column
// tiles of X_hat = T Q on the tensor core (one tcgen05 cta_group::2 MMA: fp16 T rows scaled by
// exact powers of two, the basis' fp16 Q^T, fp32 accumulation in TMEM; each CTA stages its own 128
// rows of T and half of the tile's rows of Q^T), and each CTA binds its 128 x 256 part where it
// lies: it holds 256 / L whole blocks of each of the CTA's rows, and the binding runs through block
// spectra (convolution theorem, real blocks packed as H = L / 2 complex points) with TMEM as the
// transforms' working storage:
//
//   z = IDFT_L(DFT_L(x) . DFT_L(y))          bind
//   z = IDFT_L(DFT_L(x) . conj(DFT_L(y)))    unbind
//
// TMEM has 512 columns: the accumulator and the partner's spectrum take one 256-column half
// each, swapping roles every tile, so the MMA of tile t + 1 (into the half the partner left)
// runs while tile t is transformed back and stored.  A thread owns one row (TMEM lane) of its
// warp's lane quadrant; the four warps of a quadrant split each pass's column groups.  With
// H = R1 R2 (128 = 16 x 8, 64 = 8 x 8, 32 = 8 x 4) and complex point p of block b in columns
// 2 H b + 2 p, + 1:
//
//   copy-in   partner chunks (TMA, 128 rows x 32 floats, 128-byte swizzle) -> TMEM, natural order
//   F1        (b, n2): DFT_R1 over the points n2 + R2 n1, times w_H^(n2 k1), back in place
//             (partner half, then -- once the MMA has committed -- the accumulator half, whose
//             values first take the row's scale back)
//   middle    (b, k1 with R1 - k1): DFT_R2 of the contiguous group k1 gives W_(k1 + R1 k2) of
//             both blocks; the real split, the product of the spectra and the packing of the
//             product for a real inverse transform pair k with H - k, which is element
//             R2 - 1 - k2 of group R1 - k1 (groups 0 and R1 / 2 pair with themselves); then
//             the inverse DFT_R2 along k2 and w_H^-(n2 k1), back in place (accumulator half)
//   I2        (b, n2): inverse DFT_R1 over k1, which leaves point n = n2 + R2 n1 at its own
//             position (natural order), times 1 / (4 L)
//   store     TMEM -> per-warp staging (32 rows x 16 floats, 64-byte swizzle) -> TMA store
//
// Both transforms are decimation in frequency forward and in time inverse, so no pass permutes.
// The spectra carry a factor 2 each (real split without halves), the product 4, its packing 2,
// the unnormalised inverse H: z = v / (8 H) = v / (4 L), an exact power of two.
//
// Warp roles (608 threads): 0 TMA producer of T and Q K-blocks (both CTAs' loads complete on the even
// CTA's barriers), 1 TMEM allocator + pair MMA issuer (even CTA; its commits release both CTAs'
// stages and hand both accumulators over), 2 TMA producer of the partner rows (and an L2 prefetch of
// the next tile's), 3-18 transforms (warp w reads TMEM lanes 32 (w % 4)..+31; the next MMA waits for
// the transform warps of both CTAs).  Every mbarrier wait is bounded (gs_tc_ptx.cuh); a
// quadrant's four warps decide together, at the named barrier between passes, whether to go on,
// so a timeout unwinds them without leaving one behind.

#include <stdint.h>

#include <algorithm>

#include "gs_fft.cuh"
#include "gs_internal.h"
#include "gs_tc_ptx.cuh"

namespace gs {
namespace {

using namespace ptx;
using namespace fft;

__device__ unsigned g_err_rbind = 0;

constexpr int kRbBM = 128;                               // rows of a tile (TMEM lanes)
constexpr int kRbBN = 256;                               // columns of a tile (one TMEM half)
constexpr int kRbBK = 64;                                // K-block of the MMA operands
constexpr int kRbSubs = 4;                               // transform warps per lane quadrant
constexpr int kRbEpi0 = 3;                               // first transform warp
constexpr int kRbThreads = (kRbEpi0 + 4 * kRbSubs) * 32;  // 608
constexpr int kRbStages = 3;                             // T / Q K-block stages
constexpr int kRbAStage = kRbBM * kRbBK * 2;             // 16 KB of fp16 T (this CTA's 128 rows)
constexpr int kRbBStage = kRbBN / 2 * kRbBK * 2;         // 16 KB of fp16 Q^T (this CTA's half of the tile)
constexpr int kRbYStages = 8;                            // a whole tile of partner boxes (box cc in stage cc)
constexpr int kRbYCols = 32;                             // a partner box: 128 rows x 128 bytes
constexpr int kRbYStage = kRbBM * kRbYCols * 4;          // 16 KB
constexpr int kRbChunks = kRbBN / kRbYCols;              // 8 partner boxes per tile
constexpr int kRbMaxL = 256;

struct RbParams {
    long long m;       // rows
    int D, nkb, tiles_n;
    long long tiles;
    float zscale;      // 1 / (4 L)
    const float* rowmul;
};

struct RbCtl {
    uint64_t full[kRbStages], empty[kRbStages];
    uint64_t y_full[kRbYStages], y_empty[kRbYStages];
    uint64_t d_full;    // the tile's accumulator is complete (MMA commit, to both CTAs)
    uint64_t y_free;    // both CTAs' partner halves have been read: the next tile's MMA may write them
    uint64_t mma_done;
    uint32_t tmem_base;
    int abort_flag;
};

// shared memory: the control block and the twiddle table, then (from the next 1024-byte boundary)
// the T / Q stages and the partner stages.  Dynamic shared memory starts 1024-aligned in practice,
// so the request is the whole per-block limit and the kernel checks that its layout fits (else it
// records GS_DEV_ERR_LAYOUT and returns before touching anything).
constexpr size_t kRbHead = (sizeof(RbCtl) + 15) / 16 * 16 + kRbMaxL * sizeof(float2);
constexpr size_t kRbData = (size_t)kRbStages * (kRbAStage + kRbBStage) + (size_t)kRbYStages * kRbYStage;
constexpr size_t kRbSmemBytes = 227 * 1024;
static_assert(kRbHead + kRbData <= kRbSmemBytes, "layout");

// the transform plan of a block of L = 2 H reals
template <int H>
struct RbPlan {
    static constexpr int R1 = H == 128 ? 16 : 8;
    static constexpr int R2 = H / R1;
    static constexpr int NB = kRbBN / (2 * H);  // blocks per tile row
    static constexpr int G = NB * R2;           // strided groups (F1, I2)
    static constexpr int U = NB * R1 / 2;       // group pairs (middle)
    static_assert(R1 * R2 == H && G % kRbSubs == 0 && U % kRbSubs == 0, "plan");
};

// the four warps of a lane quadrant: TMEM stores done and visible, and whether all of them go on
__device__ __forceinline__ bool quad_sync(int quad, bool ok) {
    tmem_wait_st();
    tc_fence_before();
    ok = bar_sync_and(1 + quad, 32 * kRbSubs, ok);
    tc_fence_after();
    return ok;
}

// One strided pass over this warp's groups (b, n2), elements n2 + R2 i (i < R1), in place.
// Forward (F1): the inputs times `mul` (the row's scale, or none), DFT_R1, then w_H^(n2 k1).
// Inverse (I2): inverse DFT_R1, then the outputs times `mul`.  The next group's loads are in
// flight while a group is transformed.
template <int H, bool INV, bool SCALE>
__device__ __forceinline__ void rb_strided(uint32_t tb, int sub, float mul, const float2* __restrict__ tw) {
    using P = RbPlan<H>;
    constexpr int R1 = P::R1, R2 = P::R2, NG = P::G / kRbSubs;
    uint32_t r[2][2 * R1];
    auto col = [&](int gi) {
        const int g = sub + kRbSubs * gi;
        return tb + (uint32_t)(2 * H * (g / R2) + 2 * (g % R2));
    };
    auto issue = [&](int gi, uint32_t (&q)[2 * R1]) {
        const uint32_t c0 = col(gi);
#pragma unroll
        for (int i = 0; i < R1; ++i) tmem_ld2_issue(c0 + (uint32_t)(2 * R2 * i), q[2 * i], q[2 * i + 1]);
    };
    issue(0, r[0]);
#pragma unroll
    for (int gi = 0; gi < NG; ++gi) {
        tmem_wait_ld_regs(r[gi & 1]);
        float2 v[R1];
#pragma unroll
        for (int i = 0; i < R1; ++i) v[i] = make_float2(__uint_as_float(r[gi & 1][2 * i]), __uint_as_float(r[gi & 1][2 * i + 1]));
        if (gi + 1 < NG) issue(gi + 1, r[(gi + 1) & 1]);
        const int n2 = (sub + kRbSubs * gi) % R2;
        if constexpr (!INV) {
            if constexpr (SCALE) {
#pragma unroll
                for (int i = 0; i < R1; ++i) v[i] = make_float2(v[i].x * mul, v[i].y * mul);
            }
            dft<R1>(v);
#pragma unroll
            for (int k1 = 1; k1 < R1; ++k1) v[k1] = c_mul(v[k1], tw[2 * n2 * k1]);  // w_H^(n2 k1) = w_L^(2 n2 k1)
        } else {
            dft_inv<R1>(v);
            if constexpr (SCALE) {
#pragma unroll
                for (int i = 0; i < R1; ++i) v[i] = make_float2(v[i].x * mul, v[i].y * mul);
            }
        }
        const uint32_t c0 = col(gi);
#pragma unroll
        for (int i = 0; i < R1; ++i) tmem_st2(c0 + (uint32_t)(2 * R2 * i), v[i].x, v[i].y);
    }
}

// One pair (k, k' = H - k) of the middle step.  From W (the packed transforms of x and of y) at k
// and k', the doubled real spectra at k and the conjugates of those at k':
//   E = W_k + conj(W_k'),  O = -i (W_k - conj(W_k')),  P = X_k = E + t O,  Q = conj(X_k') = E - t O
// (t = w_L^k; R = Y_k and S = conj(Y_k') the same way), the product Z = X Y (unbind: X conj(Y)) as
// Z_k = P R and conj(Z_k') = Q S (unbind: P conj(R), Q conj(S)), and the doubled packed spectrum of
// the product's real inverse transform
//   V_k = A + C,  V_k' = conj(A - C),  A = Z_k + conj(Z_k'),  C = i conj(t) (Z_k - conj(Z_k')).
// For k = 0 (k' = 0 mod H, the second spectrum being X_H) and k = H / 2 (k' = k) both outputs are
// the same value.
template <bool UNB>
__device__ __forceinline__ void rb_pair(float2 wxk, float2 wxc, float2 wyk, float2 wyc, float2 t, float2& vk,
                                        float2& vc) {
    auto spectra = [&](float2 wk, float2 wc, float2& pk, float2& qc) {
        const float2 e = make_float2(wk.x + wc.x, wk.y - wc.y);
        const float2 o = make_float2(wk.y + wc.y, wc.x - wk.x);
        const float2 to = c_mul(t, o);
        pk = c_add(e, to);
        qc = c_sub(e, to);
    };
    float2 P, Q, R, S;
    spectra(wxk, wxc, P, Q);
    spectra(wyk, wyc, R, S);
    const float2 zk = UNB ? c_mulconj(P, R) : c_mul(P, R);
    const float2 zc = UNB ? c_mulconj(Q, S) : c_mul(Q, S);  // conj(Z_k')
    const float2 a = c_add(zk, zc), b = c_sub(zk, zc);
    const float2 cc = make_float2(fmaf(t.y, b.x, -t.x * b.y), fmaf(t.x, b.x, t.y * b.y));  // i conj(t) b
    vk = c_add(a, cc);
    vc = make_float2(a.x - cc.x, cc.y - a.y);
}

template <int N>
__device__ __forceinline__ void rb_group_issue(uint32_t taddr, uint32_t (&r)[2 * N]) {
#pragma unroll
    for (int i = 0; i < N; ++i) tmem_ld2_issue(taddr + (uint32_t)(2 * i), r[2 * i], r[2 * i + 1]);
}
template <int N>
__device__ __forceinline__ void rb_group_unpack(const uint32_t (&r)[2 * N], float2 (&v)[N]) {
#pragma unroll
    for (int i = 0; i < N; ++i) v[i] = make_float2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
}
template <int N>
__device__ __forceinline__ void rb_group_store(uint32_t taddr, const float2 (&v)[N]) {
#pragma unroll
    for (int i = 0; i < N; ++i) tmem_st2(taddr + (uint32_t)(2 * i), v[i].x, v[i].y);
}

// The middle step over this warp's group pairs (b; k1 = ka with kb = R1 - ka, or the two
// self-paired groups 0 and R1 / 2), reading the F1 results of x (accumulator half tx) and of y
// (partner half ty) and writing the inverse transform's first pass over x's groups.
template <int H, bool UNB>
__device__ __forceinline__ void rb_middle(uint32_t tx, uint32_t ty, int sub, const float2* __restrict__ tw) {
    using P = RbPlan<H>;
    constexpr int R1 = P::R1, R2 = P::R2;
#pragma unroll 1
    for (int u = sub; u < P::U; u += kRbSubs) {
        const int b = u / (R1 / 2), pr = u % (R1 / 2);
        const int ka = pr, kb = pr == 0 ? R1 / 2 : R1 - pr;
        const uint32_t oa = (uint32_t)(2 * H * b + 2 * R2 * ka), ob = (uint32_t)(2 * H * b + 2 * R2 * kb);
        float2 xa[R2], xb[R2];
        {
            float2 ya[R2], yb[R2];
            {
                uint32_t r[4][2 * R2];
                rb_group_issue<R2>(tx + oa, r[0]);
                rb_group_issue<R2>(tx + ob, r[1]);
                rb_group_issue<R2>(ty + oa, r[2]);
                rb_group_issue<R2>(ty + ob, r[3]);
                tmem_wait_ld_regs(r[0]);
                tmem_wait_ld_regs(r[1]);
                tmem_wait_ld_regs(r[2]);
                tmem_wait_ld_regs(r[3]);
                rb_group_unpack<R2>(r[0], xa);
                rb_group_unpack<R2>(r[1], xb);
                rb_group_unpack<R2>(r[2], ya);
                rb_group_unpack<R2>(r[3], yb);
            }
            // second forward pass: element k2 of group k1 becomes W_(k1 + R1 k2)
            dft<R2>(xa);
            dft<R2>(xb);
            dft<R2>(ya);
            dft<R2>(yb);
            if (pr != 0) {
                // k = ka + R1 k2 pairs with H - k = kb + R1 (R2 - 1 - k2)
#pragma unroll
                for (int k2 = 0; k2 < R2; ++k2)
                    rb_pair<UNB>(xa[k2], xb[R2 - 1 - k2], ya[k2], yb[R2 - 1 - k2], tw[ka + R1 * k2], xa[k2],
                                 xb[R2 - 1 - k2]);
            } else {
                // group 0: k = R1 k2 pairs with R1 (R2 - k2) (k2 = 0: k = 0; k2 = R2 / 2: k = H / 2)
#pragma unroll
                for (int k2 = 0; k2 <= R2 / 2; ++k2) {
                    const int c2 = (R2 - k2) % R2;
                    rb_pair<UNB>(xa[k2], xa[c2], ya[k2], ya[c2], tw[R1 * k2], xa[k2], xa[c2]);
                }
                // group R1 / 2: k = R1 / 2 + R1 k2 pairs with R1 / 2 + R1 (R2 - 1 - k2)
#pragma unroll
                for (int k2 = 0; k2 < R2 / 2; ++k2)
                    rb_pair<UNB>(xb[k2], xb[R2 - 1 - k2], yb[k2], yb[R2 - 1 - k2], tw[R1 / 2 + R1 * k2], xb[k2],
                                 xb[R2 - 1 - k2]);
            }
        }
        // first inverse pass: inverse DFT_R2 along k2, then w_H^-(n2 k1)
        dft_inv<R2>(xa);
        dft_inv<R2>(xb);
#pragma unroll
        for (int n2 = 1; n2 < R2; ++n2) {
            xa[n2] = c_mulconj(xa[n2], tw[2 * n2 * ka]);
            xb[n2] = c_mulconj(xb[n2], tw[2 * n2 * kb]);
        }
        rb_group_store<R2>(tx + oa, xa);
        rb_group_store<R2>(tx + ob, xb);
    }
}

// Z (m x D) = op(T16 Q16t^T x rowmul, Y) in blocks of L = 2 H.  Maps: T16 (fp16, box {64, 128},
// 128-byte swizzle), Q16t (fp16, box {64, 256}), Y (fp32, box {32, 128}, 128-byte swizzle), Z
// (fp32, box {16, 32}, 64-byte swizzle).
template <int H, bool UNB>
__global__ void __launch_bounds__(kRbThreads, 1)
    k_rbind_tc(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
               const __grid_constant__ CUtensorMap tmap_y, const __grid_constant__ CUtensorMap tmap_z,
               const __grid_constant__ RbParams p) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    RbCtl& c = *reinterpret_cast<RbCtl*>(smem_raw);
    float2* tw = reinterpret_cast<float2*>(smem_raw + (sizeof(RbCtl) + 15) / 16 * 16);
    const uint32_t off = ((raw + (uint32_t)kRbHead + 1023u) & ~1023u) - raw;
    unsigned* err = &g_err_rbind;
    if (off + kRbData > kRbSmemBytes) {  // uniform over the grid: every thread leaves here
        if (threadIdx.x == 0 && blockIdx.x == 0) atomicOr(err, GS_DEV_ERR_LAYOUT);
        return;
    }
    uint8_t* As = smem_raw + off;
    uint8_t* Bs = As + (size_t)kRbStages * kRbAStage;
    uint8_t* Ys = Bs + (size_t)kRbStages * kRbBStage;
    volatile int* abort_flag = &c.abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool lead = rank == 0;
    const long long pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
    const int ntiles = p.tiles > pair ? (int)((p.tiles - 1 - pair) / npairs + 1) : 0;
    // pair tile lt: rows tm 256 + [0, 256) (this CTA's: + 128 rank), columns tn 256 + [0, 256)
    auto tile_mn = [&](int lt, long long& tm, int& tn) {
        const long long tg = pair + (long long)lt * npairs;
        tm = tg / p.tiles_n;
        tn = (int)(tg % p.tiles_n);
    };
    if (threadIdx.x == 0) {
        for (int s = 0; s < kRbStages; ++s) {
            mbar_init(&c.full[s], 1);
            mbar_init(&c.empty[s], 1);
        }
        for (int s = 0; s < kRbYStages; ++s) {
            mbar_init(&c.y_full[s], 1);
            mbar_init(&c.y_empty[s], 4);  // one transform warp of each lane quadrant reads a box
        }
        mbar_init(&c.d_full, 1);
        mbar_init(&c.y_free, 2 * 4 * kRbSubs);  // the transform warps of both CTAs (the even CTA's is used)
        mbar_init(&c.mma_done, 1);
        c.abort_flag = 0;
        fence_barrier_init();
    }
    // w_L^j = e^(-2 pi i j / L), j < L (sincospif: the angle pi j / H is exact in its argument)
    for (int j = threadIdx.x; j < 2 * H; j += blockDim.x) {
        float s, co;
        sincospif((float)j / (float)H, &s, &co);
        tw[j] = make_float2(co, -s);
    }
    if (warp == 1) {
        tmem_alloc2(&c.tmem_base, 512);
        tmem_relinquish2();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();  // the even CTA's barriers exist before the odd CTA signals them
    tc_fence_after();
    const uint32_t tmem = c.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------------- T and Q K-blocks
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_last();
            RingPos rp;
            int it = 0;
            bool ok = true;
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                long long tm;
                int tn;
                tile_mn(lt, tm, tn);
                for (int kb = 0; kb < p.nkb; ++kb, ++it, rp.next(kRbStages)) {
                    if (!mbar_wait_1t(&c.empty[rp.idx], rp.phase ^ 1u, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    // both CTAs' halves complete on the even CTA's full barrier
                    if (lead) mbar_arrive_expect_tx(&c.full[rp.idx], 2u * (kRbAStage + kRbBStage));
                    const uint32_t fb = mapa_shared(smem_u32(&c.full[rp.idx]), 0);
                    tma_load_2d_pair(As + (size_t)rp.idx * kRbAStage, &tmap_a, fb, kb * kRbBK,
                                     (int)(tm * 2 * kRbBM + kRbBM * rank), pol);
                    tma_load_2d_pair(Bs + (size_t)rp.idx * kRbBStage, &tmap_b, fb, kb * kRbBK,
                                     tn * kRbBN + (kRbBN / 2) * (int)rank, pol);
                }
            }
            // the even CTA waits until every stage it expected (both CTAs' loads) has landed; the
            // odd CTA leaves only after the closing cluster barrier, which the even CTA reaches
            // after this drain
            if (lead)
                for (int j = std::max(0, it - kRbStages); j < it; ++j)
                    mbar_drain(&c.full[j % kRbStages], (uint32_t)(j / kRbStages) & 1u, err);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------- pair MMA issue (even CTA)
        if (lane == 0 && lead) {
            const uint32_t idesc = idesc2_f16_f32(kRbBN);
            RingPos rp;
            bool ok = true;
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                // the half this tile accumulates into held the previous tile's partner spectra, in both
                // CTAs (arrivals at cluster scope)
                if (lt > 0 && !mbar_wait_cluster(&c.y_free, (uint32_t)(lt - 1) & 1u, abort_flag, err)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)((lt & 1) * kRbBN);
                for (int kb = 0; kb < p.nkb; ++kb, rp.next(kRbStages)) {
                    if (!mbar_wait_1t(&c.full[rp.idx], rp.phase, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = sdesc_sw128(smem_u32(As + (size_t)rp.idx * kRbAStage));
                    const uint64_t bd = sdesc_sw128(smem_u32(Bs + (size_t)rp.idx * kRbBStage));
#pragma unroll
                    for (int k = 0; k < kRbBK / 16; ++k)
                        mma2_f16_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, (kb | k) != 0 ? 1u : 0u);
                    mma2_commit(&c.empty[rp.idx], 3);
                }
                if (ok) mma2_commit(&c.d_full, 3);
            }
            mma2_commit(&c.mma_done, 1);
            mbar_drain(&c.mma_done, 0, err);
        }
    } else if (warp == 2) {
        // ------------------------------------------------------------- partner rows
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_first();
            RingPos rp;
            int it = 0;
            bool ok = true;
            for (int lt = 0; lt < ntiles && ok; ++lt) {
                long long tm;
                int tn;
                tile_mn(lt, tm, tn);
                if (lt + 1 < ntiles) {  // the next tile's partner rows into L2 while this one streams
                    long long tm2;
                    int tn2;
                    tile_mn(lt + 1, tm2, tn2);
                    for (int cc = 0; cc < kRbChunks; ++cc)
                        if (tn2 * kRbBN + cc * kRbYCols < p.D)
                            tma_prefetch_2d(&tmap_y, tn2 * kRbBN + cc * kRbYCols, (int)(tm2 * 2 * kRbBM + kRbBM * rank));
                }
                for (int cc = 0; cc < kRbChunks; ++cc, ++it, rp.next(kRbYStages)) {
                    if (!mbar_wait_1t(&c.y_empty[rp.idx], rp.phase ^ 1u, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&c.y_full[rp.idx], (uint32_t)kRbYStage);
                    tma_load_2d(Ys + (size_t)rp.idx * kRbYStage, &tmap_y, &c.y_full[rp.idx],
                                tn * kRbBN + cc * kRbYCols, (int)(tm * 2 * kRbBM + kRbBM * rank), pol);
                }
            }
            for (int j = std::max(0, it - kRbYStages); j < it; ++j)
                mbar_drain(&c.y_full[j % kRbYStages], (uint32_t)(j / kRbYStages) & 1u, err);
        }
    } else {
        // ------------------------------------------------------------- transforms
        const int quad = warp & 3, sub = (warp - kRbEpi0) >> 2;
        const uint32_t lanes = (uint32_t)(32 * quad) << 16;
        const int rr = 32 * quad + lane;  // this thread's row of the tile
        // partner box cc of tile 0 into TMEM columns 256 + 32 cc of this quadrant's lanes; the stage
        // goes back to the producer at once (box cc of every tile sits in stage cc, phase lt & 1)
        auto copy_in0 = [&](int cc) -> bool {
            if (!mbar_wait_warp(&c.y_full[cc], 0u, abort_flag, err)) return false;
            const uint8_t* ys = Ys + (size_t)cc * kRbYStage + (size_t)rr * 128;
            uint32_t v[32];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const uint4 f = *reinterpret_cast<const uint4*>(ys + ((u ^ (rr & 7)) << 4));
                v[4 * u] = f.x;
                v[4 * u + 1] = f.y;
                v[4 * u + 2] = f.z;
                v[4 * u + 3] = f.w;
            }
            // release the stage only once every lane holds its values (the TMEM store consumes
            // them) and its reads are ordered before the TMA refill's writes (async proxy)
            tmem_st32(tmem + lanes + (uint32_t)(kRbBN + kRbYCols * cc), v);
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.y_empty[cc]);
            return true;
        };
        bool ok = ntiles > 0;
        if (ok) ok = copy_in0(sub) && copy_in0(sub + 4);
        for (int lt = 0; lt < ntiles; ++lt) {
            const uint32_t hx = (uint32_t)((lt & 1) * kRbBN), hy = (uint32_t)kRbBN - hx;
            long long tm;
            int tn;
            tile_mn(lt, tm, tn);
            const long long row0 = tm * 2 * kRbBM + kRbBM * rank;
            if (!quad_sync(quad, ok)) break;
            rb_strided<H, false, false>(tmem + lanes + hy, sub, 1.f, tw);
            ok = mbar_wait_warp(&c.d_full, (uint32_t)lt & 1u, abort_flag, err);
            if (ok) {
                tc_fence_after();
                const long long row = row0 + rr;
                const float rm = row < p.m ? p.rowmul[row] : 0.f;
                rb_strided<H, false, true>(tmem + lanes + hx, sub, rm, tw);
            }
            if (!quad_sync(quad, ok)) break;
            rb_middle<H, UNB>(tmem + lanes + hx, tmem + lanes + hy, sub, tw);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {  // this warp is done with the partner half
                if (lead)
                    mbar_arrive(&c.y_free);
                else
                    mbar_arrive_cluster(mapa_shared(smem_u32(&c.y_free), 0));
            }
            if (!quad_sync(quad, true)) break;
            rb_strided<H, true, true>(tmem + lanes + hx, sub, p.zscale, tw);
            if (!quad_sync(quad, true)) break;
            // output columns 32 cc .. 32 cc + 31 of this quadrant's rows (cc = sub, sub + 4).  Sixteen
            // columns at a time: the outputs come out of TMEM, the next tile's partner values for the
            // same columns come out of this warp's 32 rows of stage cc and go into TMEM in their place
            // (this half is the next tile's partner half), and the outputs take their place in the
            // stage; the 32 x 32 box then leaves by one tensor store (128-byte swizzle, as loaded).
            // After the last tile the stage has no refill pending, so its rows are free.
            const long long y = row0 + 32 * quad;
            const bool more = lt + 1 < ntiles;
            for (int h = 0; h < 2; ++h) {
                const int cc = sub + 4 * h;
                uint8_t* slice = Ys + (size_t)cc * kRbYStage + (size_t)(32 * quad) * 128;
                if (more && ok) ok = mbar_wait_warp(&c.y_full[cc], (uint32_t)(lt + 1) & 1u, abort_flag, err);
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    const uint32_t col = tmem + lanes + hx + (uint32_t)(kRbYCols * cc + 16 * hh);
                    float z[16];
                    tmem_ld16(col, z);
                    uint8_t* rowp = slice + lane * 128;
                    if (more && ok) {
                        uint32_t v[16];
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const uint4 f = *reinterpret_cast<const uint4*>(rowp + (((4 * hh + u) ^ (lane & 7)) << 4));
                            v[4 * u] = f.x;
                            v[4 * u + 1] = f.y;
                            v[4 * u + 2] = f.z;
                            v[4 * u + 3] = f.w;
                        }
                        tmem_st16(col, v);
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        *reinterpret_cast<float4*>(rowp + (((4 * hh + u) ^ (lane & 7)) << 4)) =
                            make_float4(z[4 * u], z[4 * u + 1], z[4 * u + 2], z[4 * u + 3]);
                }
                fence_proxy_async();
                __syncwarp();
                const int x = tn * kRbBN + cc * kRbYCols;
                if (lane == 0) {
                    if (x < p.D && y < p.m) tma_store_2d(&tmap_z, slice, x, (int)y);
                    bulk_commit();
                }
            }
            // both boxes read: the stages go back to the producer for the tile after next
            if (lane == 0) bulk_wait_read_0();
            __syncwarp();
            if (more && lane == 0) {
                mbar_arrive(&c.y_empty[sub]);
                mbar_arrive(&c.y_empty[sub + 4]);
            }
        }
        if (lane == 0) bulk_wait_all();
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync_all();  // neither CTA leaves while the other may still signal its barriers
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc2(tmem, 512);
    }
}

}  // namespace

bool rbind_tc_supported(int L, int D, const float* Y, long long ldy, const float* Z, int ldz) {
    if (L != 64 && L != 128 && L != kRbMaxL) return false;
    if (D % L || ldy < D || ldz < D) return false;
    // tensor maps: 16-byte aligned bases and row pitches
    return (uintptr_t)Y % 16 == 0 && (uintptr_t)Z % 16 == 0 && ldy % 4 == 0 && ldz % 4 == 0;
}

template <int H, bool UNB>
static cudaError_t rb_launch(int grid, size_t smem, cudaStream_t s, const CUtensorMap& ta, const CUtensorMap& tb,
                             const CUtensorMap& ty, const CUtensorMap& tz, const RbParams& p, int device) {
    static bool attr[64];
    if (!attr[device]) {
        cudaError_t e = cudaFuncSetAttribute(k_rbind_tc<H, UNB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr[device] = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kRbThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_rbind_tc<H, UNB>, ta, tb, ty, tz, p);
}

cudaError_t launch_rbind_tc(const gs_basis* h, const void* T16, long long ld16, long long m, const float* rowmul,
                            const float* Y, long long ldy, int L, bool unbind, float* Z, int ldz, int device,
                            cudaStream_t s) {
    if (m <= 0) return cudaSuccess;
    if (!h->Q16t || !rbind_tc_supported(L, h->D, Y, ldy, Z, ldz) || device < 0 || device >= 64)
        return cudaErrorInvalidValue;
    RbParams p;
    p.m = m;
    p.D = h->D;
    p.nkb = (h->r + kRbBK - 1) / kRbBK;
    p.tiles_n = (h->D + kRbBN - 1) / kRbBN;
    p.tiles = ((m + 2 * kRbBM - 1) / (2 * kRbBM)) * (long long)p.tiles_n;  // pair tiles of 256 rows
    p.zscale = 1.0f / (4.0f * (float)L);
    p.rowmul = rowmul;
    CUtensorMap ta, tb, ty, tz;
    if (!make_tmap_2d(&ta, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, T16, m, h->r, ld16, kRbBK, kRbBM,
                      CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&tb, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, h->Q16t, h->D, h->r, h->ldr16, kRbBK, kRbBN / 2,
                      CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&ty, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, Y, m, h->D, ldy, kRbYCols, kRbBM,
                      CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&tz, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, Z, m, h->D, ldz, kRbYCols, 32, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    const int grid = 2 * (int)std::min<long long>(std::max(sms / 2, 1), p.tiles);  // CTA pairs
    const size_t smem = kRbSmemBytes;
    switch (L) {
        case 64:
            return unbind ? rb_launch<32, true>(grid, smem, s, ta, tb, ty, tz, p, device)
                          : rb_launch<32, false>(grid, smem, s, ta, tb, ty, tz, p, device);
        case 128:
            return unbind ? rb_launch<64, true>(grid, smem, s, ta, tb, ty, tz, p, device)
                          : rb_launch<64, false>(grid, smem, s, ta, tb, ty, tz, p, device);
        default:
            return unbind ? rb_launch<128, true>(grid, smem, s, ta, tb, ty, tz, p, device)
                          : rb_launch<128, false>(grid, smem, s, ta, tb, ty, tz, p, device);
    }
}

unsigned take_device_error_rbind() {
    unsigned v = 0, z = 0;
    cudaMemcpyFromSymbol(&v, g_err_rbind, sizeof(v));
    if (v) cudaMemcpyToSymbol(g_err_rbind, &z, sizeof(z));
    return v;
}

}  // namespace gs
