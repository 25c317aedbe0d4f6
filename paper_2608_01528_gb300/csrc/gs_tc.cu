// gs_tc.cu -- tcgen05 (5th-generation tensor core) kernels for sm_103a.
//
// k_ps_tc: fused project + similarity for large query batches (paper Sec. 3.1
// t = U^T x, Sec. 2.2 scaled dot-product similarity, Sec. 3.2 Eq. 2-3).
//
//   GEMM1  Y = X Q^T   tcgen05.mma kind::f16, M = 128 queries, N = r (<= 256),
//                      fp32 accumulator in TMEM (two 256-column buffers so the
//                      epilogue of one tile overlaps the MMAs of the next).
//                      A = X: fp32 in HBM, streamed once by 16 loader warps with
//                      128-bit loads, rounded to fp16 (RN) and written straight
//                      into the 128-byte-swizzled K-major layout the MMA reads.
//                      B = Q: the basis' fixed fp16 copy (dithered rounding, see
//                      gs_build.cu), fetched per K-block by TMA (L2-resident).
//   GEMM2  S = Y R^T   fp32 FMA on CUDA cores in the epilogue warps, reading Y
//                      from TMEM with tcgen05.ld and skipping the zero tail of
//                      each row of R (R is lower echelon).  The dominant terms of
//                      S are single products Y_i R_ii, so this product needs fp32
//                      rather than a single fp16/tf32 rounding.
//   epilogue           scale / cosine (full-D ||x|| accumulated by the loaders
//                      from the fp32 input) / online softmax, argmax (lowest index
//                      on ties), maxval, optional Y and S stores.
//
// Work split: one persistent CTA per SM; each CTA takes a contiguous, balanced
// range of rows and cuts it into tiles of at most 128 rows, so every CTA moves
// the same number of bytes.  Warp roles:
//   warps 0-3   epilogue (warp w reads TMEM lanes 32w..32w+31 = rows of the tile)
//   warp  4     TMA producer of the Q tiles
//   warp  5     TMEM allocator and MMA issuer (one elected lane)
//   warps 6-17  X loaders / fp16 converters
// Every wait on an mbarrier is bounded (wall-clock limit): on expiry the CTA
// records GS_DEV_ERR_TIMEOUT, raises a CTA-wide abort flag so the other roles
// leave their loops, waits (bounded) for its own TMA copies and MMAs to land,
// frees TMEM and returns.

#include <float.h>

#include <algorithm>

#include "gs_internal.h"

namespace gs {
namespace {

__device__ unsigned g_err_tc = 0;

constexpr int kBM = 128;           // queries per tile (MMA M)
constexpr int kBK = 64;            // fp16 elements per K-block (one 128-byte row)
constexpr int kStagesMax = 4;
constexpr int kEpiWarps = 4;
constexpr int kLoadWarps = 12;
constexpr int kTmaWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kLoad0 = 6;
constexpr int kThreads = (kLoad0 + kLoadWarps) * 32;  // 576
constexpr int kRowGroups = kLoadWarps * 2;            // 24 rows per float4 column sweep
constexpr int kRowsPerLoader = (kBM + kRowGroups - 1) / kRowGroups;  // 6
constexpr int kTmemCols = 512;
constexpr int kCwChunk = 16;       // codewords per epilogue accumulator chunk
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // 2 s

// ----------------------------------------------------------------- PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ unsigned long long globaltimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait.  Returns false (and leaves the caller to unwind) on abort or timeout.
__device__ __noinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 255u) == 0) {
            if (*abort_flag) return false;
            if (globaltimer() - t0 > kWaitLimitNs) {
                *abort_flag = 1;
                atomicOr(&g_err_tc, GS_DEV_ERR_TIMEOUT);
                return false;
            }
        }
    }
}
// The same wait taken by a whole warp: every lane waits (each acquires the
// barrier's phase) and the warp leaves only together, so .sync.aligned
// instructions and warp shuffles after it always see a converged warp.
__device__ __forceinline__ bool mbar_wait_warp(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    const bool ok = mbar_wait(bar, parity, abort_flag);
    return __all_sync(0xffffffffu, ok);
}
// Wait used while unwinding: bounded, ignores the abort flag.
__device__ __noinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
    const unsigned long long t0 = globaltimer();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer() - t0 > kWaitLimitNs) {
            atomicOr(&g_err_tc, GS_DEV_ERR_TIMEOUT);
            return;
        }
    }
}
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ uint64_t l2_evict_last_policy() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                                            uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
        "l"(map), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(policy)
        : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, fp16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_f16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrives once on `bar` when every previously issued MMA of this thread has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_u32(bar))
                 : "memory");
}
// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
          "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
          "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (SBO), LBO unused for this layout (encoded 1), descriptor
// version 1 (bits 46-48), swizzle mode 2 = 128B (bits 61-63).
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}
// Instruction descriptor, kind::f16: D f32, A = B = f16, both K-major, N, M = 128.
__host__ __device__ constexpr uint32_t idesc_f16_f32(int n) {
    return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
}

struct TileRange {
    long long row0;
    int nrows;
};

// Balanced contiguous row range of CTA c, cut into at most-128-row tiles.
struct CtaRows {
    long long rb;
    long long rows;
    int ntiles;
    int tsize;
    __device__ CtaRows(long long N, int G, int c) {
        const long long base = N / G, rem = N % G;
        rows = base + (c < rem ? 1 : 0);
        rb = (long long)c * base + (c < rem ? c : rem);
        ntiles = (int)((rows + kBM - 1) / kBM);
        tsize = ntiles ? (int)((rows + ntiles - 1) / ntiles) : 0;
    }
    __device__ TileRange tile(int t) const {
        TileRange tr;
        tr.row0 = rb + (long long)t * tsize;
        const long long left = rb + rows - tr.row0;
        tr.nrows = (int)(left < tsize ? left : tsize);
        return tr;
    }
};

struct PsParams {
    const float* X;
    long long N;
    int ldx, D, r, npad, M, mpad, nkb, stages;
    const float* Rpad;      // mpad x npad fp32, zero padded copy of R
    const int* jlen16;      // per 16-codeword chunk: columns of R that can be nonzero
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

struct Smem {
    uint64_t a_full[kStagesMax], b_full[kStagesMax], empty[kStagesMax];
    uint64_t y_full[2], y_empty[2], xn_full[2], xn_empty[2], mma_done;
    float xn[2][kBM];
    uint32_t tmem_base;
    int abort_flag;
};

__global__ void __launch_bounds__(kThreads, 1)
    k_ps_tc(const __grid_constant__ CUtensorMap tmap_q, const PsParams p) {
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte aligned operand area (SW128 atoms), control block after it
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    const int S = p.stages;
    const uint32_t a_bytes = kBM * 128;
    const uint32_t b_bytes = (uint32_t)p.npad * 128;
    uint8_t* A = base;
    uint8_t* B = base + (size_t)S * a_bytes;
    Smem& sm = *reinterpret_cast<Smem*>(B + (size_t)S * b_bytes);
    volatile int* abort_flag = &sm.abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const CtaRows cr(p.N, gridDim.x, blockIdx.x);
    const int total_it = cr.ntiles * p.nkb;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&sm.a_full[s], kLoadWarps);
            mbar_init(&sm.b_full[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sm.y_full[b], 1);
            mbar_init(&sm.y_empty[b], kEpiWarps);
            mbar_init(&sm.xn_full[b], kLoadWarps);
            mbar_init(&sm.xn_empty[b], kEpiWarps);
        }
        mbar_init(&sm.mma_done, 1);
        sm.abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(&sm.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem_base;

    if (warp == kTmaWarp) {
        // ------------------------------------------------------------- Q tiles via TMA
        if (lane == 0) {
            const uint64_t pol = l2_evict_last_policy();
            int it = 0;
            for (; it < total_it; ++it) {
                const int s = it % S;
                const uint32_t ph = (uint32_t)(it / S) & 1u;
                if (!mbar_wait(&sm.empty[s], ph ^ 1u, abort_flag)) break;
                mbar_arrive_expect_tx(&sm.b_full[s], b_bytes);
                tma_load_2d(B + (size_t)s * b_bytes, &tmap_q, &sm.b_full[s], (it % p.nkb) * kBK, 0, pol);
            }
            // make sure every copy this thread started has landed before the CTA exits
            for (int j = std::max(0, it - S); j < it; ++j)
                mbar_drain(&sm.b_full[j % S], (uint32_t)(j / S) & 1u);
        }
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc = idesc_f16_f32(p.npad);
            int it = 0;
            bool ok = true;
            for (int t = 0; t < cr.ntiles && ok; ++t) {
                const int b = t & 1;
                if (!mbar_wait(&sm.y_empty[b], ((uint32_t)(t >> 1) & 1u) ^ 1u, abort_flag)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(b * 256);
                for (int kb = 0; kb < p.nkb; ++kb, ++it) {
                    const int s = it % S;
                    const uint32_t ph = (uint32_t)(it / S) & 1u;
                    if (!mbar_wait(&sm.a_full[s], ph, abort_flag) || !mbar_wait(&sm.b_full[s], ph, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = sdesc_sw128(smem_u32(A + (size_t)s * a_bytes));
                    const uint64_t bd = sdesc_sw128(smem_u32(B + (size_t)s * b_bytes));
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k)
                        mma_f16_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                                   (kb | k) != 0 ? 1u : 0u);
                    mma_commit(&sm.empty[s]);
                }
                if (ok) mma_commit(&sm.y_full[b]);
            }
            // all MMAs issued by this thread complete before TMEM is released
            mma_commit(&sm.mma_done);
            mbar_drain(&sm.mma_done, 0);
        }
    } else if (warp >= kLoad0) {
        // ------------------------------------------------------------- X loaders
        const int l = threadIdx.x - kLoad0 * 32;  // 0..383
        // thread l covers float4 column c4 = l % 16 of rows l/16 + 24u (u < 6, row < 128)
        float nrm[kRowsPerLoader];
#pragma unroll
        for (int u = 0; u < kRowsPerLoader; ++u) nrm[u] = 0.f;
        float amax = 0.f;
        float4 cur[kRowsPerLoader], nxt[kRowsPerLoader];
        const int c4 = l & 15;
        auto fetch = [&](int it, float4* v) {
            const int t = it / p.nkb, kb = it % p.nkb;
            const TileRange tr = cr.tile(t);
            const int col = kb * kBK + c4 * 4;
#pragma unroll
            for (int u = 0; u < kRowsPerLoader; ++u) {
                const int row = (l >> 4) + kRowGroups * u;
                float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
                if (row < tr.nrows) {
                    const float* src = p.X + (size_t)(tr.row0 + row) * p.ldx + col;
                    if (col + 3 < p.D) {
                        x = __ldcs(reinterpret_cast<const float4*>(src));
                    } else if (col < p.D) {
                        x.x = src[0];
                        if (col + 1 < p.D) x.y = src[1];
                        if (col + 2 < p.D) x.z = src[2];
                    }
                }
                v[u] = x;
            }
        };
        if (total_it > 0) fetch(0, cur);
        for (int it = 0; it < total_it; ++it) {
            if (it + 1 < total_it) fetch(it + 1, nxt);
            const int s = it % S;
            const uint32_t ph = (uint32_t)(it / S) & 1u;
            if (!mbar_wait_warp(&sm.empty[s], ph ^ 1u, abort_flag)) break;
            uint8_t* At = A + (size_t)s * a_bytes;
#pragma unroll
            for (int u = 0; u < kRowsPerLoader; ++u) {
                const int row = (l >> 4) + kRowGroups * u;
                if (row >= kBM) break;
                const float4 x = cur[u];
                nrm[u] = fmaf(x.x, x.x, fmaf(x.y, x.y, fmaf(x.z, x.z, fmaf(x.w, x.w, nrm[u]))));
                amax = fmaxf(amax, fmaxf(fmaxf(fabsf(x.x), fabsf(x.y)), fmaxf(fabsf(x.z), fabsf(x.w))));
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
            if (lane == 0) mbar_arrive(&sm.a_full[s]);
#pragma unroll
            for (int u = 0; u < kRowsPerLoader; ++u) cur[u] = nxt[u];
            if (it % p.nkb == p.nkb - 1) {
                // tile finished: ||x||^2 of this thread's rows -> shared, for cosine scores
                const int t = it / p.nkb, b = t & 1;
#pragma unroll
                for (int u = 0; u < kRowsPerLoader; ++u) {
                    float v = nrm[u];
                    v += __shfl_xor_sync(0xffffffffu, v, 8);
                    v += __shfl_xor_sync(0xffffffffu, v, 4);
                    v += __shfl_xor_sync(0xffffffffu, v, 2);
                    v += __shfl_xor_sync(0xffffffffu, v, 1);
                    nrm[u] = v;
                }
                if (!mbar_wait_warp(&sm.xn_empty[b], ((uint32_t)(t >> 1) & 1u) ^ 1u, abort_flag)) break;
                if ((lane & 15) == 0) {
#pragma unroll
                    for (int u = 0; u < kRowsPerLoader; ++u) {
                        const int row = (l >> 4) + kRowGroups * u;
                        if (row < kBM) sm.xn[b][row] = nrm[u];
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&sm.xn_full[b]);
#pragma unroll
                for (int u = 0; u < kRowsPerLoader; ++u) nrm[u] = 0.f;
            }
        }
        if (amax > 65504.f) atomicOr(&g_err_tc, GS_DEV_ERR_RANGE);
    } else {
        // ------------------------------------------------------------- epilogue (warps 0-3)
        const int i = threadIdx.x;  // row within the tile = TMEM lane
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        for (int t = 0; t < cr.ntiles; ++t) {
            const int b = t & 1;
            const uint32_t ph = (uint32_t)(t >> 1) & 1u;
            if (!mbar_wait_warp(&sm.y_full[b], ph, abort_flag)) break;
            tc_fence_after();
            if (!mbar_wait_warp(&sm.xn_full[b], ph, abort_flag)) break;
            const float xnorm = sqrtf(sm.xn[b][i]);
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.xn_empty[b]);
            const TileRange tr = cr.tile(t);
            const bool valid = i < tr.nrows;
            const long long row = tr.row0 + i;
            const uint32_t tb = tmem + lane_base + (uint32_t)(b * 256);
            float y[32];
            if (p.Y) {
                for (int jc = 0; jc < p.npad; jc += 32) {
                    tmem_ld32(tb + (uint32_t)jc, y);
                    if (valid) {
                        float* dst = p.Y + (size_t)row * p.ldy + jc;
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (jc + j < p.r) dst[j] = y[j];
                    }
                }
            }
            float best = -FLT_MAX, run_max = -FLT_MAX, run_sum = 0.f;
            int besti = 0;
            for (int ic = 0; ic < p.mpad; ic += kCwChunk) {
                float acc[kCwChunk];
#pragma unroll
                for (int q = 0; q < kCwChunk; ++q) acc[q] = 0.f;
                const int jl = p.jlen16[ic / kCwChunk];
                for (int jc = 0; jc < jl; jc += 16) {
                    float y16[16];
                    tmem_ld16(tb + (uint32_t)jc, y16);
#pragma unroll
                    for (int q = 0; q < kCwChunk; ++q) {
                        const float4* Rq = reinterpret_cast<const float4*>(p.Rpad + (size_t)(ic + q) * p.npad + jc);
#pragma unroll
                        for (int j4 = 0; j4 < 4; ++j4) {
                            const float4 rv = __ldg(Rq + j4);
                            acc[q] = fmaf(y16[4 * j4 + 0], rv.x, acc[q]);
                            acc[q] = fmaf(y16[4 * j4 + 1], rv.y, acc[q]);
                            acc[q] = fmaf(y16[4 * j4 + 2], rv.z, acc[q]);
                            acc[q] = fmaf(y16[4 * j4 + 3], rv.w, acc[q]);
                        }
                    }
                }
#pragma unroll
                for (int q = 0; q < kCwChunk; ++q) {
                    const int ci = ic + q;
                    if (ci >= p.M) break;
                    float g = p.scale * acc[q];
                    if (p.mode == GS_SCORE_COSINE) {
                        const float den = xnorm * p.cnorm[ci];
                        g = den > 0.f ? g / den : 0.f;
                    }
                    if (g > best) {
                        best = g;
                        besti = ci;
                    }
                    if (p.mode == GS_SCORE_SOFTMAX) {
                        const float nm = fmaxf(run_max, g);
                        run_sum = run_sum * __expf(run_max - nm) + __expf(g - nm);
                        run_max = nm;
                    }
                    if (p.S && valid) p.S[(size_t)row * p.lds + ci] = g;
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.y_empty[b]);
            if (!valid) continue;
            float outmax = best;
            if (p.mode == GS_SCORE_SOFTMAX) {
                const float inv = 1.f / run_sum;
                outmax = __expf(best - run_max) * inv;
                if (p.S) {
                    float* sr = p.S + (size_t)row * p.lds;
                    for (int ci = 0; ci < p.M; ++ci) sr[ci] = __expf(sr[ci] - run_max) * inv;
                }
            }
            if (p.argmax) p.argmax[row] = besti;
            if (p.maxval) p.maxval[row] = outmax;
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ----------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)p;
    }
    return fn;
}

// 2-D fp16 tensor map over a row-major (rows x cols, ld elements) matrix with a
// {64, box_rows} box and 128-byte swizzle; out-of-range elements read as zero.
bool make_tmap_f16(CUtensorMap* m, const void* ptr, int rows, int cols, int ld, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

__global__ void k_pad_r(const float* __restrict__ R, int M, int r, int ldr, float* __restrict__ Rp, int mpad,
                        int npad) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)mpad * npad) return;
    const int i = (int)(idx / npad), j = (int)(idx % npad);
    Rp[idx] = (i < M && j < r) ? R[(size_t)i * ldr + j] : 0.f;
}

// Per 16-codeword chunk: the leading columns of R (rounded up to the epilogue's
// 16-column step, never past npad) that hold any nonzero coefficient.
__global__ void k_jlen16(const int* __restrict__ rlen, int M, int nchunks, int npad, int* __restrict__ out) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= nchunks) return;
    int m = 0;
    for (int i = c * kCwChunk; i < min(M, c * kCwChunk + kCwChunk); ++i) m = max(m, rlen[i]);
    out[c] = min((m + 15) / 16 * 16, npad);
}

int num_sms(int dev) {
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

size_t ps_smem_bytes(int npad, int stages) {
    return 1024 + (size_t)stages * (kBM * 128 + (size_t)npad * 128) + sizeof(Smem);
}

int ps_stages(int npad) {
    for (int s = kStagesMax; s >= 2; --s)
        if (ps_smem_bytes(npad, s) <= 227 * 1024) return s;
    return 2;
}

}  // namespace

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
    if (h->r < 1 || h->r > 256) return GS_OK;  // no tensor-core similarity kernel for this basis
    const int npad = (h->r + 15) / 16 * 16;
    const int mpad = (h->M + kCwChunk - 1) / kCwChunk * kCwChunk;
    if (cudaMalloc(&h->tc_Rpad, sizeof(float) * (size_t)mpad * npad) != cudaSuccess) return GS_ERR_NOMEM;
    if (cudaMalloc(&h->tc_jlen16, sizeof(int) * (size_t)(mpad / kCwChunk)) != cudaSuccess) return GS_ERR_NOMEM;
    k_pad_r<<<(unsigned)(((long long)mpad * npad + 255) / 256), 256>>>(h->R, h->M, h->r, h->ldr, h->tc_Rpad, mpad,
                                                                       npad);
    k_jlen16<<<(mpad / kCwChunk + 127) / 128, 128>>>(h->rlen, h->M, mpad / kCwChunk, npad, h->tc_jlen16);
    if (cudaGetLastError() != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) return GS_ERR_CUDA;
    if (!make_tmap_f16(&h->tmap_q16, h->Q16, h->r, h->D, h->ldq16, npad)) return GS_ERR_CUDA;
    h->tc_npad = npad;
    h->tc_mpad = mpad;
    if (cudaFuncSetAttribute(k_ps_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)ps_smem_bytes(npad, ps_stages(npad))) != cudaSuccess)
        return GS_ERR_CUDA;
    // the fused kernel needs all of its threads resident in one CTA; otherwise the
    // basis simply has no tensor-core similarity path
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, k_ps_tc) != cudaSuccess) return GS_ERR_CUDA;
    h->has_tmap_q16 = fa.maxThreadsPerBlock >= kThreads;
    return GS_OK;
}

cudaError_t launch_ps_tc(const gs_basis* h, const float* X, long long N, int ldx, int mode, float scale, float* Y,
                         int ldy, float* S, int lds, int* argmax, float* maxval, cudaStream_t s) {
    if (!h->has_tmap_q16) return cudaErrorNotSupported;
    PsParams p;
    p.X = X;
    p.N = N;
    p.ldx = ldx;
    p.D = h->D;
    p.r = h->r;
    p.npad = h->tc_npad;
    p.M = h->M;
    p.mpad = h->tc_mpad;
    p.nkb = (h->D + kBK - 1) / kBK;
    p.stages = ps_stages(p.npad);
    p.Rpad = h->tc_Rpad;
    p.jlen16 = h->tc_jlen16;
    p.cnorm = h->cnorm;
    p.mode = mode;
    p.scale = scale;
    p.Y = Y;
    p.ldy = ldy;
    p.S = S;
    p.lds = lds;
    p.argmax = argmax;
    p.maxval = maxval;
    const long long tiles = (N + kBM - 1) / kBM;
    const int grid = (int)std::min<long long>(num_sms(h->device), tiles);
    k_ps_tc<<<grid, kThreads, ps_smem_bytes(p.npad, p.stages), s>>>(h->tmap_q16, p);
    return cudaGetLastError();
}

}  // namespace gs
