// gs_simt.cu -- fp32 CUDA-core kernels of the Gram-Space apply path.
//
// These kernels carry the small workloads (a handful of codewords, a few
// hundred queries: launch-latency bound) and the precise fp32 path that any
// shape can take (GS_PATH_SIMT).  The large-batch hot path is on tcgen05 in
// gs_tc.cu.
//
//  k_ps_warp      fused project + similarity, one warp per query, r <= 32
//                 (Sec. 3.1 t = U^T x; Sec. 2.2 similarity; Eq. 2-3)
//  k_coeffs_warp  similarity of Gram-loc queries, one warp per query, r <= 64 (Sec. 3.2, Eq. 2)
//  k_gemm         tiled fp32 GEMM with scale / cosine / bf16 epilogues; used for
//                 Y = X Q^T, S = Y R^T, V = P R (Sec. 2.2 / 3.3), Xhat = T Q
//                 (Sec. 3.1 / 3.3) and batched attention logits (Sec. 2.2)
//  k_row_finish   argmax / maxval / softmax over each score row
//  k_row_softmax  softmax over each attention row
//  k_rownorm      full-D query norms for cosine scores
//  k_group_argmax argmax / max of each score row within each group of a grouped codebook
//  k_bind16       block circular convolution / correlation (binding / unbinding), L % 16 == 0
//  k_bind8        the same for L % 8 == 0
//  k_bind_reg     the same for short blocks (L <= 32), one block per thread in registers
//  k_bind1        the same for any block length, one output per thread

#include <float.h>

#include <algorithm>

#include "gs_internal.h"

namespace gs {
namespace {

__device__ __forceinline__ float warp_sum(float v) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
// (value, index) argmax across a warp: larger value wins, lower index on ties.
__device__ __forceinline__ void warp_argmax(float& v, int& i) {
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, v, o);
        const int oi = __shfl_xor_sync(0xffffffffu, i, o);
        if (ov > v || (ov == v && oi < i)) {
            v = ov;
            i = oi;
        }
    }
}

// ----------------------------------------------------------------- fused small-r kernel
constexpr int kWarpR = 32;

__global__ void __launch_bounds__(256) k_ps_warp(const float* __restrict__ X, long long N, int ldx,
                                                  int D, const float* __restrict__ Q, int r,
                                                  const float* __restrict__ R, int ldr, int M,
                                                  const float* __restrict__ cnorm, int mode,
                                                  float scale, float* __restrict__ Y, int ldy,
                                                  float* __restrict__ S, int lds,
                                                  int* __restrict__ argmax,
                                                  float* __restrict__ maxval) {
    const int lane = threadIdx.x & 31;
    const long long n = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (n >= N) return;
    const float* x = X + (size_t)n * ldx;
    float y[kWarpR];
#pragma unroll
    for (int j = 0; j < kWarpR; ++j) y[j] = 0.f;
    float xx = 0.f;
    for (int d = lane; d < D; d += 32) {
        const float xv = x[d];
        xx = fmaf(xv, xv, xx);
#pragma unroll
        for (int j = 0; j < kWarpR; ++j)
            if (j < r) y[j] = fmaf(xv, __ldg(Q + (size_t)j * D + d), y[j]);
    }
#pragma unroll
    for (int j = 0; j < kWarpR; ++j)
        if (j < r) y[j] = warp_sum(y[j]);
    xx = warp_sum(xx);
    if (Y) {
        float mine = 0.f;
#pragma unroll
        for (int j = 0; j < kWarpR; ++j)
            if (j == lane) mine = y[j];
        if (lane < r) Y[(size_t)n * ldy + lane] = mine;
    }
    const float xnorm = sqrtf(xx);
    // scores: lane handles codewords i = lane, lane + 32, ...
    auto score = [&](int i) {
        const float* Ri = R + (size_t)i * ldr;
        float g = 0.f;
#pragma unroll
        for (int j = 0; j < kWarpR; ++j)
            if (j < r) g = fmaf(y[j], __ldg(Ri + j), g);
        g *= scale;
        if (mode == GS_SCORE_COSINE) {
            const float den = xnorm * cnorm[i];
            g = den > 0.f ? g / den : 0.f;
        }
        return g;
    };
    float bv = -FLT_MAX;
    int bi = 0x7fffffff;
    for (int i = lane; i < M; i += 32) {
        const float g = score(i);
        if (g > bv) {
            bv = g;
            bi = i;
        }
        if (S && mode != GS_SCORE_SOFTMAX) S[(size_t)n * lds + i] = g;
    }
    warp_argmax(bv, bi);
    if (bi == 0x7fffffff) bi = 0;
    float outmax = bv;
    if (mode == GS_SCORE_SOFTMAX) {
        float z = 0.f;
        for (int i = lane; i < M; i += 32) z += __expf(score(i) - bv);
        z = warp_sum(z);
        const float inv = 1.f / z;
        if (S)
            for (int i = lane; i < M; i += 32) S[(size_t)n * lds + i] = __expf(score(i) - bv) * inv;
        outmax = inv;
    }
    if (lane == 0) {
        if (argmax) argmax[n] = M > 0 ? bi : 0;
        if (maxval) maxval[n] = M > 0 ? outmax : 0.f;
    }
}

// Scores of queries given by their Gram-loc rows y (r <= 64): every lane holds the whole row
// (broadcast loads), lane l scores codewords l, l + 32, ...; ||y|| stands for ||x|| in the
// cosine mode (Eq. 3: equal for x in span(C)).  One launch for a small-batch lookup.
constexpr int kCoefR = 64;

__global__ void __launch_bounds__(256) k_coeffs_warp(const float* __restrict__ Yg, long long N, int ldy, int r,
                                                      const float* __restrict__ R, int ldr, int M,
                                                      const float* __restrict__ cnorm, int mode, float scale,
                                                      float* __restrict__ S, int lds, int* __restrict__ argmax,
                                                      float* __restrict__ maxval) {
    const int lane = threadIdx.x & 31;
    const long long n = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (n >= N) return;
    const float* yr = Yg + (size_t)n * ldy;
    float y[kCoefR];
    float yy = 0.f;
#pragma unroll
    for (int j = 0; j < kCoefR; ++j) {
        y[j] = j < r ? __ldg(yr + j) : 0.f;
        yy = fmaf(y[j], y[j], yy);
    }
    const float ynorm = sqrtf(yy);
    auto score = [&](int i) {
        const float* Ri = R + (size_t)i * ldr;
        float g = 0.f;
#pragma unroll
        for (int j = 0; j < kCoefR; ++j)
            if (j < r) g = fmaf(y[j], __ldg(Ri + j), g);
        g *= scale;
        if (mode == GS_SCORE_COSINE) {
            const float den = ynorm * cnorm[i];
            g = den > 0.f ? g / den : 0.f;
        }
        return g;
    };
    float bv = -FLT_MAX;
    int bi = 0x7fffffff;
    for (int i = lane; i < M; i += 32) {
        const float g = score(i);
        if (g > bv) {
            bv = g;
            bi = i;
        }
        if (S && mode != GS_SCORE_SOFTMAX) S[(size_t)n * lds + i] = g;
    }
    warp_argmax(bv, bi);
    if (bi == 0x7fffffff) bi = 0;
    float outmax = bv;
    if (mode == GS_SCORE_SOFTMAX) {
        float z = 0.f;
        for (int i = lane; i < M; i += 32) z += __expf(score(i) - bv);
        z = warp_sum(z);
        const float inv = 1.f / z;
        if (S)
            for (int i = lane; i < M; i += 32) S[(size_t)n * lds + i] = __expf(score(i) - bv) * inv;
        outmax = inv;
    }
    if (lane == 0) {
        if (argmax) argmax[n] = M > 0 ? bi : 0;
        if (maxval) maxval[n] = M > 0 ? outmax : 0.f;
    }
}

// ----------------------------------------------------------------- tiled GEMM
constexpr int kTM = 64, kTN = 64, kTK = 16;

template <int T>
__device__ __forceinline__ float ld_elem(const void* p, long long i) {
    if (T == MAT_F32) return __ldg((const float*)p + i);
    return __bfloat162float(((const __nv_bfloat16*)p)[i]);
}

// One 64 x 64 output tile (rows m0.., columns n0..) of batch b, or of K chunk kz with ksplit;
// called by every thread of the block.
template <int TA, int TB, int TC, bool BT>
__device__ __forceinline__ void gemm_tile(const GemmArgs& g, long long m0, int n0, int kz,
                                          float (&As)[kTK][kTM + 4], float (&Bs)[kTK][kTN + 4]) {
    const int tid = threadIdx.x;
    const int tx = tid % 16, ty = tid / 16;
    const bool split = g.ksplit > 1;
    const int b = split ? 0 : kz;
    const char* Ab = (const char*)g.A + (size_t)b * g.a_bstride * (TA == MAT_F32 ? 4 : 2);
    const char* Bb = (const char*)g.B + (size_t)b * g.b_bstride * (TB == MAT_F32 ? 4 : 2);
    int kend = g.k;
    if (BT && g.b_rowlen) {
        // rows n0..n0+63 of B are zero beyond their row length: stop at the max
        int mx = 0;
        for (int j = tid; j < kTN; j += 256)
            if (n0 + j < g.n) mx = max(mx, g.b_rowlen[n0 + j]);
        for (int o = 16; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        __shared__ int smx[8];
        if ((tid & 31) == 0) smx[tid >> 5] = mx;
        __syncthreads();
        mx = 0;
        for (int w = 0; w < 8; ++w) mx = max(mx, smx[w]);
        kend = min(kend, mx);
    }
    int kbeg = 0;
    if (split) {  // this block's chunk of K (chunks are whole kTK steps)
        const int chunk = ((g.k + g.ksplit - 1) / g.ksplit + kTK - 1) / kTK * kTK;
        kbeg = kz * chunk;
        kend = min(kend, kbeg + chunk);
    }
    float acc[4][4] = {};
    for (int k0 = kbeg; k0 < kend; k0 += kTK) {
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            const int e = tid + 256 * t;
            const int row = e / kTK, kk = e % kTK;
            const long long gm = m0 + row;
            const int gk = k0 + kk;
            As[kk][row] = (gm < g.m && gk < kend) ? ld_elem<TA>(Ab, gm * g.lda + gk) : 0.f;
            if (BT) {
                const int gn = n0 + row;
                Bs[kk][row] = (gn < g.n && gk < kend) ? ld_elem<TB>(Bb, (long long)gn * g.ldb + gk) : 0.f;
            } else {
                const int kk2 = e / kTN, col = e % kTN;
                const int gk2 = k0 + kk2, gn = n0 + col;
                Bs[kk2][col] = (gn < g.n && gk2 < kend) ? ld_elem<TB>(Bb, (long long)gk2 * g.ldb + gn) : 0.f;
            }
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kTK; ++kk) {
            float a[4], bb[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
            const float4 bv = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
            bb[0] = bv.x; bb[1] = bv.y; bb[2] = bv.z; bb[3] = bv.w;
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], bb[j], acc[i][j]);
        }
        __syncthreads();
    }
    char* Cb = (char*)g.C + (size_t)b * g.c_bstride * (TC == MAT_F32 ? 4 : 2);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const long long gm = m0 + ty * 4 + i;
        if (gm >= g.m) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int gn = n0 + tx * 4 + j;
            if (gn >= g.n) continue;
            float v = g.alpha * acc[i][j];
            if (g.rownorm) {
                const float den = g.rownorm[gm] * g.colnorm[gn];
                v = den > 0.f ? v / den : 0.f;
            }
            if (TC == MAT_F32) {
                if (split) g.kpart[((size_t)kz * g.m + gm) * g.n + gn] = v;
                else ((float*)Cb)[gm * g.ldc + gn] = v;
            } else {
                ((__nv_bfloat16*)Cb)[gm * g.ldc + gn] = __float2bfloat16_rn(v);
            }
        }
    }
}

template <int TA, int TB, int TC, bool BT>
__global__ void __launch_bounds__(256) k_gemm(GemmArgs g) {
    __shared__ float As[kTK][kTM + 4];
    __shared__ __align__(16) float Bs[kTK][kTN + 4];
    gemm_tile<TA, TB, TC, BT>(g, (long long)blockIdx.y * kTM, blockIdx.x * kTN, blockIdx.z, As, Bs);
}

// The gated product (gate_xn2): persistent blocks walk the 64 x 64 tiles, n fastest, and compute
// only those whose 64 rows hold a selected row; with no such row the launch is one pass over
// the norms.
template <int TA, int TB, int TC, bool BT>
__global__ void __launch_bounds__(256) k_gemm_gated(GemmArgs g) {
    __shared__ float As[kTK][kTM + 4];
    __shared__ __align__(16) float Bs[kTK][kTN + 4];
    const int tiles_n = (g.n + kTN - 1) / kTN;
    const long long tiles = (g.m + kTM - 1) / kTM * tiles_n;
    long long last_m0 = -1;
    bool any = false;
    for (long long t = blockIdx.x; t < tiles; t += gridDim.x) {
        const long long m0 = t / tiles_n * kTM;
        if (m0 != last_m0) {
            bool mine = false;
            if (threadIdx.x < kTM && m0 + threadIdx.x < g.m) {
                const long long i = m0 + threadIdx.x;
                const float xn2 = g.gate_xn2[i] + g.gate_xn2[g.gate_ld + i];
                mine = xn2 > 0.f && !(xn2 >= g.gate_lo && xn2 <= g.gate_hi);
            }
            any = __syncthreads_or(mine) != 0;
            last_m0 = m0;
        }
        if (any) gemm_tile<TA, TB, TC, BT>(g, m0, (int)(t % tiles_n) * kTN, 0, As, Bs);
    }
}

// C[i][j] = sum over z (in order) of part[z][i][j]: the split-K partials of k_gemm
__global__ void k_ksum(const float* __restrict__ part, int ks, long long m, int n, float* __restrict__ C,
                       long long ldc) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= m * n) return;
    float s = 0.f;
    for (int z = 0; z < ks; ++z) s += part[(size_t)z * m * n + idx];
    C[(idx / n) * ldc + idx % n] = s;
}

// ----------------------------------------------------------------- row kernels
__global__ void __launch_bounds__(256) k_row_finish(float* __restrict__ S, long long N, int M,
                                                     int lds, int softmax, int* __restrict__ argmax,
                                                     float* __restrict__ maxval) {
    const int lane = threadIdx.x & 31;
    const long long n = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (n >= N) return;
    float* s = S + (size_t)n * lds;
    float bv = -FLT_MAX;
    int bi = 0x7fffffff;
    for (int i = lane; i < M; i += 32) {
        const float g = s[i];
        if (g > bv) {
            bv = g;
            bi = i;
        }
    }
    warp_argmax(bv, bi);
    if (bi == 0x7fffffff) bi = 0;
    float outmax = bv;
    if (softmax) {
        float z = 0.f;
        for (int i = lane; i < M; i += 32) z += __expf(s[i] - bv);
        z = warp_sum(z);
        const float inv = 1.f / z;
        for (int i = lane; i < M; i += 32) s[i] = __expf(s[i] - bv) * inv;
        outmax = inv;
    }
    if (lane == 0) {
        if (argmax) argmax[n] = M > 0 ? bi : 0;
        if (maxval) maxval[n] = M > 0 ? outmax : 0.f;
    }
}

__global__ void __launch_bounds__(256) k_row_softmax(float* __restrict__ A, long long rows, int L,
                                                      long long ld) {
    const int lane = threadIdx.x & 31;
    const long long n = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (n >= rows) return;
    float* a = A + (size_t)n * ld;
    float mx = -FLT_MAX;
    for (int i = lane; i < L; i += 32) mx = fmaxf(mx, a[i]);
    mx = warp_max(mx);
    float z = 0.f;
    for (int i = lane; i < L; i += 32) z += __expf(a[i] - mx);
    z = warp_sum(z);
    const float inv = 1.f / z;
    for (int i = lane; i < L; i += 32) a[i] = __expf(a[i] - mx) * inv;
}

__global__ void __launch_bounds__(256) k_rownorm(const float* __restrict__ X, long long N, int ldx,
                                                  int D, float* __restrict__ out) {
    const int lane = threadIdx.x & 31;
    const long long n = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (n >= N) return;
    const float* x = X + (size_t)n * ldx;
    float s = 0.f;
    for (int d = lane; d < D; d += 32) s = fmaf(x[d], x[d], s);
    s = warp_sum(s);
    if (lane == 0) out[n] = sqrtf(s);
}

// Column ranges of the groups of a grouped codebook, passed by value.
struct GroupOffsets {
    int G;
    int off[kMaxGroups + 1];
};

// one warp per score row: for each group, the max over its columns and the index (within
// the group) of its first occurrence
__global__ void __launch_bounds__(256) k_group_argmax(const float* __restrict__ S, long long N, int lds,
                                                       const GroupOffsets go, int* __restrict__ argmax,
                                                       float* __restrict__ maxval) {
    const int lane = threadIdx.x & 31;
    const long long n = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (n >= N) return;
    const float* s = S + (size_t)n * lds;
    for (int g = 0; g < go.G; ++g) {
        const int c0 = go.off[g], c1 = go.off[g + 1];
        float bv = -INFINITY;
        int bi = c1;
        for (int j = c0 + lane; j < c1; j += 32) {
            const float v = s[j];
            if (v > bv) {  // columns rise with j: the first of equal values stays
                bv = v;
                bi = j;
            }
        }
        warp_argmax(bv, bi);
        if (lane == 0) {
            if (argmax) argmax[(size_t)n * go.G + g] = bi - c0;
            if (maxval) maxval[(size_t)n * go.G + g] = bv;
        }
    }
}

// Binding (UNB = false: Z_k = sum_j X_j Y_(k-j mod L)) or unbinding (UNB = true:
// Z_k = sum_j X_j Y_(j-k mod L)) within blocks of L components.  A CTA takes one block of
// 256 / tpr rows (tpr = min(L / 8, 256) threads per row) and stages the rows' X and Y
// blocks in shared memory, Y index-reversed for unbinding (Y'_m = Y_(-m mod L) turns the
// correlation into a convolution).  A thread computes eight consecutive outputs
// k0..k0+7: per eight-wide step of j it reads X_j..X_(j+7) (the same words for the whole
// row: broadcast) and the sixteen Y' values (k0 - j - 8 .. k0 - j + 7) mod L -- two aligned
// chunks, since L, k0 and j are multiples of 8 -- and does 64 fma.  ldy = 0: one partner row.
template <bool UNB>
__global__ void __launch_bounds__(256) k_bind8(const float* __restrict__ X, long long N, int ldx,
                                                const float* __restrict__ Y, long long ldy, int L,
                                                float* __restrict__ Z, int ldz, int zvec) {
    extern __shared__ float4 bind_sm[];
    const int tpr = min(L >> 3, 256);
    const int rpc = 256 / tpr;
    const int tr = threadIdx.x / tpr, tk = threadIdx.x - tr * tpr;
    const long long n = (long long)blockIdx.x * rpc + tr;
    const int b0 = blockIdx.y * L;
    float* xs = reinterpret_cast<float*>(bind_sm) + (size_t)tr * 2 * L;
    float* ys = xs + L;
    if (tr < rpc && n < N) {
        const float* x = X + (size_t)n * ldx + b0;
        const float* y = Y + (size_t)n * ldy + b0;
        for (int j = tk; j < L; j += tpr) {
            xs[j] = x[j];
            ys[j] = y[UNB ? (j == 0 ? 0 : L - j) : j];
        }
    }
    __syncthreads();
    if (tr >= rpc || n >= N) return;
    for (int k0 = 8 * tk; k0 < L; k0 += 8 * tpr) {
        float z[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) z[t] = 0.f;
        for (int j = 0; j < L; j += 8) {
            int a = k0 - j - 8;
            if (a < 0) a += L;
            const int c = a + 8 == L ? 0 : a + 8;
            float xv[8], w[16];
            *reinterpret_cast<float4*>(xv) = *reinterpret_cast<const float4*>(xs + j);
            *reinterpret_cast<float4*>(xv + 4) = *reinterpret_cast<const float4*>(xs + j + 4);
            *reinterpret_cast<float4*>(w) = *reinterpret_cast<const float4*>(ys + a);
            *reinterpret_cast<float4*>(w + 4) = *reinterpret_cast<const float4*>(ys + a + 4);
            *reinterpret_cast<float4*>(w + 8) = *reinterpret_cast<const float4*>(ys + c);
            *reinterpret_cast<float4*>(w + 12) = *reinterpret_cast<const float4*>(ys + c + 4);
#pragma unroll
            for (int u = 0; u < 8; ++u)
#pragma unroll
                for (int t = 0; t < 8; ++t) z[t] = fmaf(xv[u], w[8 + t - u], z[t]);
        }
        float* zo = Z + (size_t)n * ldz + b0 + k0;
        if (zvec) {
            reinterpret_cast<float4*>(zo)[0] = make_float4(z[0], z[1], z[2], z[3]);
            reinterpret_cast<float4*>(zo)[1] = make_float4(z[4], z[5], z[6], z[7]);
        } else {
#pragma unroll
            for (int t = 0; t < 8; ++t) zo[t] = z[t];
        }
    }
}

// The same with 16 x 16 register tiles (L % 16 == 0): a thread computes 16 consecutive
// outputs; per 16-wide step of j it reads X_j..X_(j+15) (broadcast within the row) and the
// 32 Y' values (k0 - j - 16 .. k0 - j + 15) mod L as two aligned 16-value segments, and does
// 256 fma.  Y' is stored with 4 words of padding after every 16 (segment i at word 20 i), so
// the segments of consecutive threads, 64 bytes apart unpadded, fall in disjoint banks.
template <bool UNB>
__global__ void __launch_bounds__(256) k_bind16(const float* __restrict__ X, long long N, int ldx,
                                                 const float* __restrict__ Y, long long ldy, int L,
                                                 float* __restrict__ Z, int ldz, int zvec) {
    extern __shared__ float4 bind_sm16[];
    const int tpr = min(L >> 4, 256);
    const int rpc = 256 / tpr;
    const int tr = threadIdx.x / tpr, tk = threadIdx.x - tr * tpr;
    const long long n = (long long)blockIdx.x * rpc + tr;
    const int b0 = blockIdx.y * L;
    const int Lp = L + (L >> 2);  // padded length of Y'
    float* xs = reinterpret_cast<float*>(bind_sm16) + (size_t)tr * (L + Lp);
    float* ys = xs + L;
    if (tr < rpc && n < N) {
        const float* x = X + (size_t)n * ldx + b0;
        const float* y = Y + (size_t)n * ldy + b0;
        for (int j = tk; j < L; j += tpr) {
            xs[j] = x[j];
            ys[j + (j >> 4) * 4] = y[UNB ? (j == 0 ? 0 : L - j) : j];
        }
    }
    __syncthreads();
    if (tr >= rpc || n >= N) return;
    for (int k0 = 16 * tk; k0 < L; k0 += 16 * tpr) {
        float z[16];
#pragma unroll
        for (int t = 0; t < 16; ++t) z[t] = 0.f;
        for (int j = 0; j < L; j += 16) {
            int a = k0 - j - 16;
            if (a < 0) a += L;
            const int c = a + 16 == L ? 0 : a + 16;
            float xv[16], w[32];
            const float* sa = ys + a + (a >> 2);
            const float* sc = ys + c + (c >> 2);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                *reinterpret_cast<float4*>(xv + 4 * q) = *reinterpret_cast<const float4*>(xs + j + 4 * q);
                *reinterpret_cast<float4*>(w + 4 * q) = *reinterpret_cast<const float4*>(sa + 4 * q);
                *reinterpret_cast<float4*>(w + 16 + 4 * q) = *reinterpret_cast<const float4*>(sc + 4 * q);
            }
#pragma unroll
            for (int u = 0; u < 16; ++u)
#pragma unroll
                for (int t = 0; t < 16; ++t) z[t] = fmaf(xv[u], w[16 + t - u], z[t]);
        }
        float* zo = Z + (size_t)n * ldz + b0 + k0;
        if (zvec) {
#pragma unroll
            for (int q = 0; q < 4; ++q)
                reinterpret_cast<float4*>(zo)[q] = make_float4(z[4 * q], z[4 * q + 1], z[4 * q + 2], z[4 * q + 3]);
        } else {
#pragma unroll
            for (int t = 0; t < 16; ++t) zo[t] = z[t];
        }
    }
}

// Short blocks (L <= 32, L % 4 == 0): one thread per block, its X and Y blocks in registers
// (float4 loads when every row start is 16-byte aligned), L sums of L products in j order;
// consecutive threads take consecutive blocks of a row, so a warp's loads and stores are
// contiguous.  The tiled kernels above would give each row's few outputs a thread group of
// their own and read rows 4 L bytes at a time.
template <int L, bool UNB>
__global__ void __launch_bounds__(256) k_bind_reg(const float* __restrict__ X, long long N, int nb, int ldx,
                                                   const float* __restrict__ Y, long long ldy,
                                                   float* __restrict__ Z, int ldz, int vec) {
    const long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= N * nb) return;
    const long long n = e / nb;
    const int b = (int)(e - n * nb);
    const float* x = X + (size_t)n * ldx + (size_t)b * L;
    const float* y = Y + (size_t)n * ldy + (size_t)b * L;
    float* z = Z + (size_t)n * ldz + (size_t)b * L;
    float xv[L], yv[L], zv[L];
    if (vec) {
#pragma unroll
        for (int q = 0; q < L / 4; ++q) {
            const float4 a = __ldcs(reinterpret_cast<const float4*>(x) + q);
            const float4 c = __ldg(reinterpret_cast<const float4*>(y) + q);
            xv[4 * q] = a.x, xv[4 * q + 1] = a.y, xv[4 * q + 2] = a.z, xv[4 * q + 3] = a.w;
            yv[4 * q] = c.x, yv[4 * q + 1] = c.y, yv[4 * q + 2] = c.z, yv[4 * q + 3] = c.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < L; ++j) {
            xv[j] = x[j];
            yv[j] = y[j];
        }
    }
#pragma unroll
    for (int k = 0; k < L; ++k) {
        float acc = 0.f;
#pragma unroll
        for (int j = 0; j < L; ++j) acc = fmaf(xv[j], yv[UNB ? (j - k + L) % L : (k - j + L) % L], acc);
        zv[k] = acc;
    }
    if (vec) {
#pragma unroll
        for (int q = 0; q < L / 4; ++q)
            __stcs(reinterpret_cast<float4*>(z) + q, make_float4(zv[4 * q], zv[4 * q + 1], zv[4 * q + 2], zv[4 * q + 3]));
    } else {
#pragma unroll
        for (int k = 0; k < L; ++k) z[k] = zv[k];
    }
}

// Any block length: one thread per output, operands read through the cache.
template <bool UNB>
__global__ void __launch_bounds__(256) k_bind1(const float* __restrict__ X, long long N, int D, int ldx,
                                                const float* __restrict__ Y, long long ldy, int L,
                                                float* __restrict__ Z, int ldz) {
    const long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= N * D) return;
    const long long n = e / D;
    const int d = (int)(e - n * D);
    const int b0 = d - d % L, k = d - b0;
    const float* x = X + (size_t)n * ldx + b0;
    const float* y = Y + (size_t)n * ldy + b0;
    float acc = 0.f;
    for (int j = 0; j < L; ++j) {
        int m = UNB ? j - k : k - j;
        if (m < 0) m += L;
        acc = fmaf(x[j], y[m], acc);
    }
    Z[(size_t)n * ldz + d] = acc;
}

inline unsigned rows_grid(long long n) { return (unsigned)((n + 7) / 8); }

}  // namespace

cudaError_t launch_ps_warp(const float* X, long long N, int ldx, int D, const float* Q, int r,
                           const float* R, int ldr, int M, const float* cnorm, int mode, float scale,
                           float* Y, int ldy, float* S, int lds, int* argmax, float* maxval,
                           cudaStream_t s) {
    k_ps_warp<<<rows_grid(N), 256, 0, s>>>(X, N, ldx, D, Q, r, R, ldr, M, cnorm, mode, scale, Y, ldy,
                                           S, lds, argmax, maxval);
    return cudaGetLastError();
}

cudaError_t launch_coeffs_warp(const float* Y, long long N, int ldy, int r, const float* R, int ldr, int M,
                               const float* cnorm, int mode, float scale, float* S, int lds, int* argmax,
                               float* maxval, cudaStream_t s) {
    if (N <= 0) return cudaSuccess;
    if (r > kCoefR) return cudaErrorInvalidValue;
    k_coeffs_warp<<<rows_grid(N), 256, 0, s>>>(Y, N, ldy, r, R, ldr, M, cnorm, mode, scale, S, lds, argmax,
                                               maxval);
    return cudaGetLastError();
}

cudaError_t launch_gemm_simt(const GemmArgs& g, cudaStream_t s) {
    if (g.m <= 0 || g.n <= 0 || g.batch <= 0) return cudaSuccess;
    if (g.ksplit > 1 && (g.batch != 1 || g.c_type != MAT_F32 || !g.kpart)) return cudaErrorInvalidValue;
    if (g.gate_xn2) {
        if (g.batch != 1 || g.ksplit > 1 || g.a_type != MAT_F32 || g.b_type != MAT_F32 || g.c_type != MAT_F32 ||
            !g.b_trans)
            return cudaErrorInvalidValue;
        int dev = 0, sms = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        const long long tiles = (g.m + kTM - 1) / kTM * ((g.n + kTN - 1) / kTN);
        const int grid = (int)std::min<long long>(tiles, 4LL * std::max(sms, 1));
        k_gemm_gated<MAT_F32, MAT_F32, MAT_F32, true><<<grid, 256, 0, s>>>(g);
        return cudaGetLastError();
    }
    dim3 grid((unsigned)((g.n + kTN - 1) / kTN), (unsigned)((g.m + kTM - 1) / kTM),
              (unsigned)(g.ksplit > 1 ? g.ksplit : g.batch));
    if (grid.y > 65535u) return cudaErrorInvalidConfiguration;
#define GS_GEMM_CASE(TA, TB, TC, BT)                                                        \
    if (g.a_type == TA && g.b_type == TB && g.c_type == TC && g.b_trans == BT) {            \
        k_gemm<TA, TB, TC, BT><<<grid, 256, 0, s>>>(g);                                     \
        if (g.ksplit > 1) {                                                                 \
            const long long mn = g.m * g.n;                                                 \
            k_ksum<<<(unsigned)((mn + 255) / 256), 256, 0, s>>>(g.kpart, g.ksplit, g.m, g.n, \
                                                                 (float*)g.C, g.ldc);       \
        }                                                                                   \
        return cudaGetLastError();                                                          \
    }
    GS_GEMM_CASE(MAT_F32, MAT_F32, MAT_F32, true)
    GS_GEMM_CASE(MAT_F32, MAT_F32, MAT_F32, false)
    GS_GEMM_CASE(MAT_F32, MAT_F32, MAT_BF16, false)
    GS_GEMM_CASE(MAT_BF16, MAT_F32, MAT_F32, false)
    GS_GEMM_CASE(MAT_BF16, MAT_BF16, MAT_F32, true)
#undef GS_GEMM_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_rownorm(const float* X, long long N, int ldx, int D, float* out, cudaStream_t s) {
    if (N <= 0) return cudaSuccess;
    k_rownorm<<<rows_grid(N), 256, 0, s>>>(X, N, ldx, D, out);
    return cudaGetLastError();
}

cudaError_t launch_row_finish(float* S, long long N, int M, int lds, bool softmax, int* argmax,
                              float* maxval, cudaStream_t s) {
    if (N <= 0) return cudaSuccess;
    k_row_finish<<<rows_grid(N), 256, 0, s>>>(S, N, M, lds, softmax ? 1 : 0, argmax, maxval);
    return cudaGetLastError();
}

cudaError_t launch_group_argmax(const float* S, long long N, int lds, const int* off, int G, int* argmax,
                                float* maxval, cudaStream_t s) {
    if (N <= 0) return cudaSuccess;
    if (G < 1 || G > kMaxGroups) return cudaErrorInvalidValue;
    GroupOffsets go;
    go.G = G;
    for (int g = 0; g <= G; ++g) go.off[g] = off[g];
    k_group_argmax<<<rows_grid(N), 256, 0, s>>>(S, N, lds, go, argmax, maxval);
    return cudaGetLastError();
}

template <int L>
static cudaError_t launch_bind_reg(const float* X, long long N, int D, int ldx, const float* Y, long long ldy,
                                   bool unbind, float* Z, int ldz, cudaStream_t s) {
    const int nb = D / L;
    const int vec = ((uintptr_t)X % 16 == 0 && (uintptr_t)Y % 16 == 0 && (uintptr_t)Z % 16 == 0 && ldx % 4 == 0 &&
                     ldy % 4 == 0 && ldz % 4 == 0)
                        ? 1
                        : 0;
    const unsigned blocks = (unsigned)((N * nb + 255) / 256);
    if (unbind)
        k_bind_reg<L, true><<<blocks, 256, 0, s>>>(X, N, nb, ldx, Y, ldy, Z, ldz, vec);
    else
        k_bind_reg<L, false><<<blocks, 256, 0, s>>>(X, N, nb, ldx, Y, ldy, Z, ldz, vec);
    return cudaGetLastError();
}

cudaError_t launch_bind(const float* X, long long N, int D, int ldx, const float* Y, long long ldy, int L, bool unbind,
                        float* Z, int ldz, cudaStream_t s) {
    if (N <= 0) return cudaSuccess;
    switch (L) {
        case 4: return launch_bind_reg<4>(X, N, D, ldx, Y, ldy, unbind, Z, ldz, s);
        case 8: return launch_bind_reg<8>(X, N, D, ldx, Y, ldy, unbind, Z, ldz, s);
        case 12: return launch_bind_reg<12>(X, N, D, ldx, Y, ldy, unbind, Z, ldz, s);
        case 16: return launch_bind_reg<16>(X, N, D, ldx, Y, ldy, unbind, Z, ldz, s);
        case 20: return launch_bind_reg<20>(X, N, D, ldx, Y, ldy, unbind, Z, ldz, s);
        case 24: return launch_bind_reg<24>(X, N, D, ldx, Y, ldy, unbind, Z, ldz, s);
        case 28: return launch_bind_reg<28>(X, N, D, ldx, Y, ldy, unbind, Z, ldz, s);
        case 32: return launch_bind_reg<32>(X, N, D, ldx, Y, ldy, unbind, Z, ldz, s);
        default: break;
    }
    // the staged kernels hold a row's X and Y blocks in shared memory: opt in past 48 KB once
    static bool opted[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!opted[dev]) {
        for (auto fn : {k_bind16<true>, k_bind16<false>, k_bind8<true>, k_bind8<false>}) {
            e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
            if (e != cudaSuccess) return e;
        }
        opted[dev] = true;
    }
    const int zvec = ((uintptr_t)Z % 16 == 0 && ldz % 4 == 0) ? 1 : 0;
    if (L % 16 == 0 && L <= kMaxBindFastL && D / L <= 65535) {
        const int tpr = std::min(L / 16, 256);
        const int rpc = 256 / tpr;
        const size_t smem = (size_t)rpc * (2 * L + L / 4) * sizeof(float);
        const dim3 grid((unsigned)((N + rpc - 1) / rpc), (unsigned)(D / L));
        if (unbind)
            k_bind16<true><<<grid, 256, smem, s>>>(X, N, ldx, Y, ldy, L, Z, ldz, zvec);
        else
            k_bind16<false><<<grid, 256, smem, s>>>(X, N, ldx, Y, ldy, L, Z, ldz, zvec);
        return cudaGetLastError();
    }
    if (L % 8 == 0 && L <= kMaxBindFastL && D / L <= 65535) {
        const int tpr = std::min(L / 8, 256);
        const int rpc = 256 / tpr;
        const size_t smem = (size_t)rpc * 2 * L * sizeof(float);
        const dim3 grid((unsigned)((N + rpc - 1) / rpc), (unsigned)(D / L));
        if (unbind)
            k_bind8<true><<<grid, 256, smem, s>>>(X, N, ldx, Y, ldy, L, Z, ldz, zvec);
        else
            k_bind8<false><<<grid, 256, smem, s>>>(X, N, ldx, Y, ldy, L, Z, ldz, zvec);
        return cudaGetLastError();
    }
    const long long total = N * D;
    const unsigned blocks = (unsigned)((total + 255) / 256);
    if (unbind)
        k_bind1<true><<<blocks, 256, 0, s>>>(X, N, D, ldx, Y, ldy, L, Z, ldz);
    else
        k_bind1<false><<<blocks, 256, 0, s>>>(X, N, D, ldx, Y, ldy, L, Z, ldz);
    return cudaGetLastError();
}

cudaError_t launch_row_softmax(float* A, long long rows, int L, long long ld, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    k_row_softmax<<<rows_grid(rows), 256, 0, s>>>(A, rows, L, ld);
    return cudaGetLastError();
}

}  // namespace gs
