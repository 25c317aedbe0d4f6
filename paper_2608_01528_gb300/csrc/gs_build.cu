// gs_build.cu -- basis construction (paper Sec. 3.1, Eq. 1; Sec. 3.3 "during
// initialization ... Gram-Schmidt orthogonalization of the codebook").
//
// Row-order Gram-Schmidt with two projection passes per row and a relative
// rank tolerance, in fp64 on the device.  Rows are taken in panels of
// kPanel.  For each panel:
//   1. load the panel rows V (fp64) and their norms ||c_i||;
//   2. twice (reorthogonalisation): H = V Q_old^T (tiled fp64 dot products
//      over D-slices, then a slice reduction that also accumulates R), and
//      V -= H Q_old -- a block projection against the basis built so far;
//   3. a cluster of CTAs (each owning a slice of the columns) runs Gram-Schmidt
//      with two passes over the panel's own new directions, row by row, decides
//      rank (||v|| > tol * ||c_i||), normalises and appends accepted rows to Q.
// In exact arithmetic this is the row-wise two-pass Gram-Schmidt of the
// paper's construction (projections onto orthonormal directions commute);
// the block passes against the old basis and the column slices within the
// panel are what make it data-parallel.
// The only host synchronisation is the read of the final rank r.
//
// Afterwards fp32 copies of Q and R are made for the caller, plus the
// fp16 operand copies of the tensor-core kernels (unbiased dithered rounding
// of the fp64 basis, see dither_half).

#include <algorithm>
#include <cmath>
#include <memory>
#include <vector>

#include "gs_internal.h"
#include "gs_tc_ptx.cuh"

namespace gs {
namespace {

constexpr int kPanel = 16;      // rows per panel
constexpr int kDotTileQ = 16;   // basis rows per dot tile
constexpr int kDotCols = 64;    // columns staged per step in the dot kernel
constexpr int kUpdCols = 64;    // columns per CTA in the update kernel
constexpr int kUpdJ = 128;      // coefficients staged per step in the update kernel

__device__ unsigned g_err_build = 0;

template <int NT>
__device__ double block_sum(double v, double* sh) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();  // protect sh from a previous use
    if (l == 0) sh[w] = v;
    __syncthreads();
    double t = 0.0;
    if (w == 0) {
        t = l < NT / 32 ? sh[l] : 0.0;
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (l == 0) sh[32] = t;
    }
    __syncthreads();
    return sh[32];
}

// 1. panel rows -> V (fp64), ||c_i||.  One CTA per panel row.
__global__ void __launch_bounds__(256) k_panel_load(const float* __restrict__ C, long long ldc, int D,
                                                     int p0, int normalize, double* __restrict__ V,
                                                     double* __restrict__ cn) {
    __shared__ double sh[33];
    const int k = blockIdx.x;
    const float* c = C + (size_t)(p0 + k) * ldc;
    double* v = V + (size_t)k * D;
    double ss = 0.0;
    for (int d = threadIdx.x; d < D; d += 256) {
        double x = (double)c[d];
        v[d] = x;
        ss += x * x;
    }
    double nrm = sqrt(block_sum<256>(ss, sh));
    if (normalize && nrm > 0.0) {
        const double sc = 1.0 / nrm;
        ss = 0.0;
        for (int d = threadIdx.x; d < D; d += 256) {
            double x = v[d] * sc;
            v[d] = x;
            ss += x * x;
        }
        nrm = sqrt(block_sum<256>(ss, sh));
    }
    if (threadIdx.x == 0) cn[p0 + k] = nrm;
}

// 2a. partial dot products Hp[slice][k][j] = sum_{d in slice} V[k][d] Qw[j][d]
//     for j < r0 (the rank at the start of this panel).  grid (q tiles, slices).
__global__ void __launch_bounds__(256) k_panel_dots(const double* __restrict__ V,
                                                     const double* __restrict__ Qw, int D, int bp,
                                                     const int* __restrict__ r_start, int dslice,
                                                     double* __restrict__ Hp, int ldh) {
    const int r0 = *r_start;
    const int j0 = blockIdx.x * kDotTileQ;
    if (j0 >= r0) return;
    const int d0 = blockIdx.y * dslice;
    const int d1 = min(D, d0 + dslice);
    __shared__ double sV[kPanel][kDotCols + 1];
    __shared__ double sQ[kDotTileQ][kDotCols + 1];
    const int ty = threadIdx.x / kDotTileQ;  // panel row
    const int tx = threadIdx.x % kDotTileQ;  // basis row within the tile
    double acc = 0.0;
    for (int dd = d0; dd < d1; dd += kDotCols) {
        for (int e = threadIdx.x; e < kPanel * kDotCols; e += 256) {
            const int rr = e / kDotCols, cc = e % kDotCols;
            const int d = dd + cc;
            sV[rr][cc] = (rr < bp && d < d1) ? V[(size_t)rr * D + d] : 0.0;
            sQ[rr][cc] = (j0 + rr < r0 && d < d1) ? Qw[(size_t)(j0 + rr) * D + d] : 0.0;
        }
        __syncthreads();
#pragma unroll 16
        for (int cc = 0; cc < kDotCols; ++cc) acc += sV[ty][cc] * sQ[tx][cc];
        __syncthreads();
    }
    if (ty < bp && j0 + tx < r0) Hp[((size_t)blockIdx.y * kPanel + ty) * ldh + j0 + tx] = acc;
}

// 2b. H[k][j] = sum over slices; R64[p0+k][j] += H[k][j].
__global__ void k_panel_reduce(const double* __restrict__ Hp, int nslices, int bp,
                               const int* __restrict__ r_start, int ldh, double* __restrict__ H,
                               double* __restrict__ R64, int ldr, int p0) {
    const int r0 = *r_start;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const int k = (int)(idx / ldh), j = (int)(idx % ldh);
    if (k >= bp || j >= r0) return;
    double s = 0.0;
    for (int t = 0; t < nslices; ++t) s += Hp[((size_t)t * kPanel + k) * ldh + j];
    H[(size_t)k * ldh + j] = s;
    R64[(size_t)(p0 + k) * ldr + j] += s;
}

// 2c. V[k][d] -= sum_{j < r0} H[k][j] Qw[j][d].  CTA = 64 columns x 4 row groups.
__global__ void __launch_bounds__(256) k_panel_update(double* __restrict__ V,
                                                       const double* __restrict__ Qw, int D, int bp,
                                                       const int* __restrict__ r_start,
                                                       const double* __restrict__ H, int ldh) {
    const int r0 = *r_start;
    if (r0 == 0) return;
    __shared__ double sH[kPanel][kUpdJ];
    const int d = blockIdx.x * kUpdCols + (threadIdx.x % kUpdCols);
    const int kg = threadIdx.x / kUpdCols;  // 4 groups of 4 rows
    double acc[4] = {0.0, 0.0, 0.0, 0.0};
    for (int jc = 0; jc < r0; jc += kUpdJ) {
        const int nj = min(kUpdJ, r0 - jc);
        for (int e = threadIdx.x; e < kPanel * kUpdJ; e += 256) {
            const int kk = e / kUpdJ, cc = e % kUpdJ;
            sH[kk][cc] = (kk < bp && cc < nj) ? H[(size_t)kk * ldh + jc + cc] : 0.0;
        }
        __syncthreads();
        if (d < D) {
            for (int cc = 0; cc < nj; ++cc) {
                const double q = Qw[(size_t)(jc + cc) * D + d];
#pragma unroll
                for (int t = 0; t < 4; ++t) acc[t] += sH[kg * 4 + t][cc] * q;
            }
        }
        __syncthreads();
    }
    if (d < D) {
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            const int k = kg * 4 + t;
            if (k < bp) V[(size_t)k * D + d] -= acc[t];
        }
    }
}

// 3. Gram-Schmidt with two passes inside the panel, rank decision, normalisation and append, on a
//    cluster of kMgsCtas CTAs: CTA c owns columns [c S, (c + 1) S) of every vector (S = ceil(D /
//    kMgsCtas)), so the fp64 arithmetic of a row is spread over kMgsCtas SMs (GB300's fp64 rate
//    per SM is low: one CTA doing this took 1.5 ms per 16-row panel of 10,000-wide rows).  Each
//    pass takes the projections of v on all of the panel's new directions at once (classical
//    Gram-Schmidt, twice: the same factorisation as the row-by-row passes in exact arithmetic, and
//    as stable with the second pass), so a row needs three sums over the whole row: the two passes'
//    projections and the norm.  A sum is reduced in each CTA (a 16-lane butterfly, then across the
//    warps), and each CTA's partials are stored into every CTA's shared memory with st.async, whose
//    bytes complete on the receiver's mbarrier for that buffer (no release fence on the sending
//    side; a cluster barrier per sum cost ~11 us); every CTA adds the partials in CTA order, so all
//    hold the same values, take the same rank decisions and run the same sums.  Partial sums
//    alternate between two buffers: a CTA posts sum n + 2 only after it has every partial of sum
//    n + 1, which each CTA posts after reading sum n, so a buffer is never overwritten while read.
//    Every wait is bounded (on expiry: GS_DEV_ERR_TIMEOUT, and the kernel runs on to its end).
constexpr int kMgsCtas = 8;
constexpr int kMgsThreads = 256;
static_assert(kPanel == 16, "the sums' butterfly gives lane l entry l & 15");

__global__ void __launch_bounds__(kMgsThreads) k_panel_gs2(double* __restrict__ V, double* __restrict__ Qw, int D,
                                                          int bp, int p0, double tau, const double* __restrict__ cn,
                                                          double* __restrict__ R64, int ldr, int* __restrict__ r_dev,
                                                          int rmax) {
    using namespace ptx;
    __shared__ double part[2][kMgsCtas][kPanel];  // per sum: every CTA's partials (stored by that CTA)
    __shared__ double red[kMgsThreads / 32][kPanel];
    __shared__ uint64_t pbar[2];                  // one barrier per partial buffer: 1 arrival + the bytes
    __shared__ double total[kPanel];              // the last sum, added once for the whole CTA
    const uint32_t rank = cluster_ctarank();
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int S = (D + kMgsCtas - 1) / kMgsCtas;
    const int c0 = (int)rank * S, c1 = min(D, c0 + S);
    const int r0 = *r_dev;
    int r = r0, nsum = 0;
    bool ok = true;  // false once a wait has run out (the results are then flagged as an error)
    if (tid == 0) {
        mbar_init(&pbar[0], 1);
        mbar_init(&pbar[1], 1);
        fence_barrier_init();
    }
    cluster_sync_all();  // every CTA's barriers exist before anyone stores into its memory

    // the sum over the cluster of acc[0..kPanel) (this thread's part): reduced in the CTA, stored into
    // every CTA, added in CTA order; the result is identical in every thread of every CTA
    auto cluster_sum = [&](double (&acc)[kPanel], double (&out)[kPanel]) {
        // warp: a butterfly over the lane bits 3..0 leaves lane l with the sum of entry l & 15 over
        // its half-warp (after the step with lane bit b a lane keeps the entries whose index has bit
        // b equal to its own), then the two half-warps are added: 16 shuffles instead of 80
#pragma unroll
        for (int wb = kPanel / 2; wb >= 1; wb >>= 1) {
            const bool up = (lane & wb) != 0;
#pragma unroll
            for (int j = 0; j < wb; ++j) {
                const double send = up ? acc[j] : acc[j + wb];
                const double keep = up ? acc[j + wb] : acc[j];
                acc[j] = keep + __shfl_xor_sync(0xffffffffu, send, wb);
            }
        }
        acc[0] += __shfl_xor_sync(0xffffffffu, acc[0], 16);
        __syncthreads();  // red and the last sum's buffer have been read by every thread of this CTA
        if (lane < kPanel) red[w][lane] = acc[0];
        __syncthreads();
        const int slot = nsum & 1;
        const uint32_t parity = (uint32_t)(nsum >> 1) & 1u;
        if (tid == 0) mbar_arrive_expect_tx(&pbar[slot], (uint32_t)(kMgsCtas * kPanel * sizeof(double)));
        if (tid < kPanel * kMgsCtas) {
            const int j = tid % kPanel, dest = tid / kPanel;
            double v = 0.0;
            for (int ww = 0; ww < kMgsThreads / 32; ++ww) v += red[ww][j];
            st_async_f64(mapa_shared(smem_u32(&part[slot][rank][j]), (uint32_t)dest), v,
                         mapa_shared(smem_u32(&pbar[slot]), (uint32_t)dest));
        }
        // sixteen threads wait for every CTA's partials and add them (fp64 adds run at a low rate
        // on GB300: every thread adding all 128 had cost ~9 us a sum)
        if (tid < kPanel) {
            if (ok) {
                const unsigned long long t0 = globaltimer();
                for (uint32_t it = 0; !mbar_try_wait_cluster(&pbar[slot], parity); ++it)
                    if ((it & 255u) == 255u && globaltimer() - t0 > kWaitLimitNs) {
                        atomicOr(&g_err_build, GS_DEV_ERR_TIMEOUT);
                        ok = false;
                        break;
                    }
            }
            double v = 0.0;
            for (int c = 0; c < kMgsCtas; ++c) v += part[slot][c][tid];
            total[tid] = v;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < kPanel; ++j) out[j] = total[j];
        ++nsum;
    };

    for (int k = 0; k < bp; ++k) {
        double* v = V + (size_t)k * D;
        double* Rrow = R64 + (size_t)(p0 + k) * ldr;
        const int nj = r - r0;  // the panel's new directions so far
        for (int pass = 0; pass < 2; ++pass) {
            double acc[kPanel], h[kPanel];
#pragma unroll
            for (int j = 0; j < kPanel; ++j) acc[j] = 0.0;
            for (int d = c0 + tid; d < c1; d += kMgsThreads) {
                const double x = v[d];
#pragma unroll
                for (int j = 0; j < kPanel; ++j)
                    if (j < nj) acc[j] += Qw[(size_t)(r0 + j) * D + d] * x;
            }
            cluster_sum(acc, h);
            for (int d = c0 + tid; d < c1; d += kMgsThreads) {
                double x = v[d];
#pragma unroll
                for (int j = 0; j < kPanel; ++j)
                    if (j < nj) x -= h[j] * Qw[(size_t)(r0 + j) * D + d];
                v[d] = x;
            }
            if (rank == 0 && tid < nj) {
                double hv = 0.0;  // h[tid] without a dynamic index (which would move h to local memory)
#pragma unroll
                for (int j = 0; j < kPanel; ++j)
                    if (j == tid) hv = h[j];
                Rrow[r0 + tid] += hv;
            }
        }
        double acc[kPanel], nn[kPanel];
#pragma unroll
        for (int j = 0; j < kPanel; ++j) acc[j] = 0.0;
        for (int d = c0 + tid; d < c1; d += kMgsThreads) acc[0] += v[d] * v[d];
        cluster_sum(acc, nn);
        const double nu = sqrt(nn[0]);
        if (nu > tau * cn[p0 + k] && r < rmax) {
            double* q = Qw + (size_t)r * D;
            for (int d = c0 + tid; d < c1; d += kMgsThreads) q[d] = v[d] / nu;
            if (rank == 0 && tid == 0) Rrow[r] = nu;
            ++r;
        }
    }
    if (rank == 0 && tid == 0) *r_dev = r;
    cluster_sync_all();  // no CTA leaves while a peer may still store into its memory
}

// ----------------------------------------------------------------- finalisation
__global__ void k_cast_rows(const double* __restrict__ src, long long lds, float* __restrict__ dst,
                            long long ldd, int rows, int cols) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)rows * cols) return;
    const int i = (int)(idx / cols), j = (int)(idx % cols);
    dst[(size_t)i * ldd + j] = (float)src[(size_t)i * lds + j];
}

// rlen[i] = 1 + last nonzero column of R_i among the first r; chunk max per 32 rows
__global__ void k_rlen(const double* __restrict__ R64, int ldr, int M, int r, int* __restrict__ rlen) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= M) return;
    int last = 0;
    for (int j = 0; j < r; ++j)
        if (R64[(size_t)i * ldr + j] != 0.0) last = j + 1;
    rlen[i] = last;
}

__global__ void k_rlen_chunk(const int* __restrict__ rlen, int M, int* __restrict__ out) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c * 32 >= M) return;
    int m = 0;
    for (int i = c * 32; i < min(M, c * 32 + 32); ++i) m = max(m, rlen[i]);
    out[c] = m;
}

// Counter-based 32-bit mixer (the "lowbias32" integer hash).
__device__ __forceinline__ uint32_t mix32(uint32_t x) {
    x ^= x >> 16;
    x *= 0x7feb352du;
    x ^= x >> 15;
    x *= 0x846ca68bu;
    x ^= x >> 16;
    return x;
}

// Unbiased dithered (stochastic) rounding of a basis entry to fp16: round to
// the fp16 neighbour below or above in magnitude with probability given by the
// remainder, using a fixed hash of the element index.  The expected value is
// the input, and the rounding errors of different elements are independent
// even where the basis has few distinct magnitudes (the first basis vector of
// a bipolar codebook is +-1/sqrt(D) everywhere), so in X Q^T they average out
// over D instead of adding up coherently.  |q| <= 1, so no overflow.
__device__ __forceinline__ __half dither_half(double qd, unsigned long long index) {
    const float f = (float)qd;
    const __half lo = __float2half_rz(f);
    const float lof = __half2float(lo);
    if (lof == f) return lo;
    const __half hi = __ushort_as_half((unsigned short)(__half_as_ushort(lo) + 1));
    const float hif = __half2float(hi);
    const float frac = (f - lof) / (hif - lof);
    const uint32_t hsh = mix32((uint32_t)index ^ mix32((uint32_t)(index >> 32) + 0x9e3779b9u));
    const float u = (float)(hsh >> 8) * (1.0f / 16777216.0f);
    return u < frac ? hi : lo;
}

// Q16[j][d] (r x ldq) and Q16t[d][j] (D x ldt) from Qw (fp64, r x D); zero padding.
__global__ void k_q16(const double* __restrict__ Qw, int r, int D, __half* __restrict__ Q16, int ldq,
                      __half* __restrict__ Q16t, int ldt) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)r * ldq) return;
    const int j = (int)(idx / ldq), d = (int)(idx % ldq);
    __half hv = __float2half(0.0f);
    if (d < D) hv = dither_half(Qw[(size_t)j * D + d], (unsigned long long)j * D + d);
    Q16[idx] = hv;
    if (Q16t && d < D) Q16t[(size_t)d * ldt + j] = hv;
}

// dst[d][j] (cols x ldt fp16) = dithered rounding of src[j][d] (rows x cols fp32, ld lds), through
// 32 x 32 tiles in shared memory (coalesced reads and writes); the transposed operand of a
// reconstruction from fp32 rows that are not the basis itself (the basis bound with a partner).
__global__ void k_f16t_dither(const float* __restrict__ src, int rows, int cols, long long lds,
                              __half* __restrict__ dst, long long ldt) {
    __shared__ float tile[32][33];
    const int j0 = blockIdx.y * 32, d0 = blockIdx.x * 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 256 threads: 8 rows per step
    for (int k = ty; k < 32; k += 8) {
        const int j = j0 + k, d = d0 + tx;
        tile[k][tx] = (j < rows && d < cols) ? src[(size_t)j * lds + d] : 0.f;
    }
    __syncthreads();
    for (int k = ty; k < 32; k += 8) {
        const int d = d0 + k, j = j0 + tx;
        if (d < cols && j < rows)
            dst[(size_t)d * ldt + j] = dither_half((double)tile[tx][k], (unsigned long long)j * cols + d);
    }
}

__global__ void k_zero_half(__half* p, long long n) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) p[i] = __float2half(0.0f);
}

inline unsigned grid1(long long n, int b) { return (unsigned)((n + b - 1) / b); }

// fp32 rows (ld lds) -> fp64 rows (ld ldd)
__global__ void k_widen_rows(const float* __restrict__ src, long long lds, double* __restrict__ dst,
                             long long ldd, int rows, int cols) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)rows * cols) return;
    const int i = (int)(idx / cols), j = (int)(idx % cols);
    dst[(size_t)i * ldd + j] = (double)src[(size_t)i * lds + j];
}

// ||R_i|| in fp64, one thread per row (C = R Q with orthonormal Q, so this is ||c_i||)
__global__ void k_row_norms64(const double* __restrict__ R64, int ldr, int M, int r, double* __restrict__ cn) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= M) return;
    double ss = 0.0;
    for (int j = 0; j < r; ++j) ss += R64[(size_t)i * ldr + j] * R64[(size_t)i * ldr + j];
    cn[i] = sqrt(ss);
}

struct DevBuf {
    void* p = nullptr;
    ~DevBuf() { if (p) cudaFree(p); }
};

}  // namespace

unsigned take_device_error_build() {
    unsigned v = 0, z = 0;
    cudaMemcpyFromSymbol(&v, g_err_build, sizeof(v));
    if (v) cudaMemcpyToSymbol(g_err_build, &z, sizeof(z));
    return v;
}

#define GS_CK(x)                                                     \
    do {                                                             \
        cudaError_t e_ = (x);                                        \
        if (e_ != cudaSuccess) {                                     \
            return e_ == cudaErrorMemoryAllocation ? GS_ERR_NOMEM : GS_ERR_CUDA; \
        }                                                            \
    } while (0)

gs_status finalize_basis(const double* Qw, const double* R64, int ldr, const double* cn, int M, int D, int r,
                         cudaStream_t s, gs_basis* h);

// The fp64 factorisation C = R Q of M rows of C (Q: r x D orthonormal rows, R: M x r lower
// echelon, ldr = min(M, D); cn: the rows' norms), kept on the device.
struct Factor {
    double* Qw = nullptr;
    double* R64 = nullptr;
    double* cn = nullptr;
    int r = 0, ldr = 1;
    Factor() = default;
    Factor(const Factor&) = delete;
    Factor& operator=(const Factor&) = delete;
    ~Factor() {
        cudaFree(Qw);
        cudaFree(R64);
        cudaFree(cn);
    }
};

gs_status factor_rows(const float* C, int M, int D, int ldc, double tau, bool normalize, cudaStream_t s,
                      Factor& f) {
    const int rmax = std::min(M, D);
    const int ldr = rmax;                       // R64 leading dimension
    const int ldh = std::max(1, ((M + 15) / 16) * 16);  // >= any r0
    const int dslice = std::max(kDotCols, ((D + 7) / 8 + kDotCols - 1) / kDotCols * kDotCols);
    const int nslices = (D + dslice - 1) / dslice;

    DevBuf bV, bH, bHp, br;
    GS_CK(cudaMalloc(&bV.p, sizeof(double) * (size_t)kPanel * D));
    GS_CK(cudaMalloc(&f.Qw, sizeof(double) * (size_t)rmax * D));
    GS_CK(cudaMalloc(&f.R64, sizeof(double) * (size_t)M * ldr));
    GS_CK(cudaMalloc(&bH.p, sizeof(double) * (size_t)kPanel * ldh));
    GS_CK(cudaMalloc(&bHp.p, sizeof(double) * (size_t)nslices * kPanel * ldh));
    GS_CK(cudaMalloc(&f.cn, sizeof(double) * (size_t)M));
    GS_CK(cudaMalloc(&br.p, sizeof(int)));
    double* V = (double*)bV.p;
    double* Qw = f.Qw;
    double* R64 = f.R64;
    double* H = (double*)bH.p;
    double* Hp = (double*)bHp.p;
    double* cn = f.cn;
    int* r_dev = (int*)br.p;
    GS_CK(cudaMemsetAsync(R64, 0, sizeof(double) * (size_t)M * ldr, s));
    GS_CK(cudaMemsetAsync(r_dev, 0, sizeof(int), s));

    for (int p0 = 0; p0 < M; p0 += kPanel) {
        const int bp = std::min(kPanel, M - p0);
        k_panel_load<<<bp, 256, 0, s>>>(C, ldc, D, p0, normalize ? 1 : 0, V, cn);
        if (p0 > 0) {
            const int qt = (std::min(p0, rmax) + kDotTileQ - 1) / kDotTileQ;
            for (int pass = 0; pass < 2; ++pass) {
                k_panel_dots<<<dim3(qt, nslices), 256, 0, s>>>(V, Qw, D, bp, r_dev, dslice, Hp, ldh);
                k_panel_reduce<<<grid1((long long)bp * ldh, 256), 256, 0, s>>>(Hp, nslices, bp, r_dev,
                                                                                ldh, H, R64, ldr, p0);
                k_panel_update<<<grid1(D, kUpdCols), 256, 0, s>>>(V, Qw, D, bp, r_dev, H, ldh);
            }
        }
        {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(kMgsCtas);
            cfg.blockDim = dim3(kMgsThreads);
            cfg.stream = s;
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = kMgsCtas;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            cfg.attrs = at;
            cfg.numAttrs = 1;
            if (kMgsCtas > 8)
                GS_CK(cudaFuncSetAttribute(k_panel_gs2, cudaFuncAttributeNonPortableClusterSizeAllowed, 1));
            GS_CK(cudaLaunchKernelEx(&cfg, k_panel_gs2, V, Qw, D, bp, p0, tau, (const double*)cn, R64, ldr, r_dev,
                                     rmax));
        }
    }
    GS_CK(cudaGetLastError());
    int r = 0;
    GS_CK(cudaMemcpyAsync(&r, r_dev, sizeof(int), cudaMemcpyDeviceToHost, s));
    GS_CK(cudaStreamSynchronize(s));
    // a bounded wait of the panel kernel that ran out leaves the factorisation unusable
    if (take_device_error_build() & GS_DEV_ERR_TIMEOUT) return GS_ERR_TIMEOUT;
    f.r = r;
    f.ldr = ldr;
    return GS_OK;
}

gs_status build_basis(const float* C, int M, int D, int ldc, double tau, bool normalize,
                      cudaStream_t s, gs_basis* h) {
    Factor f;
    gs_status st = factor_rows(C, M, D, ldc, tau, normalize, s, f);
    if (st != GS_OK) return st;
    return finalize_basis(f.Qw, f.R64, f.ldr, f.cn, M, D, f.r, s, h);
}

// Sec. 3.1, D < M: the entries are split into subsets, each gets its own orthonormal basis,
// and the reconstructions are concatenated.  Group g (rows [off[g], off[g+1]) of C) is
// factored alone; the handle holds the stacked Q = [Q_0; Q_1; ...] (r = sum of r_g rows) and
// the block-diagonal R whose row i of group g holds R_g's row in columns [s_g, s_g + r_g),
// s_g = r_0 + ... + r_(g-1).  C = R Q holds row by row, so every call on the handle works
// unchanged (Q's rows are orthonormal within a group, not across groups).
gs_status build_basis_grouped(const float* C, int M, int D, int ldc, const int* off, int G, double tau,
                              bool normalize, cudaStream_t s, gs_basis* h) {
    std::vector<std::unique_ptr<Factor>> fs;
    int rt = 0;
    for (int g = 0; g < G; ++g) {
        fs.emplace_back(new Factor());
        gs_status st = factor_rows(C + (size_t)off[g] * ldc, off[g + 1] - off[g], D, ldc, tau, normalize, s,
                                   *fs.back());
        if (st != GS_OK) return st;
        rt += fs.back()->r;
    }
    const int ldr = std::max(rt, 1);
    DevBuf bQ, bR, bcn;
    GS_CK(cudaMalloc(&bQ.p, sizeof(double) * (size_t)ldr * D));
    GS_CK(cudaMalloc(&bR.p, sizeof(double) * (size_t)M * ldr));
    GS_CK(cudaMalloc(&bcn.p, sizeof(double) * (size_t)M));
    double* Q = (double*)bQ.p;
    double* R = (double*)bR.p;
    double* cn = (double*)bcn.p;
    GS_CK(cudaMemsetAsync(R, 0, sizeof(double) * (size_t)M * ldr, s));
    h->grp_rows.assign(off, off + G + 1);
    h->grp_coeffs.assign(1, 0);
    int sg = 0;
    for (int g = 0; g < G; ++g) {
        const Factor& f = *fs[g];
        const int mg = off[g + 1] - off[g];
        if (f.r > 0) {
            GS_CK(cudaMemcpyAsync(Q + (size_t)sg * D, f.Qw, sizeof(double) * (size_t)f.r * D,
                                  cudaMemcpyDeviceToDevice, s));
            GS_CK(cudaMemcpy2DAsync(R + (size_t)off[g] * ldr + sg, sizeof(double) * ldr, f.R64,
                                    sizeof(double) * f.ldr, sizeof(double) * f.r, mg, cudaMemcpyDeviceToDevice,
                                    s));
        }
        GS_CK(cudaMemcpyAsync(cn + off[g], f.cn, sizeof(double) * mg, cudaMemcpyDeviceToDevice, s));
        sg += f.r;
        h->grp_coeffs.push_back(sg);
    }
    return finalize_basis(Q, R, ldr, cn, M, D, rt, s, h);
}

// Everything a handle holds besides the fp64 factorisation: fp32 Q, R and norms for the
// caller, R's echelon lengths, the fp16 operand copies (dithered) and the chunk scratch.
gs_status finalize_basis(const double* Qw, const double* R64, int ldr, const double* cn, int M, int D, int r,
                         cudaStream_t s, gs_basis* h) {
    h->M = M;
    h->D = D;
    h->r = r;
    h->ldr = std::max(r, 1);

    // user-visible fp32 results
    GS_CK(cudaMalloc(&h->Q, sizeof(float) * (size_t)std::max(r, 1) * D));
    GS_CK(cudaMalloc(&h->R, sizeof(float) * (size_t)M * h->ldr));
    GS_CK(cudaMalloc(&h->cnorm, sizeof(float) * (size_t)M));
    GS_CK(cudaMalloc(&h->rlen, sizeof(int) * (size_t)M));
    GS_CK(cudaMalloc(&h->rlen_chunk, sizeof(int) * (size_t)((M + 31) / 32)));
    GS_CK(cudaMemsetAsync(h->R, 0, sizeof(float) * (size_t)M * h->ldr, s));
    if (r > 0) {
        k_cast_rows<<<grid1((long long)r * D, 256), 256, 0, s>>>(Qw, D, h->Q, D, r, D);
        k_cast_rows<<<grid1((long long)M * r, 256), 256, 0, s>>>(R64, ldr, h->R, h->ldr, M, r);
    }
    k_cast_rows<<<grid1(M, 256), 256, 0, s>>>(cn, 1, h->cnorm, 1, M, 1);
    k_rlen<<<grid1(M, 128), 128, 0, s>>>(R64, ldr, M, r, h->rlen);
    k_rlen_chunk<<<grid1((M + 31) / 32, 128), 128, 0, s>>>(h->rlen, M, h->rlen_chunk);

    // tensor-core operand copies (fp16, dithered)
    if (r > 0) {
        h->ldq16 = (D + 7) / 8 * 8;
        h->ldr16 = (r + 7) / 8 * 8;
        GS_CK(cudaMalloc(&h->Q16, sizeof(__half) * (size_t)r * h->ldq16));
        GS_CK(cudaMalloc(&h->Q16t, sizeof(__half) * (size_t)D * h->ldr16));
        if (h->ldr16 != r)
            k_zero_half<<<grid1((long long)D * h->ldr16, 256), 256, 0, s>>>(h->Q16t, (long long)D * h->ldr16);
        k_q16<<<grid1((long long)r * h->ldq16, 256), 256, 0, s>>>(Qw, r, D, h->Q16, h->ldq16, h->Q16t,
                                                                  h->ldr16);
    }

    // scratch for the chunked multi-kernel paths: rows x (r + M + 1) floats
    const long long per_row = (long long)r + M + 1;
    long long rows = std::max(256LL, (64LL << 20) / per_row);
    rows = std::min(rows, 65536LL);
    h->chunk_rows = rows;
    h->scratch_floats = rows * per_row;
    GS_CK(cudaMalloc(&h->scratch, sizeof(float) * (size_t)h->scratch_floats));
    GS_CK(cudaGetLastError());
    GS_CK(cudaStreamSynchronize(s));
    return GS_OK;
}

cudaError_t launch_f16t_dither(const float* src, int rows, int cols, long long lds, void* dst, long long ldt,
                               cudaStream_t s) {
    if (rows <= 0 || cols <= 0) return cudaSuccess;
    const dim3 grid((unsigned)((cols + 31) / 32), (unsigned)((rows + 31) / 32));
    if (grid.y > 65535u) return cudaErrorInvalidConfiguration;
    k_f16t_dither<<<grid, 256, 0, s>>>(src, rows, cols, lds, static_cast<__half*>(dst), ldt);
    return cudaGetLastError();
}

}  // namespace gs

namespace gs {

gs_status import_basis(const float* Q, int ldq, const float* R, int ldr_in, const float* cnorm, int M, int D,
                       int r, cudaStream_t s, gs_basis* h) {
    const int ldr = std::max(r, 1);
    DevBuf bQw, bR64, bcn;
    GS_CK(cudaMalloc(&bQw.p, sizeof(double) * (size_t)std::max(r, 1) * D));
    GS_CK(cudaMalloc(&bR64.p, sizeof(double) * (size_t)M * ldr));
    GS_CK(cudaMalloc(&bcn.p, sizeof(double) * (size_t)M));
    double* Qw = (double*)bQw.p;
    double* R64 = (double*)bR64.p;
    double* cn = (double*)bcn.p;
    GS_CK(cudaMemsetAsync(R64, 0, sizeof(double) * (size_t)M * ldr, s));
    if (r > 0) {
        k_widen_rows<<<grid1((long long)r * D, 256), 256, 0, s>>>(Q, ldq, Qw, D, r, D);
        k_widen_rows<<<grid1((long long)M * r, 256), 256, 0, s>>>(R, ldr_in, R64, ldr, M, r);
    }
    if (cnorm)
        k_widen_rows<<<grid1(M, 256), 256, 0, s>>>(cnorm, 1, cn, 1, M, 1);
    else
        k_row_norms64<<<grid1(M, 128), 128, 0, s>>>(R64, ldr, M, r, cn);
    GS_CK(cudaGetLastError());
    return finalize_basis(Qw, R64, ldr, cn, M, D, r, s, h);
}

}  // namespace gs
