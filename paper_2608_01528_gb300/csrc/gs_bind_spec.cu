// gs_bind_spec.cu -- binding / unbinding through block spectra.
//
// Block circular convolution (binding) and correlation (unbinding) of Sec. 2.2 /
// Sec. 3.3 computed with the convolution theorem instead of the direct O(L) sum
// per output: for a block of L = 2H real components,
//   bind:   z = IDFT_L( DFT_L(x) . DFT_L(y) )
//   unbind: z = IDFT_L( DFT_L(x) . conj(DFT_L(y)) )      (real y)
// Each real transform of length L is one complex transform of length H on the
// packed pairs w_n = v_2n + i v_2n+1 plus a split step (the standard real-FFT
// packing), so a block costs three complex H-point transforms and one
// point-wise pass: ~5 L log2 L flops against the direct sum's 2 L^2.
//
// The H-point transforms are Stockham autosort passes (Govindaraju et al.,
// "High Performance Discrete Fourier Transforms on Graphics Processors", SC'08):
// pass p takes radix R_p over sub-transforms of size Ns = R_0 ... R_p-1, reading
// with stride H/R and writing to (j - j mod Ns) R + j mod Ns + r Ns, which leaves
// the result in natural order with no bit reversal.  Each radix-R butterfly is a
// radix-2 decimation-in-frequency DFT in registers.  The first forward pass reads
// the blocks straight from global memory (the packed pairs are the row's
// consecutive floats) and the last inverse pass writes the output rows, so the
// intermediate spectra live only in shared memory.
//
//  k_bind_spec<H, UNB>   teams of T threads (a warp for L <= 512, L/16 threads above)
//                        each take groups of U blocks (x and y: 16 T complex points in
//                        the team's own pair of shared buffers), persistent over the
//                        grid; a team synchronises only itself, so teams in different
//                        phases (loads in flight, transforms) overlap on an SM

#include <stdint.h>

#include <algorithm>

#include "gs_internal.h"
#include "gs_fft.cuh"

namespace gs {
namespace {

// threads of a team and complex points of its group (16 per thread: a radix-16 pass is one
// butterfly per thread), threads of a CTA (256, or one team of 512 for H = 4096) and CTAs an
// SM should hold (the register budget: 85 a thread at 3 CTAs of 256)
constexpr int spec_team(int H) { return H <= 256 ? 32 : H / 8; }
constexpr int spec_points(int H) { return 16 * spec_team(H); }
constexpr int spec_cta(int H) { return spec_team(H) > 256 ? spec_team(H) : 256; }
constexpr int spec_min_ctas(int H) { return spec_cta(H) > 256 ? 1 : 3; }
constexpr int spec_buf(int H) { return spec_points(H) + spec_points(H) / 16; }  // padded length (float2)

// one float2 of padding after every 16: the stride-R writes of a first pass and the
// strided reads of the others then fall in distinct banks
__device__ __forceinline__ int pad16(int i) { return i + (i >> 4); }

// radix of pass p for an H-point transform, and the number of passes
constexpr int spec_radix(int H, int p) {
    return H == 32     ? (p == 0 ? 8 : p == 1 ? 4 : 1)
           : H == 64   ? (p < 2 ? 8 : 1)
           : H == 128  ? (p == 0 ? 16 : p == 1 ? 8 : 1)
           : H == 256  ? (p < 2 ? 16 : 1)
           : H == 512  ? 8
           : H == 1024 ? (p == 0 ? 16 : 8)
           : H == 2048 ? (p < 2 ? 16 : 8)
           : H == 4096 ? 16
                       : 1;
}
constexpr int spec_passes(int H) { return H <= 256 ? 2 : 3; }
// twiddle-table entries of pass p (p >= 1): (R - 1) rows of Ns entries
constexpr int spec_ns(int H, int p) { return p == 0 ? 1 : spec_ns(H, p - 1) * spec_radix(H, p - 1); }
constexpr int spec_tw_len(int H, int p) { return (spec_radix(H, p) - 1) * spec_ns(H, p); }
// two padded buffers per team, then the tables
constexpr size_t spec_smem_bytes(int H) {
    return sizeof(float2) * ((size_t)(spec_cta(H) / spec_team(H)) * 2 * spec_buf(H) + H + spec_tw_len(H, 1) +
                             (spec_passes(H) > 2 ? spec_tw_len(H, 2) : 0));
}

template <int T>
__device__ __forceinline__ void team_sync(int team) {
    if constexpr (T == 32) {
        __syncwarp();
    } else {
        asm volatile("bar.sync %0, %1;\n" ::"r"(team + 1), "r"(T) : "memory");
    }
}

// complex helpers and the radix-R DFTs: gs_fft.cuh
using namespace fft;

// The rows of one launch: X, Y (ldy = 0: Y's one row partners every row), Z; N rows of nb blocks.
struct SpecRows {
    const float* X;
    const float* Y;
    float* Z;
    long long units;  // N * nb
    long long ldy;
    int nb, L, ldx, ldz;
};

// row n and block b of unit (n0, b0) + i, i < U: a few steps of b past the row's nb blocks
__device__ __forceinline__ long long unit_row(long long n0, int b0, int i, int nb, int& b) {
    long long n = n0;
    b = b0 + i;
    while (b >= nb) {
        b -= nb;
        ++n;
    }
    return n;
}

// Stockham pass of radix R over sub-transforms of size NS, src -> dst (a team's two buffers),
// nseq sequences; the team synchronises at the end
template <int H, int T, int R, int NS, bool TWR = false>
__device__ __forceinline__ void spec_pass(const float2* __restrict__ src, float2* __restrict__ dst, int nseq,
                                          const float2* __restrict__ tw, int t, int team,
                                          const float2* twr = nullptr) {
    constexpr int NB = H / R;
    for (int bf = t; bf < nseq * NB; bf += T) {
        const int s = bf / NB, j = bf % NB, k = j % NS;
        float2 v[R];
#pragma unroll
        for (int r = 0; r < R; ++r) v[r] = src[pad16(s * H + j + r * NB)];
        if constexpr (NS > 1) {
#pragma unroll
            for (int r = 1; r < R; ++r) v[r] = c_mul(v[r], TWR ? twr[r - 1] : tw[(r - 1) * NS + k]);
        }
        dft<R>(v);
        const int base = s * H + (j - k) * R + k;
#pragma unroll
        for (int r = 0; r < R; ++r) dst[pad16(base + r * NS)] = v[r];
    }
    team_sync<T>(team);
}

// first forward pass (Ns = 1, no twiddles) straight from the rows into dst: sequence s < U is
// the x block of unit u0 + s, s >= U the y block of unit u0 + s - U (BC: all 2U sequences are x
// blocks, units u0 .. u0 + 2U - 1)
template <int H, int T, int R, bool BC>
__device__ __forceinline__ void spec_pass_load(const SpecRows& p, long long u0, long long n0, int b0,
                                               float2* __restrict__ dst, int t, int team) {
    constexpr int U = spec_points(H) / 2 / H, NB = H / R;
    for (int bf = t; bf < 2 * U * NB; bf += T) {
        const int s = bf / NB, j = bf % NB;
        const bool isx = BC || s < U;
        const int i = isx ? s : s - U;
        if (u0 + i >= p.units) continue;
        int b;
        const long long n = unit_row(n0, b0, i, p.nb, b);
        const float* row = isx ? p.X + (size_t)n * p.ldx : p.Y + (size_t)n * p.ldy;
        const float2* g = reinterpret_cast<const float2*>(row + (size_t)b * p.L);
        float2 v[R];
#pragma unroll
        for (int r = 0; r < R; ++r) v[r] = __ldcs(g + j + r * NB);
        dft<R>(v);
#pragma unroll
        for (int r = 0; r < R; ++r) dst[pad16(s * H + j * R + r)] = v[r];
    }
    team_sync<T>(team);
}

// last inverse pass: z_2n + i z_2n+1 = conj(F_n) / (8H) straight to the output rows
template <int H, int T, int R, int NS, int UX, bool TWR = false>
__device__ __forceinline__ void spec_pass_store(const SpecRows& p, long long u0, long long n0, int b0,
                                                const float2* __restrict__ buf, const float2* __restrict__ tw,
                                                int t, const float2* twr = nullptr) {
    constexpr int NB = H / R;
    static_assert(NB == NS, "the last pass completes the transform");
    constexpr float scale = 1.0f / (8.0f * H);
    for (int bf = t; bf < UX * NB; bf += T) {
        const int s = bf / NB, j = bf % NB;
        if (u0 + s >= p.units) continue;
        float2 v[R];
#pragma unroll
        for (int r = 0; r < R; ++r) v[r] = buf[pad16(s * H + j + r * NB)];
#pragma unroll
        for (int r = 1; r < R; ++r) v[r] = c_mul(v[r], TWR ? twr[r - 1] : tw[(r - 1) * NS + j]);
        dft<R>(v);
        int b;
        const long long n = unit_row(n0, b0, s, p.nb, b);
        float2* g = reinterpret_cast<float2*>(p.Z + (size_t)n * p.ldz + (size_t)b * p.L);
#pragma unroll
        for (int r = 0; r < R; ++r) __stcs(g + j + r * NS, make_float2(v[r].x * scale, -v[r].y * scale));
    }
}

// 2 X_k and 2 X_H-k of a real block from W = DFT_H(packed pairs), t = e^{-2 pi i k / L}:
// with A = W_k, B = conj(W_H-k), S = A + B and G = t (A - B),
//   2 X_k = S - i G,   2 X_H-k = conj(S) - i conj(G)
// (the second is the first's formula at H - k, where the roles of A and B swap and
// t_H-k = -conj(t))
__device__ __forceinline__ void real_split(float2 wk, float2 wm, float2 t, float2& xk, float2& xm) {
    const float2 a = wk, b = c_conj(wm);
    const float2 S = c_add(a, b), G = c_mul(t, c_sub(a, b));
    xk = make_float2(S.x + G.y, S.y - G.x);
    xm = make_float2(S.x - G.y, -S.y - G.x);
}

// point-wise pass, in place: from the spectra of x (sequences 0..U-1) and y (U..2U-1), writes
// over x, per block, conj of the packed spectrum W''_k = (P_k + conj P_H-k) + i conj(t_k)
// (P_k - conj P_H-k) of the product P = X Y (X conj Y to unbind), ready for the inverse
// transform by forward passes.  With E = P_k + conj P_H-k and G = conj(t_k) (P_k - conj P_H-k):
// W''_k = E + i G and W''_H-k = conj(E) + i conj(G).  A thread owns the pair (k, H - k) (and
// k = 0 with H/2), so it alone reads and writes those positions.  BC: all 2U sequences are x
// spectra and y's spectrum of block b is ytab + pad16(b H), shared by every row.
template <int H, int T, bool UNB, bool BC>
__device__ __forceinline__ void spec_pointwise(float2* __restrict__ buf, const float2* __restrict__ tws,
                                               const float2* __restrict__ ytab, int b0, int nb, int t, int team) {
    constexpr int U = spec_points(H) / 2 / H, HH = H / 2, UX = BC ? 2 * U : U;
    for (int it = t; it < UX * HH; it += T) {
        const int i = it / HH, k = it % HH;
        // pad16(s H + k) = pad16(s H) + pad16(k): H is a multiple of 16
        float2* wx = buf + pad16(i * H);
        const float2* wy;
        if constexpr (BC) {
            int b;
            unit_row(0, b0, i, nb, b);
            wy = ytab + pad16(b * H);
        } else {
            wy = buf + pad16((U + i) * H);
        }
        if (k == 0) {
            // k = 0 and k = H (real: sums of the even and odd samples), k = H/2 (its own partner)
            const float2 ax = wx[pad16(0)], ay = wy[pad16(0)];
            const float p0 = 4.f * (ax.x + ax.y) * (ay.x + ay.y);
            const float ph = 4.f * (ax.x - ax.y) * (ay.x - ay.y);
            const float2 bx = wx[pad16(HH)], by = wy[pad16(HH)];
            // 2 X_H/2 = 2 conj(W_H/2); W''_H/2 = 2 conj(P_H/2), stored conjugated: 2 P_H/2
            const float2 xq = make_float2(2.f * bx.x, -2.f * bx.y), yq = make_float2(2.f * by.x, -2.f * by.y);
            const float2 pq = UNB ? c_mulconj(xq, yq) : c_mul(xq, yq);
            wx[pad16(0)] = make_float2(p0 + ph, ph - p0);
            wx[pad16(HH)] = make_float2(2.f * pq.x, 2.f * pq.y);
            continue;
        }
        const int km = H - k;
        const float2 t1 = tws[k];  // e^{-2 pi i k / L}
        float2 xk, xm, yk, ym;
        real_split(wx[pad16(k)], wx[pad16(km)], t1, xk, xm);
        real_split(wy[pad16(k)], wy[pad16(km)], t1, yk, ym);
        const float2 pk = UNB ? c_mulconj(xk, yk) : c_mul(xk, yk);
        const float2 pm = UNB ? c_mulconj(xm, ym) : c_mul(xm, ym);
        const float2 pmc = c_conj(pm);
        const float2 E = c_add(pk, pmc), G = c_mul(c_conj(t1), c_sub(pk, pmc));
        // stored conjugated: conj(E + iG) and conj(conj(E) + i conj(G))
        wx[pad16(k)] = make_float2(E.x - G.y, -E.y - G.x);
        wx[pad16(km)] = make_float2(E.x + G.y, E.y - G.x);
    }
    team_sync<T>(team);
}

template <int H, bool UNB, bool BC>
__global__ void __launch_bounds__(spec_cta(H), spec_min_ctas(H)) k_bind_spec(SpecRows p, long long groups) {
    constexpr int T = spec_team(H), U = spec_points(H) / 2 / H, NT = spec_cta(H), TEAMS = NT / T;
    constexpr int UX = BC ? 2 * U : U;  // blocks of x a group transforms
    constexpr int P = spec_passes(H);
    constexpr int R0 = spec_radix(H, 0), R1 = spec_radix(H, 1), R2 = spec_radix(H, 2);
    constexpr int NS1 = spec_ns(H, 1), NS2 = spec_ns(H, 2);
    extern __shared__ float2 spec_sm[];
    const int team = threadIdx.x / T, t = threadIdx.x % T;
    float2* bufA = spec_sm + (size_t)team * 2 * spec_buf(H);
    float2* bufB = bufA + spec_buf(H);
    float2* tws = spec_sm + (size_t)TEAMS * 2 * spec_buf(H);  // e^{-2 pi i k / L}, k < H
    float2* tw1 = tws + H;  // pass 1: e^{-2 pi i r k / (Ns R)}, row r - 1, column k
    float2* tw2 = tw1 + spec_tw_len(H, 1);
    float2* ytab = tw2 + (P > 2 ? spec_tw_len(H, 2) : 0);  // BC: y's spectrum of each block
    for (int k = threadIdx.x; k < H; k += NT) {
        float s, c;
        sincospif((float)k / (float)H, &s, &c);
        tws[k] = make_float2(c, -s);
    }
    for (int e = threadIdx.x; e < spec_tw_len(H, 1); e += NT) {
        const int r = e / NS1 + 1, k = e % NS1;
        float s, c;
        sincospif(2.0f * (float)(r * k) / (float)(NS1 * R1), &s, &c);
        tw1[e] = make_float2(c, -s);
    }
    if constexpr (P > 2) {
        for (int e = threadIdx.x; e < spec_tw_len(H, 2); e += NT) {
            const int r = e / NS2 + 1, k = e % NS2;
            float s, c;
            sincospif(2.0f * (float)(r * k) / (float)(NS2 * R2), &s, &c);
            tw2[e] = make_float2(c, -s);
        }
    }
    __syncthreads();
    // two-pass warp teams: a thread's butterflies all sit at the same k = t mod NS1 in the second
    // pass (and the last inverse pass), so it keeps those R1 - 1 twiddles in registers
    constexpr bool TWR = P == 2 && T % NS1 == 0 && R1 <= 8;
    float2 twr[R1 - 1];
    if constexpr (TWR) {
#pragma unroll
        for (int r = 1; r < R1; ++r) twr[r - 1] = tw1[(r - 1) * NS1 + t % NS1];
    }
    if constexpr (BC) {
        // the one partner row's block spectra, once per CTA: team by team, block by block
        constexpr int NB0 = H / R0;
        for (int b = team; b < p.nb; b += TEAMS) {
            const float2* g = reinterpret_cast<const float2*>(p.Y + (size_t)b * p.L);
            for (int j = t; j < NB0; j += T) {
                float2 v[R0];
#pragma unroll
                for (int r = 0; r < R0; ++r) v[r] = __ldg(g + j + r * NB0);
                dft<R0>(v);
#pragma unroll
                for (int r = 0; r < R0; ++r) bufA[pad16(j * R0 + r)] = v[r];
            }
            team_sync<T>(team);
            float2* yb = ytab + pad16(b * H);
            if constexpr (P == 2) {
                spec_pass<H, T, R1, NS1, TWR>(bufA, yb, 1, tw1, t, team, twr);
            } else {
                spec_pass<H, T, R1, NS1>(bufA, bufB, 1, tw1, t, team);
                spec_pass<H, T, R2, NS2>(bufB, yb, 1, tw2, t, team);
            }
        }
        __syncthreads();
    }
    const long long stride = (long long)gridDim.x * TEAMS;
    const long long g0 = (long long)blockIdx.x * TEAMS + team;
    // (row, block) of the group's first unit, stepped along with the group index
    long long n0 = g0 * UX / p.nb;
    int b0 = (int)(g0 * UX - n0 * p.nb);
    const long long dn = stride * UX / p.nb;
    const int db = (int)(stride * UX - dn * p.nb);
    for (long long g = g0; g < groups; g += stride) {
        const long long u0 = g * UX;
        // forward transforms of the group's x (and y) blocks
        spec_pass_load<H, T, R0, BC>(p, u0, n0, b0, bufA, t, team);
        spec_pass<H, T, R1, NS1, TWR>(bufA, bufB, 2 * U, tw1, t, team, twr);
        if constexpr (P == 2) {
            spec_pointwise<H, T, UNB, BC>(bufB, tws, ytab, b0, p.nb, t, team);
            // inverse transforms of the products (forward passes on conjugated spectra)
            spec_pass<H, T, R0, 1>(bufB, bufA, UX, nullptr, t, team);
            spec_pass_store<H, T, R1, NS1, UX, TWR>(p, u0, n0, b0, bufA, tw1, t, twr);
        } else {
            spec_pass<H, T, R2, NS2>(bufB, bufA, 2 * U, tw2, t, team);
            spec_pointwise<H, T, UNB, BC>(bufA, tws, ytab, b0, p.nb, t, team);
            spec_pass<H, T, R0, 1>(bufA, bufB, UX, nullptr, t, team);
            spec_pass<H, T, R1, NS1>(bufB, bufA, UX, tw1, t, team);
            spec_pass_store<H, T, R2, NS2, UX>(p, u0, n0, b0, bufA, tw2, t);
        }
        team_sync<T>(team);  // the last pass has read bufA before the next group's first pass writes it
        n0 += dn;
        b0 += db;
        if (b0 >= p.nb) {
            b0 -= p.nb;
            ++n0;
        }
    }
}

constexpr size_t kSpecSmemCap = 227 * 1024;

template <int H>
cudaError_t launch_h(const SpecRows& p, bool unbind, cudaStream_t s) {
    constexpr int U = spec_points(H) / 2 / H, NT = spec_cta(H), TEAMS = NT / spec_team(H);
    // one partner row: its block spectra are computed once per CTA and kept in shared memory
    // (nb padded blocks after the tables) when they fit
    const size_t ytab = sizeof(float2) * (size_t)p.nb * (H + H / 16);
    const bool bc = p.ldy == 0 && spec_smem_bytes(H) + ytab <= kSpecSmemCap;
    const size_t smem = spec_smem_bytes(H) + (bc ? ytab : 0);
    // per device, operator and partner layout: the shared-memory opt-in (to the cap), done once;
    // the resident CTAs per SM for this launch's shared memory
    static bool opted[64][2][2];
    auto kern = bc ? (unbind ? k_bind_spec<H, true, true> : k_bind_spec<H, false, true>)
                   : (unbind ? k_bind_spec<H, true, false> : k_bind_spec<H, false, false>);
    int dev = 0, sms = 0, occ = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!opted[dev][unbind][bc]) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSpecSmemCap);
        if (e != cudaSuccess) return e;
        opted[dev][unbind][bc] = true;
    }
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, NT, smem);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const long long per_group = bc ? 2 * U : U;
    const long long groups = (p.units + per_group - 1) / per_group;
    const long long ctas = (groups + TEAMS - 1) / TEAMS;
    const long long grid = std::min<long long>(ctas, (long long)std::max(sms, 1) * std::max(occ, 1));
    kern<<<(unsigned)grid, NT, smem, s>>>(p, groups);
    return cudaGetLastError();
}

}  // namespace

bool bind_spectral_supported(int L, const float* X, int ldx, const float* Y, long long ldy, const float* Z, int ldz) {
    if (L < kMinBindSpectralL || L > kMaxBindSpectralL || (L & (L - 1))) return false;
    // float2 accesses: every row start 8-byte aligned
    return (uintptr_t)X % 8 == 0 && (uintptr_t)Y % 8 == 0 && (uintptr_t)Z % 8 == 0 && ldx % 2 == 0 &&
           ldy % 2 == 0 && ldz % 2 == 0;
}

cudaError_t launch_bind_spectral(const float* X, long long N, int D, int ldx, const float* Y, long long ldy, int L,
                                 bool unbind, float* Z, int ldz, cudaStream_t s) {
    if (N <= 0) return cudaSuccess;
    SpecRows p;
    p.X = X;
    p.Y = Y;
    p.Z = Z;
    p.nb = D / L;
    p.units = N * p.nb;
    p.ldy = ldy;
    p.L = L;
    p.ldx = ldx;
    p.ldz = ldz;
    switch (L) {
        case 64: return launch_h<32>(p, unbind, s);
        case 128: return launch_h<64>(p, unbind, s);
        case 256: return launch_h<128>(p, unbind, s);
        case 512: return launch_h<256>(p, unbind, s);
        case 1024: return launch_h<512>(p, unbind, s);
        case 2048: return launch_h<1024>(p, unbind, s);
        case 4096: return launch_h<2048>(p, unbind, s);
        case 8192: return launch_h<4096>(p, unbind, s);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace gs
