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
//  k_bind_spec<H, UNB>   a CTA takes groups of U = 2048/H blocks (x and y: 4096
//                        complex points), persistent over the grid

#include <stdint.h>

#include <algorithm>

#include "gs_internal.h"

namespace gs {
namespace {

constexpr int kSpecThreads = 256;
constexpr int kSpecPoints = 4096;                           // complex points of a forward group
constexpr int kSpecBuf = kSpecPoints + kSpecPoints / 16;    // padded buffer length (float2)

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
                       : 1;
}
constexpr int spec_passes(int H) { return H <= 256 ? 2 : 3; }
// twiddle-table floats of pass p (p >= 1): (R - 1) rows of Ns entries
constexpr int spec_ns(int H, int p) { return p == 0 ? 1 : spec_ns(H, p - 1) * spec_radix(H, p - 1); }
constexpr int spec_tw_len(int H, int p) { return (spec_radix(H, p) - 1) * spec_ns(H, p); }
constexpr size_t spec_smem_bytes(int H) {
    return sizeof(float2) * ((size_t)2 * kSpecBuf + H + spec_tw_len(H, 1) + (spec_passes(H) > 2 ? spec_tw_len(H, 2) : 0));
}

__device__ __forceinline__ float2 c_add(float2 a, float2 b) { return make_float2(a.x + b.x, a.y + b.y); }
__device__ __forceinline__ float2 c_sub(float2 a, float2 b) { return make_float2(a.x - b.x, a.y - b.y); }
__device__ __forceinline__ float2 c_mul(float2 a, float2 b) {
    return make_float2(fmaf(a.x, b.x, -a.y * b.y), fmaf(a.x, b.y, a.y * b.x));
}
__device__ __forceinline__ float2 c_mulconj(float2 a, float2 b) {  // a * conj(b)
    return make_float2(fmaf(a.x, b.x, a.y * b.y), fmaf(a.y, b.x, -a.x * b.y));
}
__device__ __forceinline__ float2 c_conj(float2 a) { return make_float2(a.x, -a.y); }
__device__ __forceinline__ float2 c_mul_i(float2 a) { return make_float2(-a.y, a.x); }     // i a
__device__ __forceinline__ float2 c_mul_negi(float2 a) { return make_float2(a.y, -a.x); }  // -i a

// z e^{-2 pi i t / 16}, t in [0, 8): the constant twiddles of butterflies up to radix 16
__device__ __forceinline__ float2 rot16(float2 z, int t) {
    constexpr float c1 = 0.92387953251128674f;  // cos(pi/8)
    constexpr float s1 = 0.38268343236508977f;  // sin(pi/8)
    constexpr float h = 0.70710678118654752f;   // sqrt(1/2)
    switch (t) {
        case 0: return z;
        case 4: return c_mul_negi(z);
        case 2: return make_float2((z.x + z.y) * h, (z.y - z.x) * h);
        case 6: return make_float2((z.y - z.x) * h, -(z.x + z.y) * h);
        default: {
            // (c, s) = (cos, sin) of 2 pi t / 16
            const float c = t == 1 ? c1 : t == 3 ? s1 : t == 5 ? -s1 : -c1;
            const float s = t == 1 ? s1 : t == 3 ? c1 : t == 5 ? c1 : s1;
            return make_float2(fmaf(z.x, c, z.y * s), fmaf(z.y, c, -z.x * s));
        }
    }
}

constexpr int bitrev(int i, int R) {
    int r = 0;
    for (int b = 1; b < R; b <<= 1) r = (r << 1) | ((i & b) ? 1 : 0);
    return r;
}

// forward DFT of R points in registers, natural order in and out: radix-2
// decimation in frequency, then the bit-reversal permutation (register renaming)
template <int R>
__device__ __forceinline__ void dft(float2 (&v)[R]) {
#pragma unroll
    for (int half = R / 2; half >= 1; half >>= 1) {
#pragma unroll
        for (int g = 0; g < R; g += 2 * half) {
#pragma unroll
            for (int i = 0; i < half; ++i) {
                const float2 a = v[g + i], b = v[g + i + half];
                v[g + i] = c_add(a, b);
                v[g + i + half] = rot16(c_sub(a, b), i * (16 / (2 * half)));
            }
        }
    }
    float2 t[R];
#pragma unroll
    for (int i = 0; i < R; ++i) t[bitrev(i, R)] = v[i];
#pragma unroll
    for (int i = 0; i < R; ++i) v[i] = t[i];
}

// Sequence s of a group (s < U: x of block u0 + s; s >= U: y of block u0 + s - U) in global memory.
struct SpecRows {
    const float* X;
    const float* Y;
    float* Z;
    long long units;  // N * nb
    long long ldy;
    int nb, L, ldx, ldz;
};

__device__ __forceinline__ long long unit_row(long long unit, int nb, int& b) {
    const long long n = unit / nb;
    b = (int)(unit - n * nb);
    return n;
}

// Stockham pass of radix R over sub-transforms of size NS, shared -> shared, nseq sequences
template <int H, int R, int NS>
__device__ __forceinline__ void spec_pass_ss(const float2* __restrict__ src, float2* __restrict__ dst, int nseq,
                                             const float2* __restrict__ tw) {
    constexpr int NB = H / R;
    for (int bf = threadIdx.x; bf < nseq * NB; bf += kSpecThreads) {
        const int s = bf / NB, j = bf % NB, k = j % NS;
        float2 v[R];
#pragma unroll
        for (int r = 0; r < R; ++r) v[r] = src[pad16(s * H + j + r * NB)];
#pragma unroll
        for (int r = 1; r < R; ++r) v[r] = c_mul(v[r], tw[(r - 1) * NS + k]);
        dft<R>(v);
        const int base = s * H + (j - k) * R + k;
#pragma unroll
        for (int r = 0; r < R; ++r) dst[pad16(base + r * NS)] = v[r];
    }
}

// first forward pass (Ns = 1, no twiddles): the 2U blocks of a group from global memory
template <int H, int R>
__device__ __forceinline__ void spec_pass_load(const SpecRows& p, long long u0, int U, float2* __restrict__ dst) {
    constexpr int NB = H / R;
    for (int bf = threadIdx.x; bf < 2 * U * NB; bf += kSpecThreads) {
        const int s = bf / NB, j = bf % NB;
        const int i = s < U ? s : s - U;
        if (u0 + i >= p.units) continue;
        int b;
        const long long n = unit_row(u0 + i, p.nb, b);
        const float2* g = reinterpret_cast<const float2*>(
            s < U ? p.X + (size_t)n * p.ldx + (size_t)b * p.L : p.Y + (size_t)n * p.ldy + (size_t)b * p.L);
        float2 v[R];
#pragma unroll
        for (int r = 0; r < R; ++r) v[r] = __ldcs(g + j + r * NB);
        dft<R>(v);
#pragma unroll
        for (int r = 0; r < R; ++r) dst[pad16(s * H + j * R + r)] = v[r];
    }
}

// last inverse pass: z_2n + i z_2n+1 = conj(F_n) / (8H) straight to the output rows
template <int H, int R, int NS>
__device__ __forceinline__ void spec_pass_store(const SpecRows& p, long long u0, int U,
                                                const float2* __restrict__ src, const float2* __restrict__ tw) {
    constexpr int NB = H / R;
    static_assert(NB == NS, "the last pass completes the transform");
    constexpr float scale = 1.0f / (8.0f * H);
    for (int bf = threadIdx.x; bf < U * NB; bf += kSpecThreads) {
        const int s = bf / NB, j = bf % NB;
        if (u0 + s >= p.units) continue;
        float2 v[R];
#pragma unroll
        for (int r = 0; r < R; ++r) v[r] = src[pad16(s * H + j + r * NB)];
#pragma unroll
        for (int r = 1; r < R; ++r) v[r] = c_mul(v[r], tw[(r - 1) * NS + j]);
        dft<R>(v);
        int b;
        const long long n = unit_row(u0 + s, p.nb, b);
        float2* g = reinterpret_cast<float2*>(p.Z + (size_t)n * p.ldz + (size_t)b * p.L);
#pragma unroll
        for (int r = 0; r < R; ++r) __stcs(g + j + r * NS, make_float2(v[r].x * scale, -v[r].y * scale));
    }
}

// 2 X_k of a real block from W = DFT_H(packed pairs): (A + B) - i t_k (A - B),
// A = W_k, B = conj(W_(H-k) mod H), t_k = e^{-2 pi i k / L}
__device__ __forceinline__ float2 real_split(float2 a, float2 b_conj, float2 t) {
    return c_add(c_add(a, b_conj), c_mul_negi(c_mul(t, c_sub(a, b_conj))));
}

// point-wise pass: spectra of x (sequences 0..U-1) and y (U..2U-1) in src; writes, per block,
// conj of the packed spectrum W''_k = (P_k + conj P_H-k) + i conj(t_k) (P_k - conj P_H-k) of the
// product P = X Y (X conj Y to unbind), ready for the inverse transform by the forward passes
template <int H, bool UNB>
__device__ __forceinline__ void spec_pointwise(const float2* __restrict__ src, float2* __restrict__ dst, int U,
                                               const float2* __restrict__ tws) {
    constexpr int HH = H / 2;
    for (int it = threadIdx.x; it < U * HH; it += kSpecThreads) {
        const int i = it / HH, k = it % HH;
        // pad16(s H + k) = pad16(s H) + pad16(k): H is a multiple of 16
        const float2* wx = src + pad16(i * H);
        const float2* wy = src + pad16((U + i) * H);
        float2* out = dst + pad16(i * H);
        if (k == 0) {
            // k = 0 and k = H (real: sums of the even and odd samples), k = H/2 (its own partner)
            const float2 ax = wx[pad16(0)], ay = wy[pad16(0)];
            const float p0 = 4.f * (ax.x + ax.y) * (ay.x + ay.y);
            const float ph = 4.f * (ax.x - ax.y) * (ay.x - ay.y);
            out[pad16(0)] = make_float2(p0 + ph, ph - p0);
            const float2 bx = wx[pad16(HH)], by = wy[pad16(HH)];
            // 2 X_H/2 = 2 conj(W_H/2); W''_H/2 = 2 conj(P_H/2), stored conjugated: 2 P_H/2
            const float2 xq = make_float2(2.f * bx.x, -2.f * bx.y), yq = make_float2(2.f * by.x, -2.f * by.y);
            const float2 pq = UNB ? c_mulconj(xq, yq) : c_mul(xq, yq);
            out[pad16(HH)] = make_float2(2.f * pq.x, 2.f * pq.y);
            continue;
        }
        const int km = H - k;
        const float2 t = tws[k];                              // e^{-2 pi i k / L}
        const float2 tm = make_float2(-t.x, t.y);             // e^{-2 pi i (H - k) / L} = -conj(t)
        const float2 axk = wx[pad16(k)], axm = wx[pad16(km)];
        const float2 ayk = wy[pad16(k)], aym = wy[pad16(km)];
        const float2 xk = real_split(axk, c_conj(axm), t), xm = real_split(axm, c_conj(axk), tm);
        const float2 yk = real_split(ayk, c_conj(aym), t), ym = real_split(aym, c_conj(ayk), tm);
        const float2 pk = UNB ? c_mulconj(xk, yk) : c_mul(xk, yk);
        const float2 pm = UNB ? c_mulconj(xm, ym) : c_mul(xm, ym);
        // W''_k with conj(t_k); W''_H-k with conj(t_H-k) = -t_k
        const float2 dk = c_sub(pk, c_conj(pm)), dm = c_sub(pm, c_conj(pk));
        const float2 wk = c_add(c_add(pk, c_conj(pm)), c_mul_i(c_mul(c_conj(t), dk)));
        const float2 wm = c_add(c_add(pm, c_conj(pk)), c_mul_i(c_mul(make_float2(-t.x, -t.y), dm)));
        out[pad16(k)] = c_conj(wk);
        out[pad16(km)] = c_conj(wm);
    }
}

template <int H, bool UNB>
__global__ void __launch_bounds__(kSpecThreads) k_bind_spec(SpecRows p, long long groups) {
    constexpr int U = kSpecPoints / 2 / H;
    constexpr int P = spec_passes(H);
    constexpr int R0 = spec_radix(H, 0), R1 = spec_radix(H, 1), R2 = spec_radix(H, 2);
    constexpr int NS1 = spec_ns(H, 1), NS2 = spec_ns(H, 2);
    extern __shared__ float2 spec_sm[];
    float2* bufA = spec_sm;
    float2* bufB = bufA + kSpecBuf;
    float2* tws = bufB + kSpecBuf;  // e^{-2 pi i k / L}, k < H
    float2* tw1 = tws + H;          // pass 1: e^{-2 pi i r k / (Ns R)}, row r - 1, column k
    float2* tw2 = tw1 + spec_tw_len(H, 1);
    for (int k = threadIdx.x; k < H; k += kSpecThreads) {
        float s, c;
        sincospif((float)k / (float)H, &s, &c);
        tws[k] = make_float2(c, -s);
    }
    for (int e = threadIdx.x; e < spec_tw_len(H, 1); e += kSpecThreads) {
        const int r = e / NS1 + 1, k = e % NS1;
        float s, c;
        sincospif(2.0f * (float)(r * k) / (float)(NS1 * R1), &s, &c);
        tw1[e] = make_float2(c, -s);
    }
    if constexpr (P > 2) {
        for (int e = threadIdx.x; e < spec_tw_len(H, 2); e += kSpecThreads) {
            const int r = e / NS2 + 1, k = e % NS2;
            float s, c;
            sincospif(2.0f * (float)(r * k) / (float)(NS2 * R2), &s, &c);
            tw2[e] = make_float2(c, -s);
        }
    }
    __syncthreads();
    for (long long g = blockIdx.x; g < groups; g += gridDim.x) {
        const long long u0 = g * U;
        // forward transforms of the group's x and y blocks
        spec_pass_load<H, R0>(p, u0, U, bufA);
        __syncthreads();
        float2* fin;
        float2* other;
        if constexpr (P == 2) {
            spec_pass_ss<H, R1, NS1>(bufA, bufB, 2 * U, tw1);
            fin = bufB;
            other = bufA;
        } else {
            spec_pass_ss<H, R1, NS1>(bufA, bufB, 2 * U, tw1);
            __syncthreads();
            spec_pass_ss<H, R2, NS2>(bufB, bufA, 2 * U, tw2);
            fin = bufA;
            other = bufB;
        }
        __syncthreads();
        spec_pointwise<H, UNB>(fin, other, U, tws);
        __syncthreads();
        // inverse transform of the products (forward passes on conjugated spectra)
        {
            constexpr int NB = H / R0;
            for (int bf = threadIdx.x; bf < U * NB; bf += kSpecThreads) {
                const int s = bf / NB, j = bf % NB;
                float2 v[R0];
#pragma unroll
                for (int r = 0; r < R0; ++r) v[r] = other[pad16(s * H + j + r * NB)];
                dft<R0>(v);
#pragma unroll
                for (int r = 0; r < R0; ++r) fin[pad16(s * H + j * R0 + r)] = v[r];
            }
        }
        __syncthreads();
        if constexpr (P == 2) {
            spec_pass_store<H, R1, NS1>(p, u0, U, fin, tw1);
        } else {
            spec_pass_ss<H, R1, NS1>(fin, other, U, tw1);
            __syncthreads();
            spec_pass_store<H, R2, NS2>(p, u0, U, other, tw2);
        }
        // the next group's first pass writes bufA: every thread has passed the barrier after
        // the last read of bufA above, and the pass that follows it reads only the other buffer
    }
}

template <int H>
cudaError_t launch_h(const SpecRows& p, bool unbind, cudaStream_t s) {
    constexpr int U = kSpecPoints / 2 / H;
    constexpr size_t smem = spec_smem_bytes(H);
    static bool attr_set[2] = {false, false};
    auto kern = unbind ? k_bind_spec<H, true> : k_bind_spec<H, false>;
    if (!attr_set[unbind]) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr_set[unbind] = true;
    }
    int dev = 0, sms = 0, occ = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, kSpecThreads, smem);
    if (e != cudaSuccess) return e;
    const long long groups = (p.units + U - 1) / U;
    const long long grid = std::min<long long>(groups, (long long)std::max(sms, 1) * std::max(occ, 1));
    kern<<<(unsigned)grid, kSpecThreads, smem, s>>>(p, groups);
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
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace gs
