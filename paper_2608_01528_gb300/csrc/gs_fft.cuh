// gs_fft.cuh -- complex arithmetic and small in-register DFTs shared by the spectral
// binding kernels (gs_bind_spec.cu: transforms through shared memory; gs_rbind_tc.cu:
// transforms in tensor memory behind the reconstruction GEMM).
#pragma once

#include <cuda_runtime.h>

namespace gs {
namespace fft {

// complex add / subtract as one paired fp32 instruction (sm_100+), lane by lane round to
// nearest: the same results as two scalar operations
static __device__ __forceinline__ unsigned long long f2_pack(float2 a) {
    unsigned long long r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a.x), "f"(a.y));
    return r;
}
static __device__ __forceinline__ float2 f2_unpack(unsigned long long v) {
    float2 a;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a.x), "=f"(a.y) : "l"(v));
    return a;
}
static __device__ __forceinline__ float2 c_add(float2 a, float2 b) {
    unsigned long long r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(f2_pack(a)), "l"(f2_pack(b)));
    return f2_unpack(r);
}
static __device__ __forceinline__ float2 c_sub(float2 a, float2 b) {
    unsigned long long r;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(f2_pack(a)), "l"(f2_pack(b)));
    return f2_unpack(r);
}
static __device__ __forceinline__ float2 c_mul(float2 a, float2 b) {
    return make_float2(fmaf(a.x, b.x, -a.y * b.y), fmaf(a.x, b.y, a.y * b.x));
}
static __device__ __forceinline__ float2 c_mulconj(float2 a, float2 b) {  // a * conj(b)
    return make_float2(fmaf(a.x, b.x, a.y * b.y), fmaf(a.y, b.x, -a.x * b.y));
}
static __device__ __forceinline__ float2 c_conj(float2 a) { return make_float2(a.x, -a.y); }
static __device__ __forceinline__ float2 c_mul_negi(float2 a) { return make_float2(a.y, -a.x); }  // -i a

// z e^{-2 pi i t / 16}, t in [0, 8): the constant twiddles of butterflies up to radix 16
static __device__ __forceinline__ float2 rot16(float2 z, int t) {
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

static constexpr int bitrev(int i, int R) {
    int r = 0;
    for (int b = 1; b < R; b <<= 1) r = (r << 1) | ((i & b) ? 1 : 0);
    return r;
}

// forward DFT of R points in registers, natural order in and out: radix-2
// decimation in frequency, then the bit-reversal permutation (register renaming)
template <int R>
static __device__ __forceinline__ void dft(float2 (&v)[R]) {
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

// z e^{+2 pi i t / 16}, t in [0, 8): the constant twiddles of the inverse butterflies
static __device__ __forceinline__ float2 rot16i(float2 z, int t) {
    return c_conj(rot16(c_conj(z), t));
}

// inverse DFT of R points (unnormalised: sum_k v_k e^{+2 pi i n k / R}), natural order in
// and out, the mirror of dft<R> with conjugate rotations
template <int R>
static __device__ __forceinline__ void dft_inv(float2 (&v)[R]) {
#pragma unroll
    for (int half = R / 2; half >= 1; half >>= 1) {
#pragma unroll
        for (int g = 0; g < R; g += 2 * half) {
#pragma unroll
            for (int i = 0; i < half; ++i) {
                const float2 a = v[g + i], b = v[g + i + half];
                v[g + i] = c_add(a, b);
                v[g + i + half] = rot16i(c_sub(a, b), i * (16 / (2 * half)));
            }
        }
    }
    float2 t[R];
#pragma unroll
    for (int i = 0; i < R; ++i) t[bitrev(i, R)] = v[i];
#pragma unroll
    for (int i = 0; i < R; ++i) v[i] = t[i];
}

}  // namespace fft
}  // namespace gs
