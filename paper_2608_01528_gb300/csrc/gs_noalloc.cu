// gs_noalloc.cu -- project + similarity for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at all: code running while a CUDA graph is
// being captured with a capture mode that forbids allocation, plugins that must
// live inside a host framework's fixed device-memory budget, and integrations
// whose own caching allocator owns every byte of the device.  For them,
// gs_project_similarity_static runs the chunked fp32 project + similarity path
// (Y = X Q^T, S = Y R^T, argmax / maxval per row) with its scratch in a
// file-scope device array instead of memory allocated by the library.
//
// The array is a fixed 16 MiB per device (kStaticScratchFloats floats) and is
// held by every GPU that loads this library until the process exits.  In host
// code its name is only a host-side stand-in, so the entry point looks up the
// device address with cudaGetSymbolAddress once per device (the first call on
// a device, with that device current) and passes that address to the kernels.
// Every call on a device shares the one array: calls that overlap on the GPU
// (different streams, or several host threads) race on it.  Nothing in the
// array needs to start at zero: each chunk writes every scratch element it
// later reads.

#include <mutex>

#include "gs_internal.h"

namespace {

constexpr long long kStaticScratchFloats = 4LL << 20;  // 16 MiB of fp32
constexpr long long kMaxRowsPerGemm = 65535LL * 64;    // grid.y limit of the fp32 GEMM
constexpr int kMaxDevices = 64;

static __device__ __align__(256) float g_static_scratch[kStaticScratchFloats];

float* g_scratch_dev[kMaxDevices];  // device address of g_static_scratch, per device
std::mutex g_scratch_mu;

// Device address of the static scratch on `dev` (looked up on first use).
gs_status static_scratch(int dev, float** out) {
    if (dev < 0 || dev >= kMaxDevices) return GS_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_dev[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) return GS_ERR_CUDA;
        g_scratch_dev[dev] = static_cast<float*>(p);
    }
    *out = g_scratch_dev[dev];
    return GS_OK;
}

gs_status from_cuda(cudaError_t e) { return e == cudaSuccess ? GS_OK : GS_ERR_CUDA; }

}  // namespace

extern "C" GS_API gs_status gs_project_similarity_static(const float* Q, int r, int D, const float* R, int M,
                                                         const float* cnorm, const float* X, long long N,
                                                         int ldx, int mode, float scale, int* argmax,
                                                         float* maxval, void* stream) {
    if (mode < GS_SCORE_RAW || mode > GS_SCORE_SOFTMAX || !(scale == scale)) return GS_ERR_INVALID_ARG;
    if (r < 0 || D < 1 || M < 1 || N < 0 || ldx < D) return GS_ERR_SHAPE;
    const long long per_row = (long long)r + M + 1;  // Y row, norm, S row
    if (per_row > kStaticScratchFloats) return GS_ERR_SHAPE;
    if (N == 0) return GS_OK;
    if (!X || (!argmax && !maxval) || (r > 0 && (!Q || !R)) || (mode == GS_SCORE_COSINE && !cnorm))
        return GS_ERR_INVALID_ARG;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GS_ERR_CUDA;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (major != 10 || minor != 3) return GS_ERR_UNSUPPORTED;
    float* scr = nullptr;
    gs_status st = static_scratch(dev, &scr);
    if (st != GS_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    long long chunk = kStaticScratchFloats / per_row;
    if (chunk > kMaxRowsPerGemm) chunk = kMaxRowsPerGemm;
    for (long long c0 = 0; c0 < N; c0 += chunk) {
        const long long nc = N - c0 < chunk ? N - c0 : chunk;
        float* Ybuf = scr;                    // nc x r
        float* xn = scr + nc * r;             // nc
        float* Sbuf = scr + nc * (r + 1);     // nc x M
        if (mode == GS_SCORE_COSINE) {
            st = from_cuda(gs::launch_rownorm(X + c0 * ldx, nc, ldx, D, xn, s));
            if (st != GS_OK) return st;
        }
        if (r > 0) {
            gs::GemmArgs a{};
            a.A = X + c0 * ldx; a.a_type = gs::MAT_F32; a.lda = ldx;
            a.B = Q; a.b_type = gs::MAT_F32; a.ldb = D; a.b_trans = true;
            a.C = Ybuf; a.c_type = gs::MAT_F32; a.ldc = r;
            a.m = nc; a.n = r; a.k = D; a.batch = 1; a.alpha = 1.f;
            st = from_cuda(gs::launch_gemm_simt(a, s));
            if (st != GS_OK) return st;
        }
        gs::GemmArgs b{};
        b.A = Ybuf; b.a_type = gs::MAT_F32; b.lda = r > 0 ? r : 1;
        b.B = R ? R : Ybuf; b.b_type = gs::MAT_F32; b.ldb = r > 0 ? r : 1; b.b_trans = true;
        b.C = Sbuf; b.c_type = gs::MAT_F32; b.ldc = M;
        b.m = nc; b.n = M; b.k = r; b.batch = 1; b.alpha = scale;
        if (mode == GS_SCORE_COSINE) {
            b.rownorm = xn;
            b.colnorm = cnorm;
        }
        st = from_cuda(gs::launch_gemm_simt(b, s));
        if (st != GS_OK) return st;
        st = from_cuda(gs::launch_row_finish(Sbuf, nc, M, M, mode == GS_SCORE_SOFTMAX,
                                             argmax ? argmax + c0 : nullptr, maxval ? maxval + c0 : nullptr, s));
        if (st != GS_OK) return st;
    }
    return GS_OK;
}
