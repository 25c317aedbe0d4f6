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
// device address with cudaGetSymbolAddress once per device context (the first
// call on a device, with that device current) and passes that address to the
// kernels.  The address is cached together with the context's unique id: after
// cudaDeviceReset the device gets a new primary context (the module, and the
// array with it, is loaded again), the ids differ, and the next call looks the
// address up again instead of using one the old context owned.
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

float* g_scratch_dev[kMaxDevices];               // device address of g_static_scratch, per device
unsigned long long g_scratch_ctx[kMaxDevices];   // id of the context that address belongs to
std::mutex g_scratch_mu;

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// Unique id of the current context (0 when it cannot be read: the address is then looked up
// on every call, which is correct, only slower).
unsigned long long current_ctx_id() {
    static CtxGetCurrentFn get_current = nullptr;
    static CtxGetIdFn get_id = nullptr;
    static bool looked_up = false;
    if (!looked_up) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = (CtxGetCurrentFn)p;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = (CtxGetIdFn)p;
        looked_up = true;
    }
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
        return 0;
    return id;
}

// Device address of the static scratch on `dev` (looked up on first use in each context).
gs_status static_scratch(int dev, float** out) {
    if (dev < 0 || dev >= kMaxDevices) return GS_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    const unsigned long long ctx = current_ctx_id();
    if (!g_scratch_dev[dev] || ctx == 0 || ctx != g_scratch_ctx[dev]) {
        void* p = nullptr;
        g_scratch_dev[dev] = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) return GS_ERR_CUDA;
        g_scratch_dev[dev] = static_cast<float*>(p);
        g_scratch_ctx[dev] = ctx;
    }
    *out = g_scratch_dev[dev];
    return GS_OK;
}

// A stream created on another device than the current one: its kernels would get this
// device's scratch address.  The special handles (legacy and per-thread default streams)
// always belong to the current device.
bool stream_on_other_device(cudaStream_t s, int dev) {
    if (s == nullptr || s == cudaStreamLegacy || s == cudaStreamPerThread) return false;
    int sdev = -1;
    return cudaStreamGetDevice(s, &sdev) != cudaSuccess || sdev != dev;
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
    cudaStream_t s = (cudaStream_t)stream;
    if (stream_on_other_device(s, dev)) return GS_ERR_INVALID_ARG;
    float* scr = nullptr;
    gs_status st = static_scratch(dev, &scr);
    if (st != GS_OK) return st;
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
