// gs_api.cu -- the C ABI declared in include/gramspace.h: argument checks,
// device selection, path dispatch and status handling.  No arithmetic of the
// method lives here; every step runs in the kernels of gs_build.cu,
// gs_simt.cu and gs_tc.cu.

#include <math.h>
#include <stdint.h>

#include <algorithm>

#include "gs_internal.h"

namespace {

// Makes h's device current for the duration of a call and restores the caller's.
struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) { ok = false; return; }
        if (prev != dev && cudaSetDevice(dev) != cudaSuccess) ok = false;
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

gs_status from_cuda(cudaError_t e) {
    if (e == cudaSuccess) return GS_OK;
    if (e == cudaErrorMemoryAllocation) return GS_ERR_NOMEM;
    return GS_ERR_CUDA;
}

bool device_supported(int dev) {
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) return false;
    return major == 10 && minor == 3;
}

bool valid_path(unsigned flags) {
    return flags == GS_PATH_AUTO || flags == GS_PATH_SIMT || flags == GS_PATH_TENSOR;
}

void release_staging(gs_basis* h) {
    cudaFree(h->stage_x);
    cudaFree(h->stage_am);
    cudaFree(h->stage_mv);
    if (h->stage_copy) cudaStreamDestroy(h->stage_copy);
    cudaEvent_t* evs[5] = {&h->stage_start, &h->stage_in[0], &h->stage_in[1], &h->stage_done[0], &h->stage_done[1]};
    for (cudaEvent_t* ev : evs)
        if (*ev) cudaEventDestroy(*ev), *ev = nullptr;
    h->stage_x = nullptr;
    h->stage_am = nullptr;
    h->stage_mv = nullptr;
    h->stage_copy = nullptr;
    h->stage_rows = 0;
}

void free_basis(gs_basis* h) {
    if (!h) return;
    cudaFree(h->Q);
    cudaFree(h->R);
    cudaFree(h->cnorm);
    cudaFree(h->rlen);
    cudaFree(h->rlen_chunk);
    cudaFree(h->Q16);
    cudaFree(h->Q16t);
    cudaFree(h->scratch);
    release_staging(h);
    cudaFree(h->tc_Rh);
    cudaFree(h->tc_Rl);
    cudaFree(h->tc_Rth);
    cudaFree(h->tc_Rtl);
    cudaFree(h->tc_Qh);
    cudaFree(h->tc_Ql);
    delete h;
}

constexpr long long kMaxGemmRows = 65535LL * 64;  // grid.y limit of the SIMT GEMM

// Project + similarity on the tensor core for bases the fused kernel cannot hold
// in TMEM (r > 256 or M > 256): Y = X Q^T (fp16 operands, fp32 accumulation)
// into the handle's scratch, then S = Y R^T with Y and R split into bf16 hi / lo,
// then the row reductions.  Rows are processed in chunks that fit the scratch.
gs_status ps_two_gemm(const gs_basis* h, const float* X, long long N, int ldx, int mode, float scale, float* Y,
                      int ldy, float* S, int lds, int* argmax, float* maxval, cudaStream_t s) {
    const int r = h->r, M = h->M, D = h->D;
    const int r4 = (r + 3) / 4 * 4;  // padded ld of the Y scratch (16-byte rows for TMA)
    const long long per_row = (long long)r4 + M + 3;
    long long chunk = std::min(h->scratch_floats / per_row, kMaxGemmRows);
    if (chunk < 1) return GS_ERR_SHAPE;
    const bool need_s = S || argmax || maxval;
    const bool f16 = D >= gs::kMinF16Depth;  // one fp16 rounding of X (else the bf16 hi / lo split)
    for (long long c0 = 0; c0 < N; c0 += chunk) {
        const long long nc = std::min(chunk, N - c0);
        float* Ybuf = h->scratch;
        float* xn = Ybuf + nc * r4;
        float* xn2 = xn + nc;       // 2 x nc: the rows' ||x||^2 in two partial sums (fp16 GEMM1)
        float* Sscr = xn2 + 2 * nc;
        gs::GemmTcArgs g1{};
        g1.A = X + c0 * ldx; g1.lda = ldx; g1.m = nc; g1.K = D;
        g1.split = !f16;
        g1.B0 = g1.split ? h->tc_Qh : (const void*)h->Q16;
        g1.B1 = g1.split ? h->tc_Ql : nullptr;
        g1.ldb = h->ldq16; g1.n = r;
        g1.C = Ybuf; g1.ldc = r4; g1.c_bf16 = false; g1.alpha = 1.f;
        g1.xn2_out = f16 ? xn2 : nullptr;
        cudaError_t e = gs::launch_gemm_tc(g1, h->device, s);
        if (e != cudaSuccess) return from_cuda(e);
        if (f16) {
            // rows that one fp16 rounding cannot hold accurately (||x|| > 2^15, or ||x|| <
            // 2^-8 sqrt(D) where fp16's subnormals start to matter): their Y rows are computed
            // again in fp32; the 64-row blocks without such a row return at once
            gs::GemmArgs f{};
            f.A = X + c0 * ldx; f.a_type = gs::MAT_F32; f.lda = ldx;
            f.B = h->Q; f.b_type = gs::MAT_F32; f.ldb = D; f.b_trans = true;
            f.C = Ybuf; f.c_type = gs::MAT_F32; f.ldc = r4;
            f.m = nc; f.n = r; f.k = D; f.batch = 1; f.alpha = 1.f;
            f.gate_xn2 = xn2; f.gate_ld = nc; f.gate_lo = (float)D * 0x1p-16f; f.gate_hi = 0x1p30f;
            e = gs::launch_gemm_simt(f, s);
            if (e != cudaSuccess) return from_cuda(e);
        }
        if (Y) {
            e = cudaMemcpy2DAsync(Y + c0 * ldy, sizeof(float) * ldy, Ybuf, sizeof(float) * r4, sizeof(float) * r, nc,
                                  cudaMemcpyDeviceToDevice, s);
            if (e != cudaSuccess) return from_cuda(e);
        }
        if (!need_s) continue;
        if (mode == GS_SCORE_COSINE) {
            e = gs::launch_rownorm(X + c0 * ldx, nc, ldx, D, xn, s);
            if (e != cudaSuccess) return from_cuda(e);
        }
        float* Sbuf = S ? S + c0 * lds : Sscr;
        const long long ldsb = S ? lds : M;
        gs::GemmTcArgs g2{};
        g2.A = Ybuf; g2.lda = r4; g2.m = nc; g2.K = r; g2.split = true;
        g2.B0 = h->tc_Rh; g2.B1 = h->tc_Rl; g2.ldb = h->tc_npad; g2.n = M;
        g2.b_klo = h->kzero_host.data(); g2.b_khi = h->rlen_host.data();
        g2.C = Sbuf; g2.ldc = ldsb; g2.c_bf16 = false; g2.alpha = scale;
        if (mode == GS_SCORE_COSINE) { g2.rownorm = xn; g2.colnorm = h->cnorm; }
        e = gs::launch_gemm_tc(g2, h->device, s);
        if (e != cudaSuccess) return from_cuda(e);
        if (argmax || maxval || mode == GS_SCORE_SOFTMAX) {
            e = gs::launch_row_finish(Sbuf, nc, M, (int)ldsb, mode == GS_SCORE_SOFTMAX, argmax ? argmax + c0 : nullptr,
                                      maxval ? maxval + c0 : nullptr, s);
            if (e != cudaSuccess) return from_cuda(e);
        }
    }
    return GS_OK;
}

// K chunks for the fp32 GEMM of m x n outputs over depth k: enough 64 x 64 tiles x chunks to
// give every SM about two blocks, chunks of at least 512.
int gemm_ksplit(long long m, int n, int k, int dev) {
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const long long tiles = ((m + 63) / 64) * ((n + 63) / 64);
    const long long want = (2LL * std::max(sms, 1) + tiles - 1) / tiles;
    const long long most = std::max(1, k / 512);
    return (int)std::max(1LL, std::min(want, most));
}

// Whether a GEMM of m rows, n columns and depth k is worth the tensor-core kernel.
bool big_gemm(long long m, long long n, long long k) { return m >= 512 && 2.0 * m * n * k >= 2e9; }

}  // namespace

extern "C" {

int gs_version(void) { return 100; }

const char* gs_status_string(gs_status s) {
    switch (s) {
        case GS_OK: return "GS_OK";
        case GS_ERR_INVALID_ARG: return "GS_ERR_INVALID_ARG";
        case GS_ERR_ALIGNMENT: return "GS_ERR_ALIGNMENT";
        case GS_ERR_SHAPE: return "GS_ERR_SHAPE";
        case GS_ERR_NOMEM: return "GS_ERR_NOMEM";
        case GS_ERR_CUDA: return "GS_ERR_CUDA";
        case GS_ERR_TIMEOUT: return "GS_ERR_TIMEOUT";
        case GS_ERR_RANGE: return "GS_ERR_RANGE";
        case GS_ERR_UNSUPPORTED: return "GS_ERR_UNSUPPORTED";
    }
    return "GS_ERR_UNKNOWN";
}

gs_status gs_build_basis(const float* C, int M, int D, int ldc, float rank_tol, unsigned flags,
                         void* stream, gs_basis** out) {
    if (!out) return GS_ERR_INVALID_ARG;
    *out = nullptr;
    if (!C || M < 1 || D < 1 || ldc < D) return M < 1 || D < 1 || ldc < D ? GS_ERR_SHAPE : GS_ERR_INVALID_ARG;
    if (!(rank_tol > 0.f) || !isfinite(rank_tol)) return GS_ERR_INVALID_ARG;
    if (flags & ~GS_BUILD_NORMALIZE_ROWS) return GS_ERR_INVALID_ARG;
    if ((uintptr_t)C % sizeof(float)) return GS_ERR_ALIGNMENT;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GS_ERR_CUDA;
    if (!device_supported(dev)) return GS_ERR_UNSUPPORTED;
    gs_basis* h = new gs_basis();
    h->device = dev;
    gs_status st = gs::build_basis(C, M, D, ldc, (double)rank_tol, (flags & GS_BUILD_NORMALIZE_ROWS) != 0,
                                   (cudaStream_t)stream, h);
    if (st == GS_OK && gs::tc_available(dev)) st = gs::tc_prepare(h);
    if (st != GS_OK) {
        free_basis(h);
        return st;
    }
    *out = h;
    return GS_OK;
}

// increasing offsets 0 = off[0] < off[1] < ... < off[G] = M (M < 0: any last offset)
static bool valid_offsets(const int* off, int G, int M) {
    if (!off || G < 1 || G > gs::kMaxGroups || off[0] != 0) return false;
    for (int g = 0; g < G; ++g)
        if (off[g + 1] <= off[g]) return false;
    return M < 0 || off[G] == M;
}

gs_status gs_build_basis_grouped(const float* C, int M, int D, int ldc, const int* group_offsets, int G,
                                 float rank_tol, unsigned flags, void* stream, gs_basis** out) {
    if (!out) return GS_ERR_INVALID_ARG;
    *out = nullptr;
    if (!C || M < 1 || D < 1 || ldc < D) return M < 1 || D < 1 || ldc < D ? GS_ERR_SHAPE : GS_ERR_INVALID_ARG;
    if (!valid_offsets(group_offsets, G, M)) return GS_ERR_INVALID_ARG;
    if (!(rank_tol > 0.f) || !isfinite(rank_tol)) return GS_ERR_INVALID_ARG;
    if (flags & ~GS_BUILD_NORMALIZE_ROWS) return GS_ERR_INVALID_ARG;
    if ((uintptr_t)C % sizeof(float)) return GS_ERR_ALIGNMENT;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GS_ERR_CUDA;
    if (!device_supported(dev)) return GS_ERR_UNSUPPORTED;
    gs_basis* h = new gs_basis();
    h->device = dev;
    gs_status st = gs::build_basis_grouped(C, M, D, ldc, group_offsets, G, (double)rank_tol,
                                           (flags & GS_BUILD_NORMALIZE_ROWS) != 0, (cudaStream_t)stream, h);
    if (st == GS_OK && gs::tc_available(dev)) st = gs::tc_prepare(h);
    if (st != GS_OK) {
        free_basis(h);
        return st;
    }
    *out = h;
    return GS_OK;
}

gs_status gs_basis_groups(const gs_basis* h, int* G, int* row_offsets, int* coeff_offsets) {
    if (!h || !G) return GS_ERR_INVALID_ARG;
    const bool grouped = !h->grp_rows.empty();
    const int g = grouped ? (int)h->grp_rows.size() - 1 : 1;
    *G = g;
    for (int k = 0; k <= g; ++k) {
        if (row_offsets) row_offsets[k] = grouped ? h->grp_rows[k] : (k ? h->M : 0);
        if (coeff_offsets) coeff_offsets[k] = grouped ? h->grp_coeffs[k] : (k ? h->r : 0);
    }
    return GS_OK;
}

gs_status gs_group_argmax(const float* S, long long N, int lds, const int* group_offsets, int G, int* argmax,
                          float* maxval, void* stream) {
    if (N < 0) return GS_ERR_SHAPE;
    if (!valid_offsets(group_offsets, G, -1)) return GS_ERR_INVALID_ARG;
    if (lds < group_offsets[G]) return GS_ERR_SHAPE;
    if (N == 0) return GS_OK;
    if (!S || (!argmax && !maxval)) return GS_ERR_INVALID_ARG;
    return from_cuda(gs::launch_group_argmax(S, N, lds, group_offsets, G, argmax, maxval, (cudaStream_t)stream));
}

gs_status gs_basis_import(const float* Q, int r, int D, int ldq, const float* R, int M, int ldr,
                          const float* cnorm, void* stream, gs_basis** out) {
    if (!out) return GS_ERR_INVALID_ARG;
    *out = nullptr;
    if (M < 1 || D < 1 || r < 0 || r > M) return GS_ERR_SHAPE;  // r > D only for a grouped basis
    if (r > 0 && (ldq < D || ldr < r)) return GS_ERR_SHAPE;
    if (r > 0 && (!Q || !R)) return GS_ERR_INVALID_ARG;
    if (((uintptr_t)Q | (uintptr_t)R | (uintptr_t)cnorm) % sizeof(float)) return GS_ERR_ALIGNMENT;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GS_ERR_CUDA;
    if (!device_supported(dev)) return GS_ERR_UNSUPPORTED;
    gs_basis* h = new gs_basis();
    h->device = dev;
    gs_status st = gs::import_basis(Q, ldq, R, ldr, cnorm, M, D, r, (cudaStream_t)stream, h);
    if (st == GS_OK && gs::tc_available(dev)) st = gs::tc_prepare(h);
    if (st != GS_OK) {
        free_basis(h);
        return st;
    }
    *out = h;
    return GS_OK;
}

gs_status gs_basis_info(const gs_basis* h, int* M, int* D, int* r, const float** Q, const float** R,
                        const float** cnorm) {
    if (!h) return GS_ERR_INVALID_ARG;
    if (M) *M = h->M;
    if (D) *D = h->D;
    if (r) *r = h->r;
    if (Q) *Q = h->Q;
    if (R) *R = h->R;
    if (cnorm) *cnorm = h->cnorm;
    return GS_OK;
}

gs_status gs_basis_destroy(gs_basis* h) {
    if (!h) return GS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaDeviceSynchronize();
    free_basis(h);
    return GS_OK;
}

gs_status gs_project_similarity(const gs_basis* h, const float* X, long long N, int ldx, int mode,
                                float scale, unsigned flags, float* Y, int ldy, float* S, int lds,
                                int* argmax, float* maxval, void* stream) {
    if (!h || !valid_path(flags)) return GS_ERR_INVALID_ARG;
    if (mode < GS_SCORE_RAW || mode > GS_SCORE_SOFTMAX || !isfinite(scale)) return GS_ERR_INVALID_ARG;
    if (N < 0 || ldx < h->D) return GS_ERR_SHAPE;
    if ((Y && ldy < h->r) || (S && lds < h->M)) return GS_ERR_SHAPE;
    if (N == 0) return GS_OK;
    if (!Y && !S && !argmax && !maxval) return GS_ERR_INVALID_ARG;
    if (!X) return GS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    if (!g.ok) return GS_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    const int r = h->r, M = h->M, D = h->D;

    const bool aligned = (uintptr_t)X % 16 == 0 && ldx % 4 == 0;
    const bool fused = h->has_tmap_q16 && aligned && D >= gs::kMinF16Depth;  // r <= 256, M <= 256
    const bool two_gemm = h->has_split && aligned;      // any r >= 1
    const bool big = (double)N * D >= (double)(1 << 24);
    if (flags == GS_PATH_TENSOR || (flags == GS_PATH_AUTO && big && (fused || two_gemm))) {
        if (fused) return from_cuda(gs::launch_ps_tc(h, X, N, ldx, mode, scale, Y, ldy, S, lds, argmax, maxval, s));
        if (two_gemm) return ps_two_gemm(h, X, N, ldx, mode, scale, Y, ldy, S, lds, argmax, maxval, s);
        return !aligned ? GS_ERR_ALIGNMENT : GS_ERR_UNSUPPORTED;
    }
    if (r <= 32) {
        return from_cuda(gs::launch_ps_warp(X, N, ldx, D, h->Q, r, h->R, h->ldr, M, h->cnorm, mode, scale,
                                            Y, ldy, S, lds, argmax, maxval, s));
    }
    // generic chunked fp32 path: Y = X Q^T, S = Y R^T (+ cosine / scale), row finish
    const long long chunk = std::min(h->chunk_rows, kMaxGemmRows);
    for (long long c0 = 0; c0 < N; c0 += chunk) {
        const long long nc = std::min(chunk, N - c0);
        float* scr = h->scratch;
        float* Ybuf = Y ? Y + c0 * ldy : scr;
        const long long ldyb = Y ? ldy : r;
        scr += Y ? 0 : nc * r;
        float* xn = nullptr;
        if (mode == GS_SCORE_COSINE) {
            xn = scr;
            scr += nc;
            cudaError_t e = gs::launch_rownorm(X + c0 * ldx, nc, ldx, D, xn, s);
            if (e != cudaSuccess) return from_cuda(e);
        }
        gs::GemmArgs a{};
        a.A = X + c0 * ldx; a.a_type = gs::MAT_F32; a.lda = ldx;
        a.B = h->Q; a.b_type = gs::MAT_F32; a.ldb = D; a.b_trans = true;
        a.C = Ybuf; a.c_type = gs::MAT_F32; a.ldc = ldyb;
        a.m = nc; a.n = r; a.k = D; a.batch = 1; a.alpha = 1.f;
        // few output tiles (a small batch against a narrow basis): cut D into chunks so that
        // every SM gets work; the partial products go to the scratch after Y and the norms
        // (the score rows are written there only later) and are summed in a fixed order
        {
            const long long used = (long long)(scr - h->scratch);
            const long long room = (h->scratch_floats - used) / std::max(1LL, nc * r);
            a.ksplit = (int)std::min<long long>(gemm_ksplit(nc, r, D, h->device), room);
            a.kpart = a.ksplit > 1 ? scr : nullptr;
        }
        cudaError_t e = gs::launch_gemm_simt(a, s);
        if (e != cudaSuccess) return from_cuda(e);
        if (!S && !argmax && !maxval) continue;
        float* Sbuf = S ? S + c0 * lds : scr;
        const long long ldsb = S ? lds : M;
        gs::GemmArgs b{};
        b.A = Ybuf; b.a_type = gs::MAT_F32; b.lda = ldyb;
        b.B = h->R; b.b_type = gs::MAT_F32; b.ldb = h->ldr; b.b_trans = true; b.b_rowlen = h->rlen;
        b.C = Sbuf; b.c_type = gs::MAT_F32; b.ldc = ldsb;
        b.m = nc; b.n = M; b.k = r; b.batch = 1; b.alpha = scale;
        if (mode == GS_SCORE_COSINE) { b.rownorm = xn; b.colnorm = h->cnorm; }
        e = gs::launch_gemm_simt(b, s);
        if (e != cudaSuccess) return from_cuda(e);
        if (argmax || maxval || mode == GS_SCORE_SOFTMAX) {
            e = gs::launch_row_finish(Sbuf, nc, M, (int)ldsb, mode == GS_SCORE_SOFTMAX,
                                      argmax ? argmax + c0 : nullptr, maxval ? maxval + c0 : nullptr, s);
            if (e != cudaSuccess) return from_cuda(e);
        }
    }
    return GS_OK;
}

gs_status gs_basis_reserve_staging(gs_basis* h, long long rows) {
    if (!h) return GS_ERR_INVALID_ARG;
    if (rows < 0) return GS_ERR_SHAPE;
    DeviceGuard g(h->device);
    if (!g.ok) return GS_ERR_CUDA;
    release_staging(h);
    if (rows == 0) return GS_OK;
    const int ld = (h->D + 3) / 4 * 4;  // 16-byte rows, as the tensor-core path needs
    bool ok = cudaMalloc(&h->stage_x, sizeof(float) * 2 * (size_t)rows * ld) == cudaSuccess &&
              cudaMalloc(&h->stage_am, sizeof(int) * 2 * (size_t)rows) == cudaSuccess &&
              cudaMalloc(&h->stage_mv, sizeof(float) * 2 * (size_t)rows) == cudaSuccess;
    if (!ok) {
        release_staging(h);
        return GS_ERR_NOMEM;
    }
    ok = cudaStreamCreateWithFlags(&h->stage_copy, cudaStreamNonBlocking) == cudaSuccess &&
         cudaEventCreateWithFlags(&h->stage_start, cudaEventDisableTiming) == cudaSuccess;
    for (int b = 0; b < 2 && ok; ++b)
        ok = cudaEventCreateWithFlags(&h->stage_in[b], cudaEventDisableTiming) == cudaSuccess &&
             cudaEventCreateWithFlags(&h->stage_done[b], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
        release_staging(h);
        return GS_ERR_CUDA;
    }
    h->stage_rows = rows;
    h->stage_ld = ld;
    return GS_OK;
}

gs_status gs_project_similarity_host(const gs_basis* h, const float* X, long long N, int ldx, int mode,
                                     float scale, unsigned flags, int* argmax, float* maxval, void* stream) {
    if (!h || !valid_path(flags)) return GS_ERR_INVALID_ARG;
    if (mode < GS_SCORE_RAW || mode > GS_SCORE_SOFTMAX || !isfinite(scale)) return GS_ERR_INVALID_ARG;
    if (N < 0 || ldx < h->D) return GS_ERR_SHAPE;
    if (N == 0) return GS_OK;
    if (!X || (!argmax && !maxval)) return GS_ERR_INVALID_ARG;
    if (h->stage_rows < 1) return GS_ERR_INVALID_ARG;  // gs_basis_reserve_staging first
    DeviceGuard g(h->device);
    if (!g.ok) return GS_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    const long long R = h->stage_rows;
    // The copy stream starts after the work already on s (which may still read the slots).
    // Chunk i goes through slot i & 1: its copy in (copy stream) waits until chunk i - 2 has
    // finished with the slot; the kernel and the copies out (on s) wait for the copy in.
    // s waits for every copy-stream event, so work enqueued on s later follows all of it.
    cudaError_t e = cudaEventRecord(h->stage_start, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(h->stage_copy, h->stage_start, 0);
    if (e != cudaSuccess) return from_cuda(e);
    long long i = 0;
    for (long long c0 = 0; c0 < N; c0 += R, ++i) {
        const int b = (int)(i & 1);
        const long long nc = std::min(R, N - c0);
        float* sx = h->stage_x + (size_t)b * R * h->stage_ld;
        int* sam = h->stage_am + (size_t)b * R;
        float* smv = h->stage_mv + (size_t)b * R;
        if (i >= 2) e = cudaStreamWaitEvent(h->stage_copy, h->stage_done[b], 0);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(sx, sizeof(float) * h->stage_ld, X + c0 * ldx, sizeof(float) * ldx,
                                  sizeof(float) * h->D, nc, cudaMemcpyHostToDevice, h->stage_copy);
        if (e == cudaSuccess) e = cudaEventRecord(h->stage_in[b], h->stage_copy);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s, h->stage_in[b], 0);
        if (e != cudaSuccess) return from_cuda(e);
        gs_status st = gs_project_similarity(h, sx, nc, h->stage_ld, mode, scale, flags, nullptr, 0, nullptr, 0,
                                             argmax ? sam : nullptr, maxval ? smv : nullptr, stream);
        if (st != GS_OK) return st;
        if (argmax) e = cudaMemcpyAsync(argmax + c0, sam, sizeof(int) * nc, cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess && maxval)
            e = cudaMemcpyAsync(maxval + c0, smv, sizeof(float) * nc, cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaEventRecord(h->stage_done[b], s);
        if (e != cudaSuccess) return from_cuda(e);
    }
    return GS_OK;
}

gs_status gs_similarity_coeffs(const gs_basis* h, const float* Y, long long N, int ldy, int mode, float scale,
                               unsigned flags, float* S, int lds, int* argmax, float* maxval, void* stream) {
    if (!h || !valid_path(flags)) return GS_ERR_INVALID_ARG;
    if (mode < GS_SCORE_RAW || mode > GS_SCORE_SOFTMAX || !isfinite(scale)) return GS_ERR_INVALID_ARG;
    if (N < 0 || ldy < h->r || ldy < 1 || (S && lds < h->M)) return GS_ERR_SHAPE;
    if (N == 0) return GS_OK;
    if (!S && !argmax && !maxval) return GS_ERR_INVALID_ARG;
    if (!Y && h->r > 0) return GS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    if (!g.ok) return GS_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    const int r = h->r, M = h->M;
    const bool tc_ok = h->has_split && r >= 1 && (uintptr_t)Y % 16 == 0 && ldy % 4 == 0;
    const bool tensor = flags == GS_PATH_TENSOR || (flags == GS_PATH_AUTO && tc_ok && big_gemm(N, M, r));
    if (tensor && !tc_ok) return h->has_split && r >= 1 ? GS_ERR_ALIGNMENT : GS_ERR_UNSUPPORTED;
    if (!tensor && r >= 1 && r <= gs::kMaxCoeffsWarpR)  // small r: one fused launch, no scratch
        return from_cuda(gs::launch_coeffs_warp(Y, N, ldy, r, h->R, h->ldr, M, h->cnorm, mode, scale, S, lds, argmax,
                                                maxval, s));
    // scratch per row: ||y|| (cosine) and the score row when S is not an output
    const long long per_row = (mode == GS_SCORE_COSINE ? 1 : 0) + (S ? 0 : M);
    const long long chunk = std::min(per_row ? h->scratch_floats / per_row : N, kMaxGemmRows);
    if (chunk < 1) return GS_ERR_SHAPE;
    for (long long c0 = 0; c0 < N; c0 += chunk) {
        const long long nc = std::min(chunk, N - c0);
        const float* Yc = Y ? Y + c0 * ldy : nullptr;
        float* xn = nullptr;
        float* scr = h->scratch;
        if (mode == GS_SCORE_COSINE) {  // ||y|| = ||x|| for x in span(C) (Eq. 3)
            xn = scr;
            scr += nc;
            cudaError_t e = gs::launch_rownorm(Yc, nc, ldy, r, xn, s);
            if (e != cudaSuccess) return from_cuda(e);
        }
        float* Sbuf = S ? S + c0 * lds : scr;
        const long long ldsb = S ? lds : M;
        cudaError_t e;
        if (tensor) {
            // S = Yh Rh^T + Yl Rh^T + Yh Rl^T (bf16 hi / lo split, fp32 accumulation)
            gs::GemmTcArgs a{};
            a.A = Yc; a.lda = ldy; a.m = nc; a.K = r; a.split = true;
            a.B0 = h->tc_Rh; a.B1 = h->tc_Rl; a.ldb = h->tc_npad; a.n = M;
            a.b_klo = h->kzero_host.data(); a.b_khi = h->rlen_host.data();
            a.C = Sbuf; a.ldc = ldsb; a.c_bf16 = false; a.alpha = scale;
            if (xn) { a.rownorm = xn; a.colnorm = h->cnorm; }
            e = gs::launch_gemm_tc(a, h->device, s);
        } else {
            gs::GemmArgs b{};
            b.A = Yc ? (const void*)Yc : (const void*)h->scratch; b.a_type = gs::MAT_F32; b.lda = ldy;
            b.B = h->R; b.b_type = gs::MAT_F32; b.ldb = h->ldr; b.b_trans = true; b.b_rowlen = h->rlen;
            b.C = Sbuf; b.c_type = gs::MAT_F32; b.ldc = ldsb;
            b.m = nc; b.n = M; b.k = r; b.batch = 1; b.alpha = scale;
            if (xn) { b.rownorm = xn; b.colnorm = h->cnorm; }
            e = gs::launch_gemm_simt(b, s);
        }
        if (e != cudaSuccess) return from_cuda(e);
        if (argmax || maxval || mode == GS_SCORE_SOFTMAX) {
            e = gs::launch_row_finish(Sbuf, nc, M, (int)ldsb, mode == GS_SCORE_SOFTMAX, argmax ? argmax + c0 : nullptr,
                                      maxval ? maxval + c0 : nullptr, s);
            if (e != cudaSuccess) return from_cuda(e);
        }
    }
    return GS_OK;
}

gs_status gs_prob_vectorize(const gs_basis* h, const float* P, long long N, int ldp, void* V, int v_dtype,
                            int ldv, unsigned flags, void* stream) {
    if (!h || !valid_path(flags)) return GS_ERR_INVALID_ARG;
    if (v_dtype != GS_F32 && v_dtype != GS_BF16) return GS_ERR_INVALID_ARG;
    if (N < 0 || ldp < h->M || ldv < h->r) return GS_ERR_SHAPE;
    if (N == 0 || h->r == 0) return GS_OK;
    if (!P || !V) return GS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    if (!g.ok) return GS_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    const bool tc_ok = h->has_split && (uintptr_t)P % 16 == 0 && ldp % 4 == 0;
    if (flags == GS_PATH_TENSOR || (flags == GS_PATH_AUTO && tc_ok && big_gemm(N, h->r, h->M))) {
        if (!tc_ok) return h->has_split ? GS_ERR_ALIGNMENT : GS_ERR_UNSUPPORTED;
        // V = P R with P and R^T split into bf16 hi / lo (fp32-level accuracy)
        gs::GemmTcArgs a{};
        a.A = P; a.lda = ldp; a.m = N; a.K = h->M; a.split = true;
        a.B0 = h->tc_Rth; a.B1 = h->tc_Rtl; a.ldb = h->tc_mpad; a.n = h->r;
        a.b_klo = h->pivot_host.data(); a.b_khi = h->kM_host.data();
        a.C = V; a.ldc = ldv; a.c_bf16 = v_dtype == GS_BF16; a.alpha = 1.f;
        return from_cuda(gs::launch_gemm_tc(a, h->device, s));
    }
    for (long long c0 = 0; c0 < N; c0 += kMaxGemmRows) {
        const long long nc = std::min(kMaxGemmRows, N - c0);
        gs::GemmArgs a{};
        a.A = P + c0 * ldp; a.a_type = gs::MAT_F32; a.lda = ldp;
        a.B = h->R; a.b_type = gs::MAT_F32; a.ldb = h->ldr; a.b_trans = false;
        a.C = (char*)V + (size_t)c0 * ldv * (v_dtype == GS_F32 ? 4 : 2);
        a.c_type = v_dtype == GS_F32 ? gs::MAT_F32 : gs::MAT_BF16; a.ldc = ldv;
        a.m = nc; a.n = h->r; a.k = h->M; a.batch = 1; a.alpha = 1.f;
        cudaError_t e = gs::launch_gemm_simt(a, s);
        if (e != cudaSuccess) return from_cuda(e);
    }
    return GS_OK;
}

// Xhat = T B with the fp16 copy of T (tensor-core path) in `work` (work_floats floats).  B is the
// basis (Qb = h->Q, ldqb = D, Qtb = h->Q16t) or, for the one-partner reconstruct + bind, the basis
// rows bound with the partner (fp32 r x D rows, ld ldqb, and their transposed fp16 copy).
static gs_status reconstruct_rows(const gs_basis* h, const void* T, int t_dtype, long long N, int ldt, float* Xhat,
                                  int ldxh, unsigned flags, cudaStream_t s, float* work, long long work_floats,
                                  const float* Qb = nullptr, int ldqb = 0, const __half* Qtb = nullptr) {
    if (!Qb) {
        Qb = h->Q;
        ldqb = h->D;
        Qtb = h->Q16t;
    }
    // one fp16 rounding of T and of Q: each output sums r rounding errors weighted by entries of Q of
    // size ~1/sqrt(D), so the error's spread is ~2^-11 ||t|| / sqrt(D); from D = 1024 on its worst
    // case over a large output stays well inside 1e-4 ||t||, shorter rows take the fp32 path
    const bool deep = h->D >= gs::kMinF16Depth;
    const bool tc_ok = h->has_split && h->r >= 1 && t_dtype == GS_F32 && deep && (uintptr_t)T % 16 == 0 &&
                       ldt % 4 == 0;
    if (flags == GS_PATH_TENSOR || (flags == GS_PATH_AUTO && tc_ok && big_gemm(N, h->D, h->r))) {
        if (!tc_ok) return t_dtype != GS_F32 || !h->has_split || !deep ? GS_ERR_UNSUPPORTED : GS_ERR_ALIGNMENT;
        // Xhat = T Q: T rounded once to fp16 into the handle's scratch (every column tile of
        // Xhat re-reads it) after an exact power-of-two scale per row, the basis' dithered fp16
        // Q^T, fp32 accumulation, the row scales undone in the epilogue; rows in chunks that
        // fit the scratch (ld16 halves and one float per row)
        const int ld16 = (h->r + 7) / 8 * 8;  // 16-byte rows for TMA
        const long long chunk = std::min(work_floats / (ld16 / 2 + 1), kMaxGemmRows) / 128 * 128;
        if (chunk < 128) return GS_ERR_SHAPE;
        for (long long c0 = 0; c0 < N; c0 += chunk) {
            const long long nc = std::min(chunk, N - c0);
            const float* Tc = (const float*)T + (size_t)c0 * ldt;
            // T rows scaled by exact powers of two into fp16's range, the scales undone in fp32
            float* rowmul = work + (size_t)chunk * ld16 / 2;
            gs_status st = from_cuda(gs::launch_round_f16(Tc, ldt, nc, h->r, work, ld16, rowmul, s));
            if (st != GS_OK) return st;
            gs::GemmTcArgs a{};
            a.A = work; a.lda = ld16; a.m = nc; a.K = h->r; a.split = false; a.a_half = true;
            a.B0 = Qtb; a.ldb = h->ldr16; a.n = h->D;
            a.C = Xhat + (size_t)c0 * ldxh; a.ldc = ldxh; a.c_bf16 = false; a.alpha = 1.f;
            a.rowmul = rowmul;
            st = from_cuda(gs::launch_gemm_tc(a, h->device, s));
            if (st != GS_OK) return st;
        }
        return GS_OK;
    }
    for (long long c0 = 0; c0 < N; c0 += kMaxGemmRows) {
        const long long nc = std::min(kMaxGemmRows, N - c0);
        gs::GemmArgs a{};
        a.A = (const char*)T + (size_t)c0 * ldt * (t_dtype == GS_F32 ? 4 : 2);
        a.a_type = t_dtype == GS_F32 ? gs::MAT_F32 : gs::MAT_BF16; a.lda = ldt;
        a.B = Qb; a.b_type = gs::MAT_F32; a.ldb = ldqb; a.b_trans = false;
        a.C = Xhat + c0 * ldxh; a.c_type = gs::MAT_F32; a.ldc = ldxh;
        a.m = nc; a.n = h->D; a.k = h->r; a.batch = 1; a.alpha = 1.f;
        cudaError_t e = gs::launch_gemm_simt(a, s);
        if (e != cudaSuccess) return from_cuda(e);
    }
    return GS_OK;
}

gs_status gs_reconstruct(const gs_basis* h, const void* T, int t_dtype, long long N, int ldt, float* Xhat,
                         int ldxh, unsigned flags, void* stream) {
    if (!h || !valid_path(flags)) return GS_ERR_INVALID_ARG;
    if (t_dtype != GS_F32 && t_dtype != GS_BF16) return GS_ERR_INVALID_ARG;
    if (N < 0 || ldt < h->r || ldxh < h->D) return GS_ERR_SHAPE;
    if (N == 0) return GS_OK;
    if (!T || !Xhat) return GS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    if (!g.ok) return GS_ERR_CUDA;
    return reconstruct_rows(h, T, t_dtype, N, ldt, Xhat, ldxh, flags, (cudaStream_t)stream, h->scratch,
                            h->scratch_floats);
}

static gs_status check_bind_args(long long N, int D, int ldx, long long ldy, int L, int op, int ldz) {
    if (op < 0 || (op & ~(GS_UNBIND | GS_BIND_DIRECT | GS_BIND_SPECTRAL)) ||
        ((op & GS_BIND_DIRECT) && (op & GS_BIND_SPECTRAL)))
        return GS_ERR_INVALID_ARG;
    if (N < 0 || D < 1 || L < 1 || D % L || ldx < D || ldz < D || (ldy != 0 && ldy < D)) return GS_ERR_SHAPE;
    return GS_OK;
}

// why a forced spectral method cannot run: a block length it does not take, else alignment
static gs_status spectral_error(int L) {
    const bool l_ok = L >= gs::kMinBindSpectralL && L <= gs::kMaxBindSpectralL && !(L & (L - 1));
    return l_ok ? GS_ERR_ALIGNMENT : GS_ERR_UNSUPPORTED;
}

// one binding launch: the spectral kernel unless the direct sum is asked for or the spectral
// kernel cannot take the shape; a forced spectral method that cannot run is an error
static gs_status bind_rows(const float* X, long long N, int D, int ldx, const float* Y, long long ldy, int L, int op,
                           float* Z, int ldz, cudaStream_t s) {
    const bool unbind = (op & GS_UNBIND) != 0;
    const bool spec = gs::bind_spectral_supported(L, X, ldx, Y, ldy, Z, ldz);
    if ((op & GS_BIND_SPECTRAL) && !spec) return spectral_error(L);
    if (spec && !(op & GS_BIND_DIRECT))
        return from_cuda(gs::launch_bind_spectral(X, N, D, ldx, Y, ldy, L, unbind, Z, ldz, s));
    return from_cuda(gs::launch_bind(X, N, D, ldx, Y, ldy, L, unbind, Z, ldz, s));
}

gs_status gs_bind(const float* X, long long N, int D, int ldx, const float* Y, long long ldy, int L, int op, float* Z,
                  int ldz, void* stream) {
    gs_status st = check_bind_args(N, D, ldx, ldy, L, op, ldz);
    if (st != GS_OK) return st;
    if (N == 0) return GS_OK;
    if (!X || !Y || !Z) return GS_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GS_ERR_CUDA;
    if (!device_supported(dev)) return GS_ERR_UNSUPPORTED;
    return bind_rows(X, N, D, ldx, Y, ldy, L, op, Z, ldz, (cudaStream_t)stream);
}

// Reconstruct + bind with one partner row y for every row: binding is linear in its first
// operand, so op(t Q, y) = t op(Q, y) -- bind the r basis rows with y once, then reconstruct every
// row straight from those bound rows.  The reconstructed rows are never formed; the call costs one
// reconstruction GEMM (on an fp16 copy of op(Q, y), rounded like the basis' own copy) plus the
// binding of r rows.  Returns GS_ERR_SHAPE, with nothing enqueued, when the scratch cannot hold
// op(Q, y), its fp16 copy and one 128-row chunk of T.
static gs_status reconstruct_bind_one_partner(const gs_basis* h, const void* T, int t_dtype, long long N, int ldt,
                                              const float* Y, int L, int op, float* Z, int ldz, unsigned flags,
                                              cudaStream_t s) {
    const int r = h->r, D = h->D, Dp = (D + 3) / 4 * 4, ld16 = (r + 7) / 8 * 8;
    const long long qy_floats = (long long)r * Dp;
    const long long qt_floats = ((long long)D * ld16 / 2 + 3) / 4 * 4;  // 16-byte aligned after it
    const long long work_floats = h->scratch_floats - qy_floats - qt_floats;
    if (work_floats < 128LL * (ld16 / 2 + 1)) return GS_ERR_SHAPE;
    float* Qy = h->scratch;
    __half* Qyt = reinterpret_cast<__half*>(h->scratch + qy_floats);
    float* work = h->scratch + qy_floats + qt_floats;
    gs_status st = bind_rows(h->Q, r, D, D, Y, 0, L, op, Qy, Dp, s);
    if (st != GS_OK) return st;
    if (h->has_split) {  // the tensor-core reconstruction's operand (the fp32 path reads Qy)
        st = from_cuda(gs::launch_f16t_dither(Qy, r, D, Dp, Qyt, ld16, s));
        if (st != GS_OK) return st;
    }
    return reconstruct_rows(h, T, t_dtype, N, ldt, Z, ldz, flags, s, work, work_floats, Qy, Dp, Qyt);
}

// Reconstruct + bind with per-row partners in one kernel per chunk of rows (gs_rbind_tc.cu): the
// chunk's T rows rounded once to fp16 with exact power-of-two row scales (as in gs_reconstruct's
// tensor path), then each 128 x 256 tile of T Q is bound with its partner columns in tensor memory
// and only Z is written.  Returns GS_ERR_SHAPE, with nothing enqueued, when the scratch cannot
// hold one 128-row chunk of the fp16 rows.
static gs_status reconstruct_bind_fused(const gs_basis* h, const float* T, long long N, int ldt, const float* Y,
                                        long long ldy, int L, bool unbind, float* Z, int ldz, cudaStream_t s) {
    const int ld16 = (h->r + 7) / 8 * 8;  // 16-byte rows for TMA
    const long long chunk = std::min(h->scratch_floats / (ld16 / 2 + 1), kMaxGemmRows) / 128 * 128;
    if (chunk < 128) return GS_ERR_SHAPE;
    float* work = h->scratch;
    float* rowmul = work + (size_t)chunk * ld16 / 2;
    for (long long c0 = 0; c0 < N; c0 += chunk) {
        const long long nc = std::min(chunk, N - c0);
        gs_status st = from_cuda(gs::launch_round_f16(T + (size_t)c0 * ldt, ldt, nc, h->r, work, ld16, rowmul, s));
        if (st != GS_OK) return st;
        st = from_cuda(gs::launch_rbind_tc(h, work, ld16, nc, rowmul, Y + (size_t)c0 * ldy, ldy, L, unbind,
                                           Z + (size_t)c0 * ldz, ldz, h->device, s));
        if (st != GS_OK) return st;
    }
    return GS_OK;
}

gs_status gs_reconstruct_bind(const gs_basis* h, const void* T, int t_dtype, long long N, int ldt, const float* Y,
                              long long ldy, int L, int op, float* Z, int ldz, unsigned flags, void* stream) {
    if (!h || !valid_path(flags)) return GS_ERR_INVALID_ARG;
    if (t_dtype != GS_F32 && t_dtype != GS_BF16) return GS_ERR_INVALID_ARG;
    if (N < 0 || ldt < h->r) return GS_ERR_SHAPE;
    gs_status st = check_bind_args(N, h->D, h->D, ldy, L, op, ldz);
    if (st != GS_OK) return st;
    if (N == 0) return GS_OK;
    if (!T || !Y || !Z) return GS_ERR_INVALID_ARG;
    DeviceGuard g(h->device);
    if (!g.ok) return GS_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    // rows in chunks as large as the handle's scratch takes (the reconstructed rows and the fp16
    // copy of their T rows): fewer, fuller reconstruction launches.  Chunks sized for L2 (64 MiB)
    // measured slower: the GEMM's last wave per chunk cost more than the L2 hits saved.
    const int Dp = (h->D + 3) / 4 * 4, ld16 = (h->r + 7) / 8 * 8;
    if ((op & GS_BIND_SPECTRAL) && !gs::bind_spectral_supported(L, h->scratch, Dp, Y, ldy, Z, ldz))
        return spectral_error(L);
    // per-row partners on the tensor core: one kernel per chunk, the reconstructed rows kept on chip
    // (the same rounding of T and Q as gs_reconstruct's tensor path, and the same auto rule)
    const bool tc_ok = h->has_split && h->r >= 1 && t_dtype == GS_F32 && h->D >= gs::kMinF16Depth &&
                       (uintptr_t)T % 16 == 0 && ldt % 4 == 0;
    if (ldy != 0 && !(op & GS_BIND_DIRECT) && tc_ok && gs::rbind_tc_supported(L, h->D, Y, ldy, Z, ldz) &&
        (flags == GS_PATH_TENSOR || (flags == GS_PATH_AUTO && big_gemm(N, h->D, h->r)))) {
        st = reconstruct_bind_fused(h, (const float*)T, N, ldt, Y, ldy, L, (op & GS_UNBIND) != 0, Z, ldz, s);
        if (st != GS_ERR_SHAPE) return st;  // otherwise the scratch is too small: row chunks below
    }
    // one partner for more rows than the basis has: bind the basis instead of the rows
    if (ldy == 0 && N > h->r && h->r > 0) {
        st = reconstruct_bind_one_partner(h, T, t_dtype, N, ldt, Y, L, op, Z, ldz, flags, s);
        if (st != GS_ERR_SHAPE) return st;  // otherwise the scratch is too small: row chunks below
    }
    long long cr = std::min(h->scratch_floats / (Dp + ld16 / 2 + 1), kMaxGemmRows);
    if (cr >= 128) cr = cr / 128 * 128;
    if (cr < 1) return GS_ERR_SHAPE;
    float* xhat = h->scratch;
    float* work = h->scratch + cr * Dp;
    const long long work_floats = h->scratch_floats - cr * Dp;
    const size_t tsize = t_dtype == GS_F32 ? 4 : 2;
    for (long long c0 = 0; c0 < N; c0 += cr) {
        const long long nc = std::min(cr, N - c0);
        st = reconstruct_rows(h, (const char*)T + (size_t)c0 * ldt * tsize, t_dtype, nc, ldt, xhat, Dp, flags, s,
                              work, work_floats);
        if (st != GS_OK) return st;
        st = bind_rows(xhat, nc, h->D, Dp, Y + (size_t)c0 * ldy, ldy, L, op, Z + (size_t)c0 * ldz, ldz, s);
        if (st != GS_OK) return st;
    }
    return GS_OK;
}

gs_status gs_attention_scores(const void* Yq, const void* Yk, int in_dtype, int B, int Lq, int Lk, int r,
                              int ldy, float scale, int apply_softmax, float* A, unsigned flags,
                              void* stream) {
    if (!valid_path(flags)) return GS_ERR_INVALID_ARG;
    if (in_dtype != GS_F32 && in_dtype != GS_BF16) return GS_ERR_INVALID_ARG;
    if (B < 0 || Lq < 0 || Lk < 0 || r < 0 || ldy < r || !isfinite(scale)) return GS_ERR_SHAPE;
    if ((long long)B * Lq * Lk == 0) return GS_OK;
    if (!Yq || !Yk || !A) return GS_ERR_INVALID_ARG;
    if (B > 65535 || Lq > kMaxGemmRows) return GS_ERR_SHAPE;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GS_ERR_CUDA;
    if (!device_supported(dev)) return GS_ERR_UNSUPPORTED;
    cudaStream_t s = (cudaStream_t)stream;
    const bool tc_ok = in_dtype == GS_BF16 && gs::tc_available(dev) && gs::attn_tc_supported(r, ldy, Yq, Yk);
    const bool big = (double)B * Lq * Lk * r >= (double)(1 << 26);
    if (flags == GS_PATH_TENSOR || (flags == GS_PATH_AUTO && tc_ok && big)) {
        if (!tc_ok) return in_dtype != GS_BF16 || r > 512 ? GS_ERR_UNSUPPORTED : GS_ERR_ALIGNMENT;
        return from_cuda(gs::launch_attn_tc(Yq, Yk, B, Lq, Lk, r, ldy, scale, apply_softmax != 0, A, dev, s));
    }
    gs::GemmArgs a{};
    const int t = in_dtype == GS_F32 ? gs::MAT_F32 : gs::MAT_BF16;
    a.A = Yq; a.a_type = t; a.lda = ldy; a.a_bstride = (long long)Lq * ldy;
    a.B = Yk; a.b_type = t; a.ldb = ldy; a.b_bstride = (long long)Lk * ldy; a.b_trans = true;
    a.C = A; a.c_type = gs::MAT_F32; a.ldc = Lk; a.c_bstride = (long long)Lq * Lk;
    a.m = Lq; a.n = Lk; a.k = r; a.batch = B; a.alpha = scale;
    cudaError_t e = gs::launch_gemm_simt(a, s);
    if (e != cudaSuccess) return from_cuda(e);
    if (apply_softmax) {
        e = gs::launch_row_softmax(A, (long long)B * Lq, Lk, Lk, s);
        if (e != cudaSuccess) return from_cuda(e);
    }
    return GS_OK;
}

gs_status gs_selftest_wait_timeout(void* stream) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GS_ERR_CUDA;
    if (!device_supported(dev)) return GS_ERR_UNSUPPORTED;
    return from_cuda(gs::launch_wait_selftest((cudaStream_t)stream));
}

gs_status gs_stream_status(void* stream) {
    cudaError_t e = stream ? cudaStreamSynchronize((cudaStream_t)stream) : cudaDeviceSynchronize();
    if (e != cudaSuccess) return GS_ERR_CUDA;
    const unsigned w = gs::take_device_error_build() | gs::take_device_error_tc() | gs::take_device_error_gemm() |
                       gs::take_device_error_attn() | gs::take_device_error_rbind();
    if (w & GS_DEV_ERR_TIMEOUT) return GS_ERR_TIMEOUT;
    if (w & GS_DEV_ERR_RANGE) return GS_ERR_RANGE;
    if (w & GS_DEV_ERR_LAYOUT) return GS_ERR_UNSUPPORTED;
    return GS_OK;
}

}  // extern "C"
