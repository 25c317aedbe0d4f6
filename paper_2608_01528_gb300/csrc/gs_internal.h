// gs_internal.h -- host-side declarations shared by the library's translation units.
//
// Each .cu file owns its kernels; gs_api.cu validates arguments and calls the
// launch functions declared here.  Nothing here is part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <vector>

#include "../../include/gramspace.h"

struct gs_basis {
    int device = 0;
    int M = 0, D = 0, r = 0;
    // user-visible results (fp32)
    float* Q = nullptr;      // r x D, ld = D
    float* R = nullptr;      // M x max(r,1), ld = ldr
    int ldr = 1;
    float* cnorm = nullptr;  // M
    int* rlen = nullptr;     // M: 1 + index of the last nonzero of R_i (0 if none)
    int* rlen_chunk = nullptr; // ceil(M/32): max rlen over each 32-row chunk of R
    // tensor-core operand copies
    __half* Q16 = nullptr;   // r x ldq16 fp16, dithered rounding of Q (K-major B of X Q^T)
    int ldq16 = 0;
    __half* Q16t = nullptr;  // D x ldr16 fp16, dithered rounding of Q^T (K-major B of T Q)
    int ldr16 = 0;
    CUtensorMap tmap_q16;    // box {64, 256} over Q16 (valid when r <= 256 and Q16 != null)
    bool has_tmap_q16 = false;
    // fused tensor-core similarity: R split into two bf16 matrices (tc_mpad x
    // tc_npad, zero padded), Rh = bf16(R) and Rl = bf16(R - Rh), with tensor maps
    void* tc_Rh = nullptr;
    void* tc_Rl = nullptr;
    CUtensorMap tmap_rh, tmap_rl;   // boxes of tc_half_rows rows (fused kernel only, M <= 256)
    // the fused kernel runs S = Y R^T in halves of tc_half_rows codewords (min(tc_mpad, 128));
    // R is lower echelon, so half h needs only its first tc_nkr_half[h] K-blocks of 64
    int tc_nh = 0, tc_half_rows = 0, tc_nkr_half[2] = {0, 0};
    int tc_npad = 0, tc_mpad = 0;
    // R^T split the same way (tc_npad x tc_mpad), the B operand of V = P R
    void* tc_Rth = nullptr;
    void* tc_Rtl = nullptr;
    // Q split into bf16 hi / lo (r x ldq16): the projection's B operands when D is
    // too small for one fp16 rounding to average out (D < kMinF16Depth)
    void* tc_Qh = nullptr;
    void* tc_Ql = nullptr;
    bool has_split = false;         // tc_Rh / tc_Rl / tc_Rth / tc_Rtl exist
    // device staging of gs_project_similarity_host (gs_basis_reserve_staging): two slots,
    // each of stage_rows queries (row pitch stage_ld floats) and their argmax / maxval, a
    // stream for the host-to-device copies and the events that order the two streams
    float* stage_x = nullptr;   // 2 x stage_rows x stage_ld
    int* stage_am = nullptr;    // 2 x stage_rows
    float* stage_mv = nullptr;  // 2 x stage_rows
    long long stage_rows = 0;
    int stage_ld = 0;
    cudaStream_t stage_copy = nullptr;
    cudaEvent_t stage_start = nullptr, stage_in[2] = {nullptr, nullptr}, stage_done[2] = {nullptr, nullptr};
    // grouped bases (gs_build_basis_grouped): rows [grp_rows[g], grp_rows[g+1]) of the codebook
    // and coefficients [grp_coeffs[g], grp_coeffs[g+1]) belong to group g; empty otherwise
    std::vector<int> grp_rows, grp_coeffs;
    // host copies for the tensor-core GEMMs' K trimming (tc_prepare): R row i is zero from
    // column rlen_host[i] on (B = R: K range [kzero_host[i] = 0, rlen_host[i])), and R column j
    // is zero above row pivot_host[j] (B = R^T: K range [pivot_host[j], kM_host[j] = M))
    std::vector<int> rlen_host, pivot_host, kzero_host, kM_host;
    // scratch for the multi-kernel paths (rows processed in chunks)
    float* scratch = nullptr;
    long long scratch_floats = 0;
    long long chunk_rows = 0;
};

namespace gs {

// The fp16 projection rounds every x_d and q_jd once; those errors average out
// over the D terms of <x, q_j>, and D >= 1024 keeps the worst score error of the
// large workloads below half the 1e-4 ||x|| ||c|| bound.  Shorter rows use the
// bf16 hi / lo split (three products) instead.
constexpr int kMinF16Depth = 1024;

// ----------------------------------------------------------------- build (gs_build.cu)
// Runs the fp64 panel Gram-Schmidt and fills every field of h except the
// tensor maps.  Synchronises `s` once.
gs_status build_basis(const float* C, int M, int D, int ldc, double tau, bool normalize,
                      cudaStream_t s, gs_basis* h);
// one basis per group of rows (off: host, G + 1 increasing offsets from 0 to M), stacked into
// one handle: Q = [Q_0; Q_1; ...], R block diagonal
gs_status build_basis_grouped(const float* C, int M, int D, int ldc, const int* off, int G, double tau,
                              bool normalize, cudaStream_t s, gs_basis* h);
// dst[d][j] (cols x ldt fp16) = the basis' unbiased dithered fp16 rounding of src[j][d] (rows x
// cols fp32, ld lds): the transposed B operand of a reconstruction from other fp32 rows
cudaError_t launch_f16t_dither(const float* src, int rows, int cols, long long lds, void* dst, long long ldt,
                               cudaStream_t s);
// a handle from a saved basis (fp32 Q r x D, R M x r, optional norms), same finalisation as a build
gs_status import_basis(const float* Q, int ldq, const float* R, int ldr_in, const float* cnorm, int M, int D,
                       int r, cudaStream_t s, gs_basis* h);

// ----------------------------------------------------------------- SIMT kernels (gs_simt.cu)
enum { MAT_F32 = 0, MAT_BF16 = 1 };

// fused small-r project + similarity, one warp per query (r <= 32)
cudaError_t launch_ps_warp(const float* X, long long N, int ldx, int D, const float* Q, int r,
                           const float* R, int ldr, int M, const float* cnorm, int mode, float scale,
                           float* Y, int ldy, float* S, int lds, int* argmax, float* maxval,
                           cudaStream_t s);

// similarity of Gram-loc queries Y (N x r, r <= 64), one warp per query; every mode, S optional
constexpr int kMaxCoeffsWarpR = 64;
cudaError_t launch_coeffs_warp(const float* Y, long long N, int ldy, int r, const float* R, int ldr, int M,
                               const float* cnorm, int mode, float scale, float* S, int lds, int* argmax,
                               float* maxval, cudaStream_t s);

// C = alpha * A * op(B), batched over `batch` with element strides.
//   A: m x k (lda), B: trans ? n x k : k x n (ldb); types MAT_F32 / MAT_BF16.
//   rownorm/colnorm (optional): C[i][j] /= rownorm[i]*colnorm[j] (0 if product is 0)
//   out type MAT_F32 / MAT_BF16.
struct GemmArgs {
    const void* A; int a_type; long long lda; long long a_bstride;
    const void* B; int b_type; long long ldb; long long b_bstride; bool b_trans;
    void* C; int c_type; long long ldc; long long c_bstride;
    long long m; int n, k, batch;
    float alpha;
    const float* rownorm; const float* colnorm;
    const int* b_rowlen;  // optional (b_trans only): row j of B is zero beyond b_rowlen[j]
    // optional gate (batch 1, no split): only 64-row tiles holding a row i whose squared norm
    // gate_xn2[i] + gate_xn2[gate_ld + i] is nonzero and outside [gate_lo, gate_hi] are computed;
    // the other blocks return at once (rewrites the rows that one fp16 rounding could not hold)
    const float* gate_xn2; long long gate_ld; float gate_lo, gate_hi;
    int ksplit;           // > 1 (batch 1, fp32 C only): K is cut into ksplit chunks, one per
                          // grid z index; each chunk's m x n partial product goes to kpart
                          // (ksplit x m x n floats, caller's workspace) and a second kernel
                          // sums the chunks in a fixed order into C (deterministic)
    float* kpart;
};
cudaError_t launch_gemm_simt(const GemmArgs& g, cudaStream_t s);

// per-row ||x||
cudaError_t launch_rownorm(const float* X, long long N, int ldx, int D, float* out, cudaStream_t s);

// per-row, per-group argmax (index within the group) and max over S (N x M, lds); groups are
// column ranges [off[g], off[g+1]), G <= kMaxGroups; outputs N x G
constexpr int kMaxGroups = 256;
cudaError_t launch_group_argmax(const float* S, long long N, int lds, const int* off, int G, int* argmax,
                                float* maxval, cudaStream_t s);

// block circular convolution (unbind: correlation) of rows of X with rows of Y (ldy = 0: Y's
// row 0 for every row), blocks of L (L divides D): k_bind_reg for L <= 32 with L % 4 == 0,
// k_bind16 / k_bind8 for L % 16 / L % 8 == 0 up to kMaxBindFastL, k_bind1 otherwise
constexpr int kMaxBindFastL = 16384;
cudaError_t launch_bind(const float* X, long long N, int D, int ldx, const float* Y, long long ldy, int L, bool unbind,
                        float* Z, int ldz, cudaStream_t s);
// the same through block spectra (gs_bind_spec.cu): L a power of two in [kMinBindSpectralL,
// kMaxBindSpectralL], rows 8-byte aligned (bind_spectral_supported)
constexpr int kMinBindSpectralL = 64;
constexpr int kMaxBindSpectralL = 8192;
bool bind_spectral_supported(int L, const float* X, int ldx, const float* Y, long long ldy, const float* Z, int ldz);
cudaError_t launch_bind_spectral(const float* X, long long N, int D, int ldx, const float* Y, long long ldy, int L,
                                 bool unbind, float* Z, int ldz, cudaStream_t s);

// per-row argmax / maxval over S (N x M); SOFTMAX mode rewrites the row in place.
cudaError_t launch_row_finish(float* S, long long N, int M, int lds, bool softmax, int* argmax,
                              float* maxval, cudaStream_t s);

// row softmax in place over rows of length L (stride ld)
cudaError_t launch_row_softmax(float* A, long long rows, int L, long long ld, cudaStream_t s);

// ----------------------------------------------------------------- tensor-core kernels (gs_tc.cu)
bool tc_available(int device);
// creates the tensor maps of h's fp16 operand copies (after build_basis)
gs_status tc_prepare(gs_basis* h);
// fused project + similarity on tcgen05 (requires h->has_tmap_q16: r <= 256, M <= 256)
cudaError_t launch_ps_tc(const gs_basis* h, const float* X, long long N, int ldx, int mode,
                         float scale, float* Y, int ldy, float* S, int lds, int* argmax,
                         float* maxval, cudaStream_t s);

// ----------------------------------------------------------------- general tcgen05 GEMM (gs_gemm_tc.cu)
// C = alpha * A B^T (/ rownorm[i] colnorm[j] when both are given).  A: fp32 m x K
// (lda % 4 == 0, 16-byte aligned).  split = false: B0 fp16 n x K, one fp16
// rounding of A; split = true: B0 / B1 bf16 hi / lo, A split into bf16 hi / lo
// (three products).  B rows 16-byte aligned (ldb % 8 == 0).  C fp32 or bf16.
struct GemmTcArgs {
    const void* A; long long lda; long long m; int K;
    bool split;
    bool a_half;    // A already fp16 (lda in halves, multiple of 8): TMA feeds the MMA directly
    const void* B0; const void* B1; long long ldb; int n;
    void* C; long long ldc; bool c_bf16; float alpha;
    const float* rownorm; const float* colnorm;
    // optional HOST arrays (n each): B row j is zero outside K columns [b_klo[j], b_khi[j]);
    // K-blocks outside a column tile's union are skipped (exact: only zero products dropped)
    const int* b_klo; const int* b_khi;
    // fp16-rounded fp32 A only (optional): the converters write each row's squared norm, as two
    // partial sums xn2_out[row] + xn2_out[m + row] (2 x m floats), so the caller can find the rows
    // that one fp16 rounding cannot represent accurately
    float* xn2_out;
    // optional (m floats): every output of row i is multiplied by rowmul[i] (the inverse of an
    // exact power-of-two scale applied to A's row before its fp16 rounding)
    const float* rowmul;
};
cudaError_t launch_gemm_tc(const GemmTcArgs& a, int device, cudaStream_t s);
// fp32 rows -> fp16 (RN) for the fp16-A GEMM, each row first multiplied by the exact power of two
// 2^s that brings its largest magnitude to [2^14, 2^15) (inside fp16's range, far above its
// subnormals); rowmul[row] receives 2^-s.  Rows that are zero or hold a non-finite value keep s = 0.
cudaError_t launch_round_f16(const float* X, long long ldx, long long rows, int cols, void* out, long long ldo,
                             float* rowmul, cudaStream_t s);

// ----------------------------------------------------------------- reconstruct + bind on tcgen05 (gs_rbind_tc.cu)
// Z = op(T Q, Y) with per-row partners in one kernel: T16 (m x r fp16 rows, ld16 halves, each row
// scaled by an exact power of two whose inverse is rowmul[i]), the basis' Q16t, Y and Z (m rows of
// D floats, lds ldy / ldz).  L in {64, 128, 256}; Y, Z 16-byte aligned, ldy, ldz multiples of 4.
bool rbind_tc_supported(int L, int D, const float* Y, long long ldy, const float* Z, int ldz);
cudaError_t launch_rbind_tc(const gs_basis* h, const void* T16, long long ld16, long long m, const float* rowmul,
                            const float* Y, long long ldy, int L, bool unbind, float* Z, int ldz, int device,
                            cudaStream_t s);

// ----------------------------------------------------------------- attention scores on tcgen05 (gs_attn_tc.cu)
// bf16 Yq (B x Lq x r) and Yk (B x Lk x r), row stride ldy; fp32 A (B x Lq x Lk, dense).
bool attn_tc_supported(int r, long long ldy, const void* Yq, const void* Yk);
cudaError_t launch_attn_tc(const void* Yq, const void* Yk, int B, int Lq, int Lk, int r, long long ldy, float scale,
                           bool softmax, float* A, int device, cudaStream_t s);

// ----------------------------------------------------------------- device error words
// Each translation unit with kernels that can report device-side errors keeps
// its own word; gs_stream_status reads and clears all of them.
unsigned take_device_error_build();
unsigned take_device_error_tc();
// one block whose wait on a never-completed mbarrier runs out (failure-detection self-test)
cudaError_t launch_wait_selftest(cudaStream_t s);
unsigned take_device_error_gemm();
unsigned take_device_error_attn();
unsigned take_device_error_rbind();

}  // namespace gs

#define GS_DEV_ERR_TIMEOUT 0x1u
#define GS_DEV_ERR_RANGE 0x2u
#define GS_DEV_ERR_LAYOUT 0x4u  // a kernel's shared-memory buffers did not fit where they landed
