/*
 * gramspace.h -- C ABI of the GB300 (sm_103a) Gram-Space codebook library.
 *
 * Gram-Space (Wang & Li, "Gram-Space: Structure-Preserving Codebook
 * Compression for Memory-Efficient Neuro-Symbolic AI") replaces a VSA codebook
 * by an orthonormal basis of its span and the codewords' coordinates in that
 * basis ("Gram-loc"), runs matrix-space operators (similarity, probability
 * vectorization, attention scores) on the coordinates, and reconstructs
 * full vectors only before component-wise operators.
 *
 * Notation.  The paper stores the codebook as W (D x M, one atom per column),
 * the basis as U (D x k) and the Gram-loc codebook T = U^T W (k x M) (Sec. 3.1,
 * Eq. 1).  This library stores every matrix row-major with one vector per
 * row:  C = W^T (M x D),  Q = U^T (r x D, r = k),  R = T^T (M x r),  C = R Q.
 * The Gram-loc of a query x (t = U^T x, Sec. 3.1) is the row y = x Q^T.
 *
 * Conventions shared by every entry point:
 *  - Array arguments are DEVICE pointers owned by the caller unless a
 *    function says otherwise.  The library owns only what a gs_basis holds.
 *  - Matrices are row-major; ld* arguments are leading dimensions in
 *    elements (ld >= number of columns).
 *  - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *    stream) and returns before it finishes.  Argument errors are detected on
 *    the host and returned immediately with nothing enqueued.
 *  - Errors that only the device can see (a bounded wait that ran out, an
 *    input outside a fast path's numeric range) set a per-device error word;
 *    gs_stream_status() synchronises the stream and returns and clears it.
 *  - Only gs_build_basis, gs_build_basis_grouped, gs_basis_import and
 *    gs_basis_reserve_staging allocate device memory; the other calls allocate nothing.  N = 0 is a
 *    valid no-op.
 *  - All functions are callable from any host thread; a gs_basis must not be
 *    destroyed while work that uses it is in flight.  Some paths keep
 *    intermediate results in a scratch area owned by the gs_basis (the two-GEMM
 *    similarity for bases the fused kernel cannot hold, the tensor-core
 *    reconstruct, gs_similarity_coeffs), so calls on one gs_basis that may run
 *    at the same time on the GPU (different streams) must be ordered by the
 *    caller.
 */
#ifndef GRAMSPACE_H
#define GRAMSPACE_H

#ifdef __cplusplus
extern "C" {
#endif

/* Every entry point is exported from the shared library; everything else in
 * it has hidden visibility. */
#if defined(__GNUC__)
#define GS_API __attribute__((visibility("default")))
#else
#define GS_API
#endif

typedef enum gs_status {
    GS_OK = 0,
    GS_ERR_INVALID_ARG = 1,  /* null pointer, negative size or unknown enum/flag   */
    GS_ERR_ALIGNMENT = 2,    /* pointer or leading dimension not aligned as stated */
    GS_ERR_SHAPE = 3,        /* sizes inconsistent with the basis or beyond limits */
    GS_ERR_NOMEM = 4,        /* a device allocation failed                          */
    GS_ERR_CUDA = 5,         /* a CUDA runtime / driver call failed                 */
    GS_ERR_TIMEOUT = 6,      /* a bounded device-side wait gave up (device word)    */
    GS_ERR_RANGE = 7,        /* a query row of the fused tensor-core similarity has a
                                squared norm that is not a finite fp32 number (an
                                entry near 2^64 or beyond, or an infinity); results of
                                that call are invalid, rerun it with GS_PATH_SIMT
                                (device word)                                        */
    GS_ERR_UNSUPPORTED = 8   /* no sm_103 device, or a forced path cannot run (or,
                                as a device word, a kernel found its shared-memory
                                window placed so that its buffers do not fit; it
                                returned without writing)                          */
} gs_status;

typedef enum gs_dtype { GS_F32 = 0, GS_BF16 = 1 } gs_dtype;

typedef enum gs_score_mode {
    GS_SCORE_RAW = 0,      /* S = scale * <y, R_i>                          */
    GS_SCORE_COSINE = 1,   /* S = scale * <y, R_i> / (||x|| * ||c_i||)      */
    GS_SCORE_SOFTMAX = 2   /* S = softmax_i(scale * <y, R_i>) over M atoms  */
} gs_score_mode;

/* gs_build_basis flags */
#define GS_BUILD_NORMALIZE_ROWS 0x1u /* build on c_i / ||c_i|| (the atoms scaled to
                                        unit length first, Sec. 3.1)              */

/* path-selection flags of the apply calls (at most one) */
#define GS_PATH_AUTO 0x0u   /* pick by problem size                                 */
#define GS_PATH_SIMT 0x1u   /* fp32 CUDA-core kernels: fp32 accumulation, any range */
#define GS_PATH_TENSOR 0x2u /* tcgen05 tensor-core kernels (GS_ERR_UNSUPPORTED when
                               the shape has no tensor-core kernel)                 */

typedef struct gs_basis gs_basis;

/*
 * Basis construction (Sec. 3.1, Eq. 1; built once, at initialisation, by
 * Gram-Schmidt, Sec. 3.3; rank k = algebraic rank, Sec. 3.2).
 *
 * Orthonormalises the rows of C (M x D, fp32, ld = ldc) in row order by
 * Gram-Schmidt with two projection passes per row (reorthogonalisation),
 * computed in fp64 on the device in panels of rows.  Row i is accepted as a
 * new basis direction when the norm left after both passes exceeds
 * rank_tol * ||c_i||; otherwise it is dependent and keeps only its
 * coefficients.  Produces Q (r x D) with Q Q^T = I_r, R (M x r, lower echelon,
 * positive pivots) with C = R Q, ||c_i|| per row, and r.
 *
 * rank_tol: relative tolerance (> 0; 1e-6 is the library's default reading).
 * flags: 0 or GS_BUILD_NORMALIZE_ROWS.
 * out: receives a new handle owning Q, R, the norms and the derived operand
 *      copies of the tensor-core kernels.  Destroy with gs_basis_destroy.
 * Synchronises `stream` once (to learn r).  Requires 1 <= M, 1 <= D, ldc >= D.
 * Errors: GS_ERR_INVALID_ARG, GS_ERR_SHAPE, GS_ERR_NOMEM, GS_ERR_CUDA,
 *         GS_ERR_UNSUPPORTED (no sm_103 device), GS_ERR_TIMEOUT (a bounded wait
 *         between the cooperating blocks of the build ran out; no handle).
 */
GS_API gs_status gs_build_basis(const float* C, int M, int D, int ldc, float rank_tol,
                         unsigned flags, void* stream, gs_basis** out);

/*
 * Grouped basis (Sec. 3.1: when D < M the codebook is rank-deficient, so its
 * entries are partitioned into subsets of at most D, each subset gets its own
 * orthonormal basis, and the reconstructions are concatenated into the full
 * codebook layout).  The same construction holds several attribute codebooks
 * (e.g. one per RAVEN attribute) in one handle, so one launch scores a query
 * against all of them.
 *
 * Rows [group_offsets[g], group_offsets[g+1]) of C form group g; group_offsets
 * is a HOST array of G + 1 increasing ints from 0 to M (1 <= G <= 256, every
 * group non-empty).  Each group is orthonormalised alone exactly as
 * gs_build_basis does (same rank_tol and flags), giving Q_g (r_g x D) and R_g.
 * The handle holds the stacked Q = [Q_0; Q_1; ...] (r = r_0 + ... + r_(G-1)
 * rows; rows of one group are orthonormal, rows of different groups need not
 * be, and r may exceed D) and the block-diagonal R (M x r): row i of group g
 * carries R_g's row in columns [s_g, s_g + r_g), s_g = r_0 + ... + r_(g-1), and
 * zeros elsewhere.  C = R Q holds row by row, so every other call works on the
 * handle unchanged: scores cover all M entries in the original layout, Gram-loc
 * rows and prob-vectorized rows use the stacked coordinates, and reconstruction
 * returns the concatenated codebook layout.  gs_basis_groups reports the group
 * and coordinate offsets; gs_group_argmax picks the best entry per group.
 * Synchronises `stream` once per group.  Errors as gs_build_basis; invalid
 * offsets give GS_ERR_INVALID_ARG.
 */
GS_API gs_status gs_build_basis_grouped(const float* C, int M, int D, int ldc, const int* group_offsets, int G,
                                        float rank_tol, unsigned flags, void* stream, gs_basis** out);

/*
 * Group layout of a handle: *G groups; row_offsets and coeff_offsets (HOST
 * arrays of *G + 1 ints, either may be NULL; call once with both NULL to learn
 * *G) receive the codebook-row and Gram-loc-coordinate ranges of each group.
 * A handle from gs_build_basis or gs_basis_import is one group: {0, M}, {0, r}.
 */
GS_API gs_status gs_basis_groups(const gs_basis* h, int* G, int* row_offsets, int* coeff_offsets);

/*
 * Best entry of each group for each score row (hard selection per attribute,
 * Sec. 2.2, on the scores of a grouped codebook): S is N x M fp32 (ld = lds >=
 * group_offsets[G]); group g is columns [group_offsets[g], group_offsets[g+1])
 * (HOST array of G + 1 increasing ints from 0, 1 <= G <= 256).  argmax (N x G
 * int32, ld G) receives the index WITHIN the group of the first column holding
 * the group's maximum, maxval (N x G fp32, ld G) that maximum; either may be
 * NULL, not both.  N = 0 is a no-op.
 */
GS_API gs_status gs_group_argmax(const float* S, long long N, int lds, const int* group_offsets, int G,
                                 int* argmax, float* maxval, void* stream);

/*
 * Read-only view of a basis: sizes and device pointers to Q (r x D, ld = D),
 * R (M x r, ld = r) and cnorm (M, fp32 ||c_i||).  Any output pointer may be
 * NULL.  The pointers stay valid until gs_basis_destroy.
 */
GS_API gs_status gs_basis_info(const gs_basis* h, int* M, int* D, int* r, const float** Q,
                        const float** R, const float** cnorm);

/*
 * Restores a handle from a basis saved earlier: the checkpoint / restore of the
 * state gs_build_basis computes once at initialisation (Sec. 3.3), without
 * running Gram-Schmidt again.  Save what gs_basis_info returns (Q, R, cnorm,
 * with r, M, D) and pass it back here: every result of the restored handle then
 * equals the original's bit for bit (its fp16 / bf16 operand copies are derived
 * from the same fp32 values).
 *   Q      r x D fp32, ld = ldq >= D (may be NULL when r = 0)
 *   R      M x r fp32, ld = ldr >= r (may be NULL when r = 0)
 *   cnorm  M fp32 codeword norms, or NULL to use ||R_i|| (equal to ||c_i||
 *          because C = R Q with orthonormal Q)
 * Device pointers owned by the caller; the handle keeps its own copies.  The
 * rows of Q are taken as orthonormal and R as lower echelon (as a build leaves
 * them; for a grouped basis, orthonormal within each group and block diagonal,
 * with r <= M); neither is re-checked.  A restored grouped basis reports one
 * group (pass the offsets to gs_group_argmax explicitly).  Synchronises
 * `stream` before returning.
 */
GS_API gs_status gs_basis_import(const float* Q, int r, int D, int ldq, const float* R, int M, int ldr,
                                 const float* cnorm, void* stream, gs_basis** out);

/* Releases a handle and its device memory (synchronises its device first). */
GS_API gs_status gs_basis_destroy(gs_basis* h);

/*
 * Fused project + similarity (Sec. 3.1: t = U^T x; Sec. 2.2 scaled dot-product
 * similarity; Sec. 3.2, Eq. 2-3: scores computed on Gram-loc equal the
 * uncompressed ones).
 *
 * X: N x D queries (fp32, ld = ldx).  Computes Y = X Q^T (N x r) and scores
 * against the M codewords in Gram-loc, S = Y R^T, then per `mode`
 * (gs_score_mode) with `scale`; COSINE divides by the full D-dimensional
 * ||x_n|| and by ||c_i||.  Optional outputs (NULL to skip):
 *   Y      N x r fp32, ld = ldy          argmax  N int32 (lowest index on ties)
 *   S      N x M fp32, ld = lds          maxval  N fp32 (S at argmax)
 * At least one output must be non-NULL.  When r = 0 every score is 0 (softmax:
 * 1/M) and argmax is 0.
 * Tensor-core path (GS_PATH_AUTO picks it for large N): X is rounded to fp16
 * on the fly (D >= 1024; shorter rows are split into bf16 hi / lo), Q is a
 * fixed fp16 copy with unbiased dithered rounding, fp32 accumulation; the
 * scores S = Y R^T are taken with Y and R split into bf16 hi / lo.  One fp16
 * rounding of a row is accurate while 2^-8 sqrt(D) <= ||x|| <= 2^15; the kernels
 * find every other nonzero row from its norm and compute it again within the
 * same call -- the fused kernel (r <= 256, M <= 256) redoes the row's tile on
 * x 2^s with an exact power of two s that brings ||x|| 2^s to [2^14, 2^15), the
 * two-GEMM path (wider bases) recomputes the row's Y in fp32 -- so the results
 * meet the same relative bound for queries of any magnitude.  Only a row whose
 * squared norm is not a finite fp32 number raises GS_ERR_RANGE (fused kernel).
 * Requires X 16-byte aligned and ldx % 4 == 0 on the tensor-core path.
 */
GS_API gs_status gs_project_similarity(const gs_basis* h, const float* X, long long N, int ldx,
                                int mode, float scale, unsigned flags, float* Y, int ldy,
                                float* S, int lds, int* argmax, float* maxval, void* stream);

/*
 * Device staging for gs_project_similarity_host, owned by the handle: two slots,
 * each holding `rows` queries of the basis' dimension D (fp32) and their argmax /
 * maxval (2 x rows x (4 D + 8) bytes), plus a copy stream and five events.
 * rows = 0 releases it (gs_basis_destroy releases it too); a new call replaces
 * the old staging.  Reserve it once, outside any timed or latency-critical code:
 * besides the two builds this is the only call that allocates.  Must not be
 * called while work that uses the staging is in flight.
 */
GS_API gs_status gs_basis_reserve_staging(gs_basis* h, long long rows);

/*
 * Project + similarity from HOST memory (Sec. 3.1 / 2.2, as gs_project_similarity
 * with Y and S not returned): X is N x D fp32 in host memory (ld = ldx >= D),
 * argmax / maxval are host arrays of N (either may be NULL, not both).  The
 * queries go through the staging (gs_basis_reserve_staging) in chunks of its
 * rows, alternating between its two slots: chunk i is copied in on the handle's
 * copy stream while chunk i - 1 is scored on `stream`, and each chunk's results
 * are copied back on `stream`.  The work starts after what is already enqueued on
 * `stream`, and work enqueued on `stream` after the call starts after all of it.
 * The call returns before the work finishes: X must stay unchanged and the host
 * arrays valid until then.  Use page-locked host memory (cudaHostAlloc, torch
 * pin_memory) for the copies to run asynchronously at the link's rate.
 * Returns GS_ERR_INVALID_ARG when no staging has been reserved.  The staging is
 * shared by every call on the handle: calls on different streams must be ordered.
 */
GS_API gs_status gs_project_similarity_host(const gs_basis* h, const float* X, long long N, int ldx, int mode,
                                            float scale, unsigned flags, int* argmax, float* maxval,
                                            void* stream);

/*
 * Similarity of queries given by their Gram-loc coordinates (Sec. 3.2, Eq. 2:
 * inner products between vectors in span(C) equal those of their Gram-loc
 * coordinates; Sec. 2.2 scaled dot-product similarity).  This is the lookup that
 * never touches a D-dimensional vector: its cost does not grow with D (the
 * "compressed" row of the paper's latency-versus-dimension table).
 *
 * Y: N x r fp32 Gram-loc queries (ld = ldy >= r), e.g. V from gs_prob_vectorize
 * or Y from gs_project_similarity.  S = scale * Y R^T (N x M); COSINE divides by
 * ||y_n|| (equal to ||x_n|| for x in span(C), Eq. 3) and ||c_i||; SOFTMAX as in
 * gs_project_similarity.  Outputs S (ld = lds), argmax, maxval as in
 * gs_project_similarity; at least one must be non-NULL.  Y may be NULL only when
 * r = 0 (every score is then 0).
 * Tensor-core path (GS_PATH_AUTO for large N·M·r): Y and R split into bf16 hi /
 * lo, three products, fp32 accumulation (~2^-16 relative); needs Y 16-byte
 * aligned and ldy % 4 == 0.  Otherwise fp32 CUDA cores.  Uses the basis'
 * scratch for cosine norms and, when S is NULL, for the scores.
 */
GS_API gs_status gs_similarity_coeffs(const gs_basis* h, const float* Y, long long N, int ldy, int mode,
                                      float scale, unsigned flags, float* S, int lds, int* argmax,
                                      float* maxval, void* stream);

/*
 * Probability vectorization on Gram-loc (Sec. 2.2: weighted sum of codewords
 * with attribute probabilities as weights; Sec. 3.1 / 3.3: run on Gram-loc).
 * V = P R: P is N x M (fp32, ld = ldp), V is N x r of type v_dtype
 * (GS_F32 or GS_BF16, ld = ldv).  V is the Gram-loc of P C.
 * fp32 V: fp32 CUDA-core arithmetic.  bf16 V: bf16 tensor-core product with
 * fp32 accumulation when GS_PATH_AUTO/TENSOR and the shape allows it.
 */
GS_API gs_status gs_prob_vectorize(const gs_basis* h, const float* P, long long N, int ldp, void* V,
                            int v_dtype, int ldv, unsigned flags, void* stream);

/*
 * Reconstruction, the "decompose" step (Sec. 3.1 and Sec. 3.3: x = U t before
 * component-wise operators).  Xhat = T Q: T is N x r coefficients of type
 * t_dtype (GS_F32 or GS_BF16, ld = ldt), Xhat is N x D fp32 (ld = ldxh).
 * Reconstructing R itself returns the codebook C (exact up to rounding).
 * Tensor-core path (GS_PATH_AUTO for large N with fp32 T, D >= 1024, T 16-byte
 * aligned, ldt % 4 == 0; GS_PATH_TENSOR returns GS_ERR_UNSUPPORTED for D <
 * 1024, where one fp16 rounding no longer averages out over the rows of Q):
 * each row of T is multiplied by an exact power of two that
 * brings its largest magnitude to [2^14, 2^15), rounded once to fp16 into the
 * handle's scratch, multiplied by the dithered fp16 Q with fp32 accumulation,
 * and the row's scale is undone in fp32, so the result is accurate for rows of
 * any magnitude (down to a largest entry of 2^-112).  Otherwise fp32 CUDA cores.
 */
GS_API gs_status gs_reconstruct(const gs_basis* h, const void* T, int t_dtype, long long N, int ldt,
                         float* Xhat, int ldxh, unsigned flags, void* stream);

/* binding operators of gs_bind / gs_reconstruct_bind, optionally OR-ed with one method */
#define GS_BIND 0   /* block circular convolution  */
#define GS_UNBIND 1 /* block circular correlation  */
#define GS_BIND_DIRECT 2   /* the direct sum: one fp32 sum of L products per output    */
#define GS_BIND_SPECTRAL 4 /* through block spectra (convolution theorem): L a power
                              of two in [64, 8192], rows 8-byte aligned               */

/*
 * Binding and unbinding, the component-wise operators of rule execution
 * (Sec. 2.2: binding / unbinding with a modulo-style index computation;
 * Sec. 3.3: the operators after reconstruction are based on circular
 * convolution).  Rows are cut into blocks of L consecutive components (L
 * divides D; L = D is one circular convolution over the whole vector) and,
 * within block b of row n,
 *   GS_BIND:   Z[n][bL+k] = sum_j X[n][bL+j] * Y[n][bL + ((k - j) mod L)]
 *   GS_UNBIND: Z[n][bL+k] = sum_j X[n][bL+j] * Y[n][bL + ((j - k) mod L)]
 * (unbinding with y undoes binding with y when y's block spectra have unit
 * modulus, and approximately for random y).  X, Z: N x D fp32 (ld = ldx,
 * ldz >= D); Y: N x D fp32 with ld = ldy >= D, or ldy = 0: Y's single row
 * binds every row.  Methods (op | method), both fp32 CUDA-core arithmetic:
 *   GS_BIND_DIRECT: one sum per output in j order; |error| <= L 2^-22
 *     ||x_b|| ||y_b|| per output of block b.
 *   GS_BIND_SPECTRAL: z = IDFT(DFT(x) DFT(y)) per block (conj(DFT(y)) to
 *     unbind) with fp32 radix-2^k transforms, ~5 L log2 L flops per block
 *     instead of 2 L^2; |error| <= sqrt(2L) (3 e + 4u) ||x_b|| ||y_b||, where
 *     u = 2^-24, e = K eta / (1 - K eta) + 10u, eta = 10u and K = log2(L) + 2
 *     (log2(L) + 1 for L <= 512): the transform error bound of the radix-2
 *     FFT (Higham, Accuracy and Stability of Numerical Algorithms, Thm 24.2)
 *     carried through the product and the inverse; typical errors are far
 *     smaller than the direct sum's.
 *   neither: GS_BIND_SPECTRAL where it applies, else GS_BIND_DIRECT.
 * Z must not overlap X or Y.
 * Errors: GS_ERR_SHAPE (L does not divide D, ld too small), GS_ERR_INVALID_ARG
 * (unknown op or both methods), GS_ERR_UNSUPPORTED (GS_BIND_SPECTRAL with an L
 * it does not take), GS_ERR_ALIGNMENT (GS_BIND_SPECTRAL with a pointer or ld
 * that leaves a row start off an 8-byte boundary).
 */
GS_API gs_status gs_bind(const float* X, long long N, int D, int ldx, const float* Y, long long ldy, int L, int op,
                         float* Z, int ldz, void* stream);

/*
 * Reconstruction followed by binding at the transition into component-wise
 * operators (Sec. 3.3: reconstruction is placed immediately before binding and
 * unbinding): Z = op(T Q, Y) with gs_reconstruct's T (N x r, t_dtype, ldt) and
 * gs_bind's Y, L, op (with its method) and Z.  With one partner row for more
 * rows than the basis has (ldy = 0, N > r), binding is applied to the basis
 * instead of the rows: op(t Q, y) = t op(Q, y) by linearity, so the r basis rows
 * are bound once and every row is reconstructed straight from them -- the
 * reconstructed rows are never formed, and the call costs one reconstruction
 * plus the binding of r rows; its error is then at most (f + eps) ||y_b||
 * sum_j |t_j| ||q_j,b|| per output of block b, with f the multiplier of
 * ||x_b|| ||y_b|| in gs_bind's bound for the method, and eps = 2^-10 + r 2^-23 on the tensor-core path (r 2^-23 in fp32).
 * With per-row partners on the tensor-core path, L in {64, 128, 256}, Y and Z
 * 16-byte aligned with ldy, ldz multiples of 4, and a spectral (or default)
 * method, one kernel per chunk of rows reconstructs each 128-row x 256-column
 * tile on the tensor core and binds it through block spectra held in tensor
 * memory: only Z is written (the reconstruction's error, 1e-4 ||t||, carried
 * through the binding, plus the spectral bound).  Otherwise the rows are
 * processed in chunks whose reconstruction lives in the handle's scratch
 * between the two kernels (the caller needs no N x D buffer for the
 * reconstructed vectors).  flags picks the reconstruction path as in
 * gs_reconstruct.
 * Shares the handle's scratch with the other multi-kernel calls: order calls
 * on one handle.
 */
GS_API gs_status gs_reconstruct_bind(const gs_basis* h, const void* T, int t_dtype, long long N, int ldt,
                                     const float* Y, long long ldy, int L, int op, float* Z, int ldz, unsigned flags,
                                     void* stream);

/*
 * Attention scores between compressed vectors (Sec. 2.2 attention score;
 * Sec. 3.2: attention computed by matrix multiplication is preserved on
 * Gram-loc).  For each of B sequences: A[b] = scale * Yq[b] Yk[b]^T
 * (Lq x Lk, fp32), followed by a row softmax over the Lk keys when
 * apply_softmax != 0.  Yq is B x Lq x r and Yk is B x Lk x r, both of type
 * in_dtype (GS_F32 or GS_BF16) with row stride ldy elements; A is
 * B x Lq x Lk fp32, dense.  scale = 1/sqrt(D) reproduces full-dimension
 * attention.  Tensor-core path: bf16 inputs, fp32 accumulation.
 */
GS_API gs_status gs_attention_scores(const void* Yq, const void* Yk, int in_dtype, int B, int Lq,
                              int Lk, int r, int ldy, float scale, int apply_softmax, float* A,
                              unsigned flags, void* stream);

/*
 * Project + similarity that allocates nothing (the paper has no counterpart;
 * this is a deployment variant).  For callers that cannot call cudaMalloc:
 * code running under a CUDA graph capture that forbids allocation, plugins
 * confined to a host framework's fixed device-memory budget, integrations whose
 * own allocator owns all device memory.  No basis handle is needed: the caller
 * passes the basis it holds, Q (r x D fp32, ld = D), R (M x r fp32, ld = r)
 * and cnorm (M fp32, only read for GS_SCORE_COSINE), plus X (N x D fp32,
 * ld = ldx) and receives argmax and/or maxval (N each; either may be NULL, not
 * both).  Scores are computed like gs_project_similarity with GS_PATH_SIMT
 * (fp32 CUDA cores, any value range).
 * Scratch lives in a fixed 16 MiB device array inside the library (held by
 * every GPU that loads it until exit), processed in chunks of rows; a problem
 * with r + M + 1 > 4,194,304 is rejected with GS_ERR_SHAPE.  The first call on
 * a device looks up that array's device address (cudaGetSymbolAddress) with
 * the device current, so make that first call before any stream capture; the
 * address is kept per device context and looked up again after the context
 * changes (cudaDeviceReset), so the first call after a reset must also come
 * before any capture.  All calls on a device share the array: calls that
 * overlap on the GPU race.  `stream` must belong to the current device
 * (GS_ERR_INVALID_ARG otherwise).
 * Errors: GS_ERR_INVALID_ARG, GS_ERR_SHAPE, GS_ERR_CUDA, GS_ERR_UNSUPPORTED.
 */
GS_API gs_status gs_project_similarity_static(const float* Q, int r, int D, const float* R, int M,
                                              const float* cnorm, const float* X, long long N, int ldx,
                                              int mode, float scale, int* argmax, float* maxval,
                                              void* stream);

/*
 * Synchronises `stream` (NULL = the whole device) and returns the first error
 * the device recorded since the last call (GS_ERR_TIMEOUT, GS_ERR_RANGE), or
 * GS_ERR_CUDA if the stream itself failed; clears the recorded word.
 */
GS_API gs_status gs_stream_status(void* stream);

/*
 * Self-test of the device-side failure detection (the paper has no counterpart:
 * this checks the library's own machinery).  Every wait of the tensor-core
 * kernels on a pipeline barrier is bounded (2 s); when one runs out the kernel
 * records a timeout in the device error word, unwinds and returns, so the CUDA
 * context stays usable.  This call enqueues one block on `stream` whose single
 * thread waits, through that same bounded wait, on a barrier that nothing will
 * ever complete: about 2 s later gs_stream_status() on that stream returns
 * GS_ERR_TIMEOUT.  Returns GS_ERR_UNSUPPORTED on devices other than sm_103.
 */
GS_API gs_status gs_selftest_wait_timeout(void* stream);

/* Static, human-readable name of a status code. */
GS_API const char* gs_status_string(gs_status s);

/* Library version, major*10000 + minor*100 + patch. */
GS_API int gs_version(void);

#ifdef __cplusplus
}
#endif

#endif /* GRAMSPACE_H */
