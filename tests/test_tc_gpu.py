"""GPU parity of the tcgen05 kernels against the oracle.

Same bar as the fp32 paths: |S - S*| <= 1e-4 ||x|| ||c_i||, Y within 1e-4 ||x||,
argmax bit-exact wherever the oracle's top-2 margin exceeds twice the score
tolerance, V within 1e-4 sum_i |p_i| ||c_i|| (plus 2^-8 |V*| for bf16 output),
Xhat within 1e-4 ||t||.  The kernels round X (or T) to fp16 (RN) against a
dithered fp16 copy of the basis with fp32 accumulation, and take the products
whose terms do not average out (S = Y R^T, V = P R) with both operands split
into bf16 hi / lo.
"""
import numpy as np
import pytest
import torch

import synth
from test_parity_gpu import TOL_S, check_scores, cuda, host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def large_ref(orc):
    C = synth.large_codebook()
    return C, orc.build_basis(C)


def test_tc_large_full_size(gs, orc, large_ref):
    """The full large-batch workload on the tensor-core path: every argmax equals
    its generating label; Y, S and maxval of a seeded sample of rows match the
    oracle, and S of every row stays within the bound of the label score."""
    C, (Qo, Ro, cno) = large_ref
    w = synth.large()
    b = gs.build_basis(cuda(C))
    X = cuda(w["X"])
    out = gs.project_similarity(b, X, path="tensor", want_S=True, want_Y=True)
    gs.stream_status()
    assert np.array_equal(out["argmax"].cpu().numpy(), w["labels"])
    rows = np.sort(np.random.default_rng(11).choice(w["N"], 768, replace=False))
    ref = orc.project_similarity(w["X"][rows], Qo, Ro, cno)
    sub = {k: out[k][torch.from_numpy(rows).to(X.device)] for k in ("S", "Y", "argmax", "maxval")}
    check_scores(sub, ref, w["X"][rows], cno)
    xn = ref["xnorm"]
    assert np.all(np.abs(host(sub["Y"]) - ref["Y"]) <= TOL_S * xn[:, None])
    # every row: the label's score against the closed form <x, c_label>, on this launch
    # and on launches back to back (a stale pipeline stage shows up as one K-block of
    # one row scored from old data, and only when launches follow each other closely)
    lab = torch.from_numpy(w["labels"]).to(X.device)
    Xd = w["X"].astype(np.float64)
    full = np.einsum("nd,nd->n", Xd, C[w["labels"]].astype(np.float64))
    bound = TOL_S * np.linalg.norm(Xd, axis=1) * np.sqrt(C.shape[1])
    outs = [out] + [gs.project_similarity(b, X, path="tensor", want_S=True) for _ in range(3)]
    gs.stream_status()
    for o in outs:
        s_lab = o["S"].gather(1, lab[:, None].long())[:, 0].double().cpu().numpy()
        assert np.all(np.abs(s_lab - full) <= bound)
        assert np.array_equal(o["argmax"].cpu().numpy(), w["labels"])


@pytest.mark.parametrize("mode,scale", [("raw", 1.0), ("raw", -0.5), ("cosine", 2.0), ("softmax", 1 / 90.0)])
def test_tc_modes(gs, orc, large_ref, mode, scale):
    C, (Qo, Ro, cno) = large_ref
    w = synth.large(rows=(1000, 5096))
    b = gs.build_basis(cuda(C))
    out = gs.project_similarity(b, cuda(w["X"]), mode=mode, scale=scale, path="tensor", want_S=True)
    gs.stream_status()
    ref = orc.project_similarity(w["X"], Qo, Ro, cno, mode=getattr(orc, mode.upper()), scale=scale)
    check_scores(out, ref, w["X"], cno, mode, scale)


@pytest.mark.parametrize("N,M,D,ld", [(1, 40, 1000, 1000), (3, 40, 1000, 1000), (1000, 40, 1000, 1000),
                                       (777, 40, 1002, 1004), (129, 256, 2048, 2048),
                                       (4099, 100, 4096, 4100)])
def test_tc_ragged(gs, orc, N, M, D, ld):
    """Ragged batches (tiles of < 128 rows), D not a multiple of the 64-wide
    K-block or of 4, r not a multiple of 16, leading dimension > D."""
    rng = np.random.default_rng(N + M + D)
    C = (rng.integers(0, 2, size=(M, D)) * 2 - 1).astype(np.float32)
    X, _ = synth.noisy_rows(C, 5, 0, N, 1.0)
    Xp = np.zeros((N, ld), np.float32)
    Xp[:, :D] = X
    Xp[:, D:] = np.nan  # padding must never be read
    b = gs.build_basis(cuda(C))
    Qo, Ro, cno = orc.build_basis(C)
    Xd = cuda(Xp)[:, :D]
    out = gs.project_similarity(b, Xd, path="tensor", want_S=True, want_Y=True)
    gs.stream_status()
    ref = orc.project_similarity(X, Qo, Ro, cno)
    check_scores(out, ref, X, cno)
    assert np.all(np.abs(host(out["Y"]) - ref["Y"]) <= TOL_S * ref["xnorm"][:, None])


def test_tc_rank_deficient(gs, orc):
    """Dependent codewords: R has rows that end early (lower echelon, r < M)."""
    rng = np.random.default_rng(8)
    ind = rng.integers(0, 2, size=(48, 3000)).astype(np.float32)
    dep = np.stack([ind[3], ind[5] - ind[7], ind[0] + ind[1], ind[47]] * 4)
    C = np.concatenate([ind[:20], dep, ind[20:]])[:64]
    C = C[rng.permutation(64)]
    b = gs.build_basis(cuda(C))
    Qo, Ro, cno = orc.build_basis(C)
    assert b.r == Qo.shape[0] < 64
    X, _ = synth.noisy_rows(C, 6, 0, 2000, 1.0)
    out = gs.project_similarity(b, cuda(X), path="tensor", want_S=True)
    gs.stream_status()
    check_scores(out, orc.project_similarity(X, Qo, Ro, cno), X, cno)


def test_tc_auto_picks_tensor_and_matches_simt(gs, large_ref):
    """The auto path and the fp32 SIMT path agree on argmax for the large batch."""
    C, _ = large_ref
    w = synth.large(rows=(0, 8192))
    b = gs.build_basis(cuda(C))
    X = cuda(w["X"])
    a = gs.project_similarity(b, X, path="auto")
    s = gs.project_similarity(b, X, path="simt")
    assert torch.equal(a["argmax"], s["argmax"])
    assert np.array_equal(a["argmax"].cpu().numpy(), w["labels"])


def test_tc_out_of_range_rows(gs, orc, large_ref):
    """An entry beyond fp16's range (1e5) no longer breaks the tensor-core path: the kernel finds
    the row from its norm and computes its tile again with an exact power-of-two scale, so the
    results meet the usual bound and the device reports nothing.  Only a row whose squared norm
    is not a finite fp32 number (an entry of 1e20) still raises GS_ERR_RANGE, and the library
    stays usable afterwards."""
    C, (Qo, Ro, cno) = large_ref
    w = synth.large(rows=(0, 256))
    b = gs.build_basis(cuda(C))
    X = cuda(w["X"])
    X[17, 3] = 1.0e5
    out = gs.project_similarity(b, X, path="tensor", want_S=True)
    gs.stream_status()
    Xh = host(X)
    check_scores(out, orc.project_similarity(Xh, host(b.Q), host(b.R), host(b.cnorm)), Xh, host(b.cnorm))
    X[17, 3] = 1.0e20
    gs.project_similarity(b, X, path="tensor")
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.stream_status()
    assert ei.value.status == gs.GS_ERR_RANGE
    X[17, 3] = 0.0
    o = gs.project_similarity(b, X, path="tensor")
    gs.stream_status()
    assert np.array_equal(o["argmax"].cpu().numpy()[:17], w["labels"][:17])


# ----------------------------------------------------------------- general tcgen05 GEMM paths
@pytest.fixture(scope="module")
def rankdef_ref(orc):
    C, rank = synth.rankdef_codebook()
    return C, orc.build_basis(C)


@pytest.mark.parametrize("mode", ["raw", "cosine", "softmax"])
def test_tc_two_gemm_rank_deficient(gs, orc, rankdef_ref, mode):
    """r = 922 > 256: Y = X Q^T (fp16) then S = Y R^T (bf16 hi/lo split) on the tensor core."""
    C, (Qo, Ro, cno) = rankdef_ref
    X, _ = synth.noisy_rows(C, synth.SEEDS["rankdef"], 0, 1500, 1.0)
    b = gs.build_basis(cuda(C))
    scale = 1.0 if mode != "softmax" else 1.0 / 100.0
    out = gs.project_similarity(b, cuda(X), mode=mode, scale=scale, path="tensor", want_S=True, want_Y=True)
    gs.stream_status()
    ref = orc.project_similarity(X, Qo, Ro, cno, mode=getattr(orc, mode.upper()), scale=scale)
    check_scores(out, ref, X, cno, mode, scale)
    assert np.all(np.abs(host(out["Y"]) - ref["Y"]) <= TOL_S * ref["xnorm"][:, None])


@pytest.mark.parametrize("M,D,N", [(600, 2048, 700), (1024, 2048, 1100), (300, 2304, 257)])
def test_tc_two_gemm_widths(gs, orc, M, D, N):
    """The projection of the two-GEMM path for r > 256 (128 x 512 tiles, two 256-column
    accumulators fed by each converted K-block): r = 600 (a second tile 88 columns wide), 1,024 (two
    full tiles) and 300 (one tile, the second accumulator 44 columns wide); N = 700, 1,100 and 257
    end in a partial row tile."""
    rng = np.random.default_rng(M + D)
    C = np.where(rng.random((M, D)) < 0.5, -1.0, 1.0).astype(np.float32)
    X, _ = synth.noisy_rows(C, 23, 0, N, 1.0)
    b = gs.build_basis(cuda(C))
    Qo, Ro, cno = orc.build_basis(C)
    assert b.r == M
    for mode in ("raw", "cosine"):
        out = gs.project_similarity(b, cuda(X), mode=mode, path="tensor", want_S=True, want_Y=True)
        gs.stream_status()
        ref = orc.project_similarity(X, Qo, Ro, cno, mode=getattr(orc, mode.upper()))
        check_scores(out, ref, X, cno, mode)
        assert np.all(np.abs(host(out["Y"]) - ref["Y"]) <= TOL_S * ref["xnorm"][:, None])


def test_tc_two_gemm_wide_codebook(gs, orc):
    """M = 300 > 256 codewords in D = 200 (rank 200 < M, Sec. 3.1's D < M case)."""
    rng = np.random.default_rng(21)
    C = (rng.integers(0, 2, size=(300, 200)) * 2 - 1).astype(np.float32)
    X, _ = synth.noisy_rows(C, 22, 0, 3000, 1.0)
    b = gs.build_basis(cuda(C))
    Qo, Ro, cno = orc.build_basis(C)
    assert b.r == Qo.shape[0] == 200
    out = gs.project_similarity(b, cuda(X), path="tensor", want_S=True)
    gs.stream_status()
    check_scores(out, orc.project_similarity(X, Qo, Ro, cno), X, cno)


def test_tc_reconstruct_round_trips(gs, orc, rankdef_ref):
    """Reconstructing R itself returns the integer codebook bit-exactly after rounding."""
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    assert np.array_equal(np.rint(gs.reconstruct(b, b.R.contiguous(), path="tensor").cpu().numpy()), t["C"])
    C, _ = rankdef_ref
    b = gs.build_basis(cuda(C))
    r4 = (b.r + 3) // 4 * 4  # 16-byte rows for the TMA loads of T
    T = torch.zeros((b.M, r4), device=b.R.device)
    T[:, :b.r] = b.R
    Xh = gs.reconstruct(b, T[:, :b.r], path="tensor")
    gs.stream_status()
    assert np.array_equal(np.rint(Xh.cpu().numpy()), C)


@pytest.mark.parametrize("N,M,D", [(777, 40, 1030), (130, 8, 1024), (4096, 256, 8192), (300, 40, 1100),
                                   (513, 64, 1030), (260, 96, 2000), (1000, 130, 1024)])
def test_tc_reconstruct_matches_oracle(gs, orc, N, M, D):
    """Reconstruction on the tensor core: CTA pairs (each staging half of every Q tile) for at
    least 256 rows and 256 columns, single CTAs otherwise (fewer rows, or outputs narrower than one
    256-column tile); a last column tile that is mostly past D, a last pair tile whose odd CTA has
    few or no rows, and a depth r below one 64-wide K-block."""
    rng = np.random.default_rng(N + D)
    C = (rng.integers(0, 2, size=(M, D)) * 2 - 1).astype(np.float32)
    b = gs.build_basis(cuda(C))
    Qo, _, _ = orc.build_basis(C)
    T = rng.standard_normal((N, b.r)).astype(np.float32) * 3.0
    Tp = torch.zeros((N, (b.r + 3) // 4 * 4), device="cuda:0")  # 16-byte rows, as the tensor path needs
    Tp[:, :b.r] = cuda(T)
    Xh = gs.reconstruct(b, Tp[:, :b.r], path="tensor")
    gs.stream_status()
    ref = orc.reconstruct(T, Qo)
    assert np.all(np.abs(host(Xh) - ref) <= 1e-4 * np.linalg.norm(T.astype(np.float64), axis=1)[:, None])


def test_tc_reconstruct_short_rows_take_fp32(gs, orc):
    """D < 1024: one fp16 rounding of T and Q would not average out over the rows of Q (error spread
    ~2^-11 ||t|| / sqrt(D)), so the tensor-core reconstruction refuses the shape and the default
    path computes it in fp32, within the bound."""
    rng = np.random.default_rng(3)
    C = (rng.integers(0, 2, size=(40, 200)) * 2 - 1).astype(np.float32)
    b = gs.build_basis(cuda(C))
    T = rng.standard_normal((300, b.r)).astype(np.float32)
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.reconstruct(b, cuda(T), path="tensor")
    assert ei.value.status == gs.GS_ERR_UNSUPPORTED
    Xh = gs.reconstruct(b, cuda(T))
    gs.stream_status()
    ref = orc.reconstruct(T, host(b.Q))
    assert np.all(np.abs(host(Xh) - ref) <= 1e-4 * np.linalg.norm(T.astype(np.float64), axis=1)[:, None])


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_tc_prob_vectorize(gs, orc, dtype):
    cases = [synth.tiny(), synth.multiattr()[2], {"C": synth.attention(B=1, L=1)["C"],
                                                   "P": synth.attention_probs(5, 3, 700, 512, 1)}]
    for t in cases:
        b = gs.build_basis(cuda(t["C"]))
        _, Ro, cno = orc.build_basis(t["C"])
        Vo = orc.prob_vectorize(t["P"], Ro)
        bound = 1e-4 * (np.abs(t["P"].astype(np.float64)) @ cno)[:, None]
        if dtype == torch.bfloat16:
            bound = bound + 2.0 ** -8 * np.abs(Vo)
        N, M = t["P"].shape
        Pp = torch.zeros((N, (M + 3) // 4 * 4), device="cuda:0")  # 16-byte rows for TMA
        Pp[:, :M] = cuda(t["P"])
        V = gs.prob_vectorize(b, Pp[:, :M], dtype=dtype, path="tensor")
        gs.stream_status()
        assert np.all(np.abs(host(V) - Vo) <= bound)


# ----------------------------------------------------------------- attention on tcgen05
@pytest.fixture(scope="module")
def attn_R(orc):
    return orc.build_basis(synth.attention(B=1, L=1)["C"])[1]


def _attn_inputs(orc, R, B, Lq, Lk, seed=5):
    """Compressed query / key vectors V = P R from the oracle, rounded to bf16."""
    Vq = orc.prob_vectorize(synth.attention_probs(seed, B, Lq, 512, 1), R).astype(np.float32)
    Vk = orc.prob_vectorize(synth.attention_probs(seed, B, Lk, 512, 2), R).astype(np.float32)
    tq = torch.from_numpy(Vq).to("cuda:0").to(torch.bfloat16).reshape(B, Lq, -1).contiguous()
    tk = torch.from_numpy(Vk).to("cuda:0").to(torch.bfloat16).reshape(B, Lk, -1).contiguous()
    return tq, tk


@pytest.mark.parametrize("B,Lq,Lk,r", [(3, 40, 40, 512), (2, 300, 700, 512), (1, 128, 256, 512),
                                        (2, 1024, 1024, 512), (2, 130, 520, 512), (1, 200, 1500, 512),
                                        (2, 257, 900, 200), (1, 64, 2100, 72), (2, 50, 301, 512),
                                        (3, 300, 512, 136)])
def test_tc_attention(gs, orc, attn_R, B, Lq, Lk, r):
    """bf16 compressed vectors, fp32 accumulation, row softmax over all keys; against
    the oracle run on the same bf16 inputs.  Lk <= 1024 (a multiple of 4) runs one pass
    with the key units of a row spread over a cluster of ceil(Lk / 256) CTAs (520: the
    last unit has an empty key half; 512: a cluster of two); longer rows and Lk = 301 run
    the two-pass kernel.
    r < 512 (the first r coordinates) leaves the last K-block partly beyond r."""
    tq, tk = _attn_inputs(orc, attn_R, B, Lq, Lk)
    if r < tq.shape[2]:
        tq, tk = tq[:, :, :r].contiguous(), tk[:, :, :r].contiguous()
    scale = 1.0 / 64.0
    A = gs.attention_scores(tq, tk, scale, path="tensor")
    L = gs.attention_scores(tq, tk, scale, apply_softmax=False, path="tensor")
    gs.stream_status()
    q64, k64 = tq.double().cpu().numpy(), tk.double().cpu().numpy()
    ref = orc.attention(q64, k64, B, Lq, Lk, scale)
    refl = orc.attention(q64, k64, B, Lq, Lk, scale, apply_softmax=False)
    assert (np.abs(host(A) - ref) / ref).max() <= 2e-2
    assert np.allclose(host(A).sum(axis=2), 1.0, atol=1e-4)
    assert np.abs(host(L) - refl).max() <= 1e-4 * np.abs(refl).max()


@pytest.mark.parametrize("M,D", [(256, 1024), (256, 2048), (256, 4096), (100, 1024), (40, 8192), (200, 6000)])
@pytest.mark.parametrize("outputs", ["lookup", "all"])
def test_tc_score_paths(gs, orc, M, D, outputs):
    """The fused kernel across basis sizes (full 256 x 256 TMEM accumulators down to codebooks that
    are not multiples of 16 or 32) and depths, with argmax / maxval only (the lookup kernel) and
    with every output, two launches back to back, against the oracle."""
    rng = np.random.default_rng(M * 7 + D)
    C = (rng.integers(0, 2, size=(M, D)) * 2 - 1).astype(np.float32)
    X, labels = synth.noisy_rows(C, 9, 0, 3000, 1.0)
    b = gs.build_basis(cuda(C))
    Qo, Ro, cno = orc.build_basis(C)
    full = outputs == "all"
    outs = [gs.project_similarity(b, cuda(X), path="tensor", want_S=full, want_Y=full) for _ in range(2)]
    gs.stream_status()
    ref = orc.project_similarity(X, Qo, Ro, cno)
    for out in outs:
        check_scores(out, ref, X, cno)
        if full:
            assert np.all(np.abs(host(out["Y"]) - ref["Y"]) <= TOL_S * ref["xnorm"][:, None])
    assert torch.equal(outs[0]["argmax"], outs[1]["argmax"])


@pytest.mark.parametrize("mode", ["raw", "cosine"])
def test_tc_two_gemm_argmax_without_scores(gs, orc, rankdef_ref, mode):
    """Argmax / maxval without S on the two-GEMM path (the call the bench times: the scores go to
    the handle's scratch and a row reduction reads them back).  Identical to the call that writes S
    (duplicate codewords tie exactly: lowest index; a row of NaN queries: index 0
    either way, with maxval -FLT_MAX for raw scores, none of which is a number, and 0 for cosine
    scores, which a norm that is not a number sends to 0), and within the bound of the oracle."""
    C, (Qo, Ro, cno) = rankdef_ref
    X, _ = synth.noisy_rows(C, synth.SEEDS["rankdef"], 0, 3000, 1.0)
    X[5] = np.nan
    b = gs.build_basis(cuda(C))
    Xd = cuda(X)
    only = gs.project_similarity(b, Xd, mode=mode, path="tensor")
    withS = gs.project_similarity(b, Xd, mode=mode, path="tensor", want_S=True)
    gs.stream_status()
    assert torch.equal(only["argmax"], withS["argmax"])
    assert torch.equal(only["maxval"], withS["maxval"])
    nan_row_max = -np.finfo(np.float32).max if mode == "raw" else 0.0
    assert int(only["argmax"][5]) == 0 and float(only["maxval"][5]) == nan_row_max
    keep = np.arange(3000) != 5
    ref = orc.project_similarity(X[keep], Qo, Ro, cno, mode=getattr(orc, mode.upper()))
    idx = torch.from_numpy(np.nonzero(keep)[0]).to(Xd.device)
    check_scores({k: only[k][idx] for k in ("argmax", "maxval")}, ref, X[keep], cno, mode)


def test_tc_two_gemm_argmax_two_codewords(gs, orc):
    """Two codewords in D = 512 (the split two-GEMM path, D < 1024), argmax / maxval only: the
    smallest score rows the scratch holds, identical to the call that writes S and within the
    bound of the oracle."""
    rng = np.random.default_rng(31)
    C = (rng.integers(0, 2, size=(2, 512)) * 2 - 1).astype(np.float32)
    X, _ = synth.noisy_rows(C, 32, 0, 5000, 1.0)
    b = gs.build_basis(cuda(C))
    only = gs.project_similarity(b, cuda(X), path="tensor")
    withS = gs.project_similarity(b, cuda(X), path="tensor", want_S=True)
    gs.stream_status()
    assert torch.equal(only["argmax"], withS["argmax"]) and torch.equal(only["maxval"], withS["maxval"])
    Qo, Ro, cno = orc.build_basis(C)
    check_scores(only, orc.project_similarity(X, Qo, Ro, cno), X, cno)
