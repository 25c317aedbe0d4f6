"""GPU parity: the CUDA path (through the C ABI) against the float64 oracle.

Tolerances (fp32 paths): |S - S*| <= 1e-4 ||x|| ||c_i|| elementwise and
||Q Q^T - I||_max <= 1e-5; Y within 1e-4 ||x||; V within 1e-4 sum_i |p_i| ||c_i||
(fp32) or additionally 2^-8 |V*| (bf16 output); Xhat within 1e-4 ||t||;
attention with bf16 inputs within relative 2e-2.  argmax is compared bit-exact
wherever the oracle's top-2 margin exceeds twice the score tolerance; elsewhere
the GPU's choice must score within tolerance of the maximum.
"""
import math

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

TOL_S = 1e-4
DEV = "cuda:0"


def cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def host(t):
    return t.double().cpu().numpy()


@pytest.fixture(scope="session")
def oracle_cache(orc):
    cache = {}

    def get(name, C):
        if name not in cache:
            cache[name] = orc.build_basis(C)
        return cache[name]
    return get


def check_build(b, C, Qo, Ro, cno):
    assert b.r == Qo.shape[0]
    Q = host(b.Q)
    R = host(b.R)
    assert np.abs(Q @ Q.T - np.eye(b.r)).max() <= 1e-5
    assert np.abs(Q - Qo).max() <= 1e-5
    assert np.all(np.abs(R - Ro).max(axis=1) <= 1e-5 * np.maximum(cno, 1.0))
    assert np.allclose(host(b.cnorm), cno, rtol=1e-6)
    Cd = C.astype(np.float64)
    assert np.all(np.abs(R @ Q - Cd).max(axis=1) <= 1e-5 * np.maximum(cno, 1.0))


def check_scores(out, ref, X, cno, mode="raw", scale=1.0):
    xn = np.linalg.norm(X.astype(np.float64), axis=1)
    if mode == "raw":
        bound = TOL_S * abs(scale) * xn[:, None] * cno[None, :]
    elif mode == "cosine":
        bound = np.full(ref["S"].shape, TOL_S * abs(scale))
    else:
        # a logit error of at most d moves each probability p by at most p (e^(2d) - 1);
        # d is the raw-score bound times the scale
        d = TOL_S * abs(scale) * xn[:, None] * cno.max()
        bound = ref["S"] * np.expm1(2 * d) + 1e-9
    if "S" in out:
        assert np.all(np.abs(host(out["S"]) - ref["S"]) <= bound + 1e-12)
    if "maxval" in out:
        mv = ref["S"][np.arange(len(xn)), ref["argmax"]]
        assert np.all(np.abs(host(out["maxval"]) - mv) <= bound.max(axis=1) + 1e-12)
    if "argmax" in out:
        am = out["argmax"].cpu().numpy().astype(np.int64)
        Ss = np.sort(ref["S"], axis=1)
        margin = Ss[:, -1] - Ss[:, -2] if ref["S"].shape[1] > 1 else np.full(len(xn), np.inf)
        sure = margin > 2 * bound.max(axis=1)
        assert np.array_equal(am[sure], ref["argmax"][sure])
        picked = ref["S"][np.arange(len(xn)), am]
        assert np.all(picked >= Ss[:, -1] - 2 * bound.max(axis=1) - 1e-12)


# ----------------------------------------------------------------- build
def test_build_tiny_and_multiattr(gs, orc):
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    check_build(b, t["C"], *orc.build_basis(t["C"]))
    for a in synth.multiattr():
        b = gs.build_basis(cuda(a["C"]))
        check_build(b, a["C"], *orc.build_basis(a["C"]))


def test_build_large_and_attention_codebooks(gs, oracle_cache):
    C = synth.large_codebook()
    check_build(gs.build_basis(cuda(C)), C, *oracle_cache("large", C))
    Ca = synth.attention(B=1, L=1)["C"]
    check_build(gs.build_basis(cuda(Ca)), Ca, *oracle_cache("attn", Ca))


def test_build_rank_deficient_full_size(gs, oracle_cache):
    C, rank = synth.rankdef_codebook()
    Qo, Ro, cno = oracle_cache("rankdef", C)
    b = gs.build_basis(cuda(C))
    assert b.r == rank == 922
    check_build(b, C, Qo, Ro, cno)
    # exact reconstruction of the binary / integer codebook (Sec. 3.2, Table 4)
    Xh = gs.reconstruct(b, b.R, path="simt")
    assert np.array_equal(np.rint(Xh.cpu().numpy()), C)


@pytest.mark.parametrize("M,D", [(1, 7), (5, 3), (33, 1000), (40, 256), (17, 4099)])
def test_build_ragged_shapes(gs, orc, M, D):
    rng = np.random.default_rng(M * 1000 + D)
    C = (rng.integers(0, 2, size=(M, D)) * 2 - 1).astype(np.float32)
    if M > 4:
        C[3] = C[1] - C[2]  # a dependent row
        C[4] = 0.0          # a zero row
    b = gs.build_basis(cuda(C))
    check_build(b, C, *orc.build_basis(C))


def test_build_zero_codebook_and_normalize(gs, orc):
    b = gs.build_basis(cuda(np.zeros((6, 64), np.float32)))
    assert b.r == 0
    X = cuda(np.ones((5, 64), np.float32))
    o = gs.project_similarity(b, X, want_S=True)
    assert torch.all(o["S"] == 0) and torch.all(o["argmax"] == 0)
    o = gs.project_similarity(b, X, mode="softmax", want_S=True)
    assert torch.allclose(o["S"], torch.full_like(o["S"], 1 / 6))
    C = synth.tiny()["C"] * np.arange(1, 9, dtype=np.float32)[:, None]
    b = gs.build_basis(cuda(C), normalize_rows=True)
    check_build(b, C / np.linalg.norm(C, axis=1, keepdims=True), *orc.build_basis(C, normalize_rows=True))


# ----------------------------------------------------------------- project + similarity
@pytest.mark.parametrize("mode,scale", [("raw", 1.0), ("raw", 0.25), ("cosine", 1.0), ("softmax", 1 / 32)])
@pytest.mark.parametrize("path", ["auto", "simt"])
def test_similarity_tiny(gs, orc, mode, scale, path):
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Qo, Ro, cno = orc.build_basis(t["C"])
    out = gs.project_similarity(b, cuda(t["X"]), mode=mode, scale=scale, path=path, want_Y=True, want_S=True)
    ref = orc.project_similarity(t["X"], Qo, Ro, cno, mode=getattr(orc, mode.upper()), scale=scale)
    xn = np.linalg.norm(t["X"].astype(np.float64), axis=1)
    assert np.all(np.abs(host(out["Y"]) - ref["Y"]) <= TOL_S * xn[:, None])
    check_scores(out, ref, t["X"], cno, mode, scale)
    assert np.array_equal(out["argmax"].cpu().numpy(), t["labels"])


def test_similarity_multiattr(gs, orc):
    for a in synth.multiattr():
        b = gs.build_basis(cuda(a["C"]))
        Qo, Ro, cno = orc.build_basis(a["C"])
        for mode in ("raw", "cosine", "softmax"):
            out = gs.project_similarity(b, cuda(a["X"]), mode=mode, want_S=True)
            ref = orc.project_similarity(a["X"], Qo, Ro, cno, mode=getattr(orc, mode.upper()))
            check_scores(out, ref, a["X"], cno, mode)


def test_similarity_generic_path_large_r(gs, oracle_cache):
    """r > 32 takes the chunked GEMM path: attention codebook (r = 512)."""
    a = synth.attention(B=1, L=1)
    Qo, Ro, cno = oracle_cache("attn", a["C"])
    X, _ = synth.noisy_rows(a["C"], 99, 0, 700, 1.0)
    b = gs.build_basis(cuda(a["C"]))
    for mode in ("raw", "cosine", "softmax"):
        out = gs.project_similarity(b, cuda(X), mode=mode, path="simt", want_S=True, want_Y=True)
        ref = __import__("oracle.oracle", fromlist=["x"]).project_similarity(
            X, Qo, Ro, cno, mode={"raw": 0, "cosine": 1, "softmax": 2}[mode])
        check_scores(out, ref, X, cno, mode)


def test_similarity_large_full_size(gs, orc, oracle_cache):
    """65,536 x 8192 queries: argmax of every row equals its generating label;
    scores and Gram-loc of a seeded sample of rows match the oracle."""
    w = synth.large()
    Qo, Ro, cno = oracle_cache("large", w["C"])
    b = gs.build_basis(cuda(w["C"]))
    X = cuda(w["X"])
    out = gs.project_similarity(b, X)
    assert np.array_equal(out["argmax"].cpu().numpy(), w["labels"])
    rows = np.sort(np.random.default_rng(3).choice(w["N"], 512, replace=False))
    o2 = gs.project_similarity(b, X[torch.from_numpy(rows).to(DEV)], want_S=True, want_Y=True)
    ref = orc.project_similarity(w["X"][rows], Qo, Ro, cno)
    check_scores(o2, ref, w["X"][rows], cno)
    mv = host(out["maxval"])[rows]
    assert np.all(np.abs(mv - ref["maxval"]) <= TOL_S * ref["xnorm"] * cno.max())


def test_similarity_rankdef_sample(gs, orc, oracle_cache):
    C, _ = synth.rankdef_codebook()
    Qo, Ro, cno = oracle_cache("rankdef", C)
    X, L = synth.noisy_rows(C, synth.SEEDS["rankdef"], 0, 1024, 1.0)
    b = gs.build_basis(cuda(C))
    out = gs.project_similarity(b, cuda(X), want_S=True, want_Y=True)
    ref = orc.project_similarity(X, Qo, Ro, cno)
    check_scores(out, ref, X, cno)
    xn = np.linalg.norm(X.astype(np.float64), axis=1)
    assert np.all(np.abs(host(out["Y"]) - ref["Y"]) <= TOL_S * xn[:, None])


# ----------------------------------------------------------------- prob-vectorize
def test_prob_vectorize_tiny_multiattr(gs, orc):
    cases = [synth.tiny()] + synth.multiattr()
    for t in cases:
        b = gs.build_basis(cuda(t["C"]))
        _, Ro, cno = orc.build_basis(t["C"])
        Vo = orc.prob_vectorize(t["P"], Ro)
        bound = 1e-4 * (np.abs(t["P"].astype(np.float64)) @ cno)[:, None]
        V = gs.prob_vectorize(b, cuda(t["P"]))
        assert np.all(np.abs(host(V) - Vo) <= bound)
        Vb = gs.prob_vectorize(b, cuda(t["P"]), dtype=torch.bfloat16)
        assert np.all(np.abs(host(Vb) - Vo) <= bound + 2.0 ** -8 * np.abs(Vo))


# ----------------------------------------------------------------- reconstruct
def test_reconstruct_tiny(gs, orc):
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Qo, Ro, _ = orc.build_basis(t["C"])
    assert np.array_equal(np.rint(gs.reconstruct(b, b.R).cpu().numpy()), t["C"])
    T = np.random.default_rng(4).standard_normal((37, b.r)).astype(np.float32)
    Xh = gs.reconstruct(b, cuda(T))
    ref = orc.reconstruct(T, Qo)
    assert np.all(np.abs(host(Xh) - ref) <= 1e-4 * np.linalg.norm(T.astype(np.float64), axis=1)[:, None])
    Tb = torch.from_numpy(T).to(DEV).to(torch.bfloat16)
    Xb = gs.reconstruct(b, Tb)
    refb = orc.reconstruct(Tb.float().cpu().numpy(), Qo)
    assert np.all(np.abs(host(Xb) - refb) <= 1e-4 * np.linalg.norm(T.astype(np.float64), axis=1)[:, None])


def test_reconstruct_projector_round_trip(gs, orc):
    """reconstruct(project(x)) is the projection of x onto span(C) (Eq. 4)."""
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Qo, _, _ = orc.build_basis(t["C"])
    Y = gs.project_similarity(b, cuda(t["X"]), want_Y=True, want_argmax=False, want_maxval=False)["Y"]
    Xp = gs.reconstruct(b, Y)
    Yo, _ = orc.project(t["X"], Qo)
    ref = orc.reconstruct(Yo, Qo)
    assert np.all(np.abs(host(Xp) - ref) <= 1e-4 * np.linalg.norm(t["X"].astype(np.float64), axis=1)[:, None])


# ----------------------------------------------------------------- attention
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_attention_small(gs, orc, oracle_cache, dtype):
    a = synth.attention(B=3, L=40)
    _, Ro, _ = oracle_cache("attn", a["C"])
    Vq = orc.prob_vectorize(a["Pq"], Ro)
    Vk = orc.prob_vectorize(a["Pk"], Ro)
    tq = torch.from_numpy(Vq.astype(np.float32)).to(DEV).to(dtype).reshape(3, 40, -1).contiguous()
    tk = torch.from_numpy(Vk.astype(np.float32)).to(DEV).to(dtype).reshape(3, 40, -1).contiguous()
    scale = 1.0 / math.sqrt(a["D"])
    A = gs.attention_scores(tq, tk, scale)
    ref = orc.attention(tq.double().cpu().numpy(), tk.double().cpu().numpy(), 3, 40, 40, scale)
    rel = np.abs(host(A) - ref) / ref
    assert rel.max() <= (1e-4 if dtype == torch.float32 else 2e-2)
    L = gs.attention_scores(tq, tk, scale, apply_softmax=False)
    refl = orc.attention(tq.double().cpu().numpy(), tk.double().cpu().numpy(), 3, 40, 40, scale, False)
    assert np.abs(host(L) - refl).max() <= 1e-4 * np.abs(refl).max()


def test_attention_full_size_sampled(gs, orc, oracle_cache):
    """64 x 1024 tokens, r = 512: prob-vectorize to bf16 on the GPU, attention
    scores + softmax; rows of two sequences against the float64 oracle run
    end to end from the probabilities (bf16 tolerance 2e-2)."""
    a = synth.attention()
    B, L, D = a["B"], a["L"], a["D"]
    _, Ro, _ = oracle_cache("attn", a["C"])
    b = gs.build_basis(cuda(a["C"]))
    Vq = gs.prob_vectorize(b, cuda(a["Pq"]), dtype=torch.bfloat16).reshape(B, L, -1)
    Vk = gs.prob_vectorize(b, cuda(a["Pk"]), dtype=torch.bfloat16).reshape(B, L, -1)
    scale = 1.0 / math.sqrt(D)
    A = gs.attention_scores(Vq.contiguous(), Vk.contiguous(), scale)
    for bb in (0, B - 1):
        rows = slice(bb * L, (bb + 1) * L)
        q = orc.prob_vectorize(a["Pq"][rows][:64], Ro)
        k = orc.prob_vectorize(a["Pk"][rows], Ro)
        ref = orc.attention(q, k, 1, 64, L, scale)[0]
        got = host(A[bb, :64])
        assert (np.abs(got - ref) / ref).max() <= 2e-2
        assert np.allclose(got.sum(axis=1), 1.0, atol=1e-4)


# ----------------------------------------------------------------- edge cases / errors
def test_empty_and_argument_errors(gs):
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    e = torch.empty((0, 1024), device=DEV)
    o = gs.project_similarity(b, e)
    assert o["argmax"].numel() == 0
    assert gs.prob_vectorize(b, torch.empty((0, 8), device=DEV)).shape == (0, 8)
    assert gs.reconstruct(b, torch.empty((0, 8), device=DEV)).shape == (0, 1024)
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.project_similarity(b, cuda(t["X"][:, :512]))
    assert ei.value.status == gs.GS_ERR_SHAPE
    with pytest.raises(gs.GramSpaceError):
        gs.project_similarity(b, cuda(t["X"]), want_argmax=False, want_maxval=False)
    gs.stream_status()


def test_strided_inputs(gs, orc):
    """Leading dimensions larger than the row length."""
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Qo, Ro, cno = orc.build_basis(t["C"])
    big = torch.zeros((64, 1100), device=DEV)
    big[:, :1024] = cuda(t["X"])
    out = gs.project_similarity(b, big[:, :1024], want_S=True)
    ref = orc.project_similarity(t["X"], Qo, Ro, cno)
    check_scores(out, ref, t["X"], cno)


def test_reconstruct_multiattr(gs, orc):
    """The multi-attribute workload's reconstruct step: each attribute's prob-vectorized rows
    V = P R (512 per attribute) back to D = 1024, against the oracle's reconstruction with the
    GPU's basis (1e-4 ||v||) and against the basis-free P C (1e-4 sum_i |p_i| ||c_i||)."""
    for a in synth.multiattr():
        b = gs.build_basis(cuda(a["C"]))
        V = gs.prob_vectorize(b, cuda(a["P"]))
        Xh = gs.reconstruct(b, V)
        gs.stream_status()
        Vh = host(V)
        ref = orc.reconstruct(Vh, host(b.Q))
        assert np.all(np.abs(host(Xh) - ref) <= 1e-4 * np.linalg.norm(Vh, axis=1)[:, None])
        P = a["P"].astype(np.float64)
        cn = np.linalg.norm(a["C"].astype(np.float64), axis=1)
        PC = P @ a["C"].astype(np.float64)
        assert np.all(np.abs(host(Xh) - PC) <= 1e-4 * (np.abs(P) @ cn)[:, None])
