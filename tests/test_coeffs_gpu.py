"""GPU parity of gs_similarity_coeffs: scores of queries given by their Gram-loc
coordinates (Sec. 3.2, Eq. 2), S = Y R^T with the row epilogues, against the
float64 oracle's similarity on the same Y.

Bound: |S - S*| <= 1e-4 ||y|| ||c_i|| elementwise (raw; ||y|| = ||x|| for x in the
span), 1e-4 for cosine, and the derived softmax bound; argmax bit-exact wherever
the oracle's top-2 margin exceeds twice the bound, otherwise within the bound of
the maximum.  Both paths (fp32 CUDA cores, tcgen05 with bf16 hi / lo split) run.
"""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

TOL = 1e-4
DEV = "cuda:0"
MODES = ("raw", "cosine", "softmax")


def cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def host(t):
    return t.double().cpu().numpy()


def reference(orc, Y, Ro, cno, mode, scale):
    yn = np.linalg.norm(Y, axis=1)
    S, am, mv = orc.similarity(Y, Ro, getattr(orc, mode.upper()), scale, yn, cno)
    return S, am, yn


def check(out, S_ref, am_ref, yn, cno, mode, scale):
    if mode == "raw":
        bound = TOL * abs(scale) * yn[:, None] * cno[None, :]
    elif mode == "cosine":
        bound = np.full(S_ref.shape, TOL * abs(scale))
    else:
        d = TOL * abs(scale) * yn[:, None] * cno.max()
        bound = S_ref * np.expm1(2 * d) + 1e-9
    if "S" in out:
        assert np.all(np.abs(host(out["S"]) - S_ref) <= bound + 1e-12)
    n = len(yn)
    if "maxval" in out:
        assert np.all(np.abs(host(out["maxval"]) - S_ref[np.arange(n), am_ref]) <= bound.max(axis=1) + 1e-12)
    am = out["argmax"].cpu().numpy().astype(np.int64)
    Ss = np.sort(S_ref, axis=1)
    margin = Ss[:, -1] - Ss[:, -2] if S_ref.shape[1] > 1 else np.full(n, np.inf)
    sure = margin > 2 * bound.max(axis=1)
    assert np.array_equal(am[sure], am_ref[sure])
    assert np.all(S_ref[np.arange(n), am] >= Ss[:, -1] - 2 * bound.max(axis=1) - 1e-12)


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("path", ["auto", "simt"])
def test_tiny_gramloc_queries(gs, orc, mode, path):
    """Gram-loc of noisy queries (oracle projection) and of probability mixes (V = P R)."""
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Qo, Ro, cno = orc.build_basis(t["C"])
    Yx, _ = orc.project(t["X"], Qo)
    for Y in (Yx, orc.prob_vectorize(t["P"], Ro)):
        out = gs.similarity_coeffs(b, cuda(Y.astype(np.float32)), mode=mode, scale=0.5, path=path, want_S=True)
        S, am, yn = reference(orc, Y.astype(np.float32).astype(np.float64), Ro, cno, mode, 0.5)
        check(out, S, am, yn, cno, mode, 0.5)
    # projected noisy codewords still point at their codeword
    out = gs.similarity_coeffs(b, cuda(Yx.astype(np.float32)), path=path)
    assert np.array_equal(out["argmax"].cpu().numpy(), t["labels"])


def test_multiattr_matches_project_similarity(gs, orc):
    """The same scores whether the query arrives as x (D-dim) or as its Gram-loc y = x Q^T."""
    for a in synth.multiattr():
        b = gs.build_basis(cuda(a["C"]))
        X = cuda(a["X"])
        full = gs.project_similarity(b, X, want_Y=True, want_S=True)
        out = gs.similarity_coeffs(b, full["Y"], want_S=True)
        xn = np.linalg.norm(a["X"].astype(np.float64), axis=1)
        cno = host(b.cnorm)
        assert np.all(np.abs(host(out["S"]) - host(full["S"])) <= TOL * xn[:, None] * cno[None, :])


@pytest.mark.parametrize("mode", MODES)
def test_tensor_path_attention_codebook(gs, orc, oracle_cache_coeffs, mode):
    """r = 512, M = 512, 2,000 rows (ragged last tile) on the tcgen05 path."""
    a = synth.attention(B=1, L=2000)
    Qo, Ro, cno = oracle_cache_coeffs("attn", a["C"])
    b = gs.build_basis(cuda(a["C"]))
    Y = orc.prob_vectorize(a["Pq"], Ro).astype(np.float32)
    out = gs.similarity_coeffs(b, cuda(Y), mode=mode, scale=1 / 64.0, path="tensor", want_S=True)
    S, am, yn = reference(orc, Y.astype(np.float64), Ro, cno, mode, 1 / 64.0)
    check(out, S, am, yn, cno, mode, 1 / 64.0)


@pytest.mark.parametrize("path", ["tensor", "simt"])
def test_rank_deficient_codebook(gs, orc, oracle_cache_coeffs, path):
    """r = 922 < M = 1024 (duplicate rows tie exactly; the margin rule handles them)."""
    C, _ = synth.rankdef_codebook()
    Qo, Ro, cno = oracle_cache_coeffs("rankdef", C)
    b = gs.build_basis(cuda(C))
    X, _ = synth.noisy_rows(C, synth.SEEDS["rankdef"], 0, 700, 1.0)
    Y, _ = orc.project(X, Qo)
    Y = Y.astype(np.float32)
    # rows padded to 924 floats: the tensor-core path needs 16-byte row strides
    Yd = torch.zeros((Y.shape[0], (Y.shape[1] + 3) // 4 * 4), dtype=torch.float32, device=DEV)
    Yd[:, :Y.shape[1]] = cuda(Y)
    out = gs.similarity_coeffs(b, Yd[:, :Y.shape[1]], path=path, want_S=True)
    S, am, yn = reference(orc, Y.astype(np.float64), Ro, cno, "raw", 1.0)
    check(out, S, am, yn, cno, "raw", 1.0)


def test_edges_and_errors(gs, orc):
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Y = torch.zeros((0, b.r), dtype=torch.float32, device=DEV)
    out = gs.similarity_coeffs(b, Y)                     # N = 0: no-op
    assert out["argmax"].numel() == 0
    # strided Y (ld > r) on the CUDA-core path
    big = torch.randn(64, b.r + 5, device=DEV)
    Ys = big[:, :b.r]
    o1 = gs.similarity_coeffs(b, Ys, want_S=True)
    o2 = gs.similarity_coeffs(b, Ys.contiguous(), want_S=True)
    assert torch.equal(o1["S"], o2["S"])
    # a forced tensor path with a misaligned row stride is refused, not silently rerouted
    with pytest.raises(gs.GramSpaceError) as e:
        gs.similarity_coeffs(b, Ys, path="tensor")
    assert e.value.status == gs.GS_ERR_ALIGNMENT
    # zero codebook: r = 0, every score 0, argmax 0, softmax uniform
    z = gs.build_basis(torch.zeros((5, 64), device=DEV))
    assert z.r == 0
    Y0 = torch.zeros((7, 0), dtype=torch.float32, device=DEV)
    o = gs.similarity_coeffs(z, Y0, mode="softmax", want_S=True)
    assert torch.allclose(o["S"], torch.full((7, 5), 0.2, device=DEV))
    assert torch.equal(o["argmax"].cpu(), torch.zeros(7, dtype=torch.int32))
    gs.stream_status()


@pytest.fixture(scope="module")
def oracle_cache_coeffs(orc):
    cache = {}

    def get(name, C):
        if name not in cache:
            cache[name] = orc.build_basis(C)
        return cache[name]
    return get
