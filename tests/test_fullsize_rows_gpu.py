"""GPU parity of the bench's side rows at their full sizes, in the launch configuration the bench
times: every output computed, a seeded sample of rows checked against the oracle run with the
GPU's own basis (so only the kernels' arithmetic differs), bounds as in the other parity tests:
X̂ within 1e-4 ||t|| (fp16 tensor-core reconstruction), V within 1e-4 sum_i |p_i| ||c_i|| +
2^-8 |V*| (bf16 output), binding within the spectral method's bound plus the reconstruction error carried
through the block (see test_bind_gpu).
"""
import numpy as np
import pytest
import torch

import synth
from test_bind_gpu import check_bind
from test_parity_gpu import check_scores, cuda, host

pytestmark = pytest.mark.gpu


def sample_rows(n, k, seed):
    return np.sort(np.random.default_rng(seed).choice(n, k, replace=False))


def test_reconstruct_rankdef_full_size(gs, orc):
    """16,384 x 922 coefficients -> 16,384 x 10,000 (the bench's reconstruct row)."""
    C4, _ = synth.rankdef_codebook()
    b = gs.build_basis(cuda(C4))
    r4 = (b.r + 3) // 4 * 4
    g = torch.Generator().manual_seed(17)
    T = torch.randn(16384, r4, generator=g).to("cuda:0")[:, :b.r]
    Xh = gs.reconstruct(b, T)
    gs.stream_status()
    rows = sample_rows(16384, 64, 1)
    Tr = host(T[torch.from_numpy(rows).to(T.device)])
    ref = orc.reconstruct(Tr, host(b.Q))
    got = host(Xh[torch.from_numpy(rows).to(T.device)])
    bound = 1e-4 * np.linalg.norm(Tr, axis=1)
    assert np.all(np.abs(got - ref).max(axis=1) <= bound)


def test_prob_vectorize_attention_full_size(gs, orc):
    """65,536 x 512 probabilities -> bf16 Gram-loc rows (the bench's prob-vectorize row)."""
    a = synth.attention()
    b = gs.build_basis(cuda(a["C"]))
    V = gs.prob_vectorize(b, cuda(a["Pq"]), dtype=torch.bfloat16)
    gs.stream_status()
    rows = sample_rows(a["Pq"].shape[0], 256, 2)
    P = a["Pq"][rows].astype(np.float64)
    R = host(b.R)
    ref = P @ R
    got = host(V[torch.from_numpy(rows).to(V.device)])
    cn = np.linalg.norm(R, axis=1)
    bound = 1e-4 * (np.abs(P) @ cn)[:, None] + 2.0 ** -8 * np.abs(ref)
    assert np.all(np.abs(got - ref) <= bound)


def test_reconstruct_bind_full_size(gs, orc):
    """8,192 rows of the attention basis bound with per-row partners in blocks of 256 (the bench's
    reconstruct + bind row)."""
    a = synth.attention(B=1, L=1)
    b = gs.build_basis(cuda(a["C"]))
    N, L = 8192, 256
    P = synth.attention_probs(12, 1, N, b.M, 1)
    T = (torch.from_numpy(P).to("cuda:0") @ b.R).contiguous()
    g = torch.Generator().manual_seed(19)
    Y = torch.randn(N, b.D, generator=g).to("cuda:0")
    Z = gs.reconstruct_bind(b, T, Y, L)
    gs.stream_status()
    rows = sample_rows(N, 32, 3)
    idx = torch.from_numpy(rows).to(T.device)
    Tr, Yr = host(T[idx]), host(Y[idx])
    Xo = orc.reconstruct(Tr, host(b.Q))
    Zo = orc.bind(Xo, Yr, L)
    check_bind(Z[idx], Zo, Xo, Yr, L, e_rec=1e-4 * np.linalg.norm(Tr, axis=1), method="spectral")


def test_reconstruct_bind_one_partner_full_size(gs, orc):
    """8,192 rows of the attention basis bound with one partner row in blocks of 256 (the bench's
    one-partner reconstruct + bind: the basis rows bound once, one reconstruction GEMM), sampled
    rows against the oracle's reconstruction followed by binding."""
    from test_bind_gpu import one_partner_bound
    a = synth.attention(B=1, L=1)
    b = gs.build_basis(cuda(a["C"]))
    N, L = 8192, 256
    P = synth.attention_probs(12, 1, N, b.M, 1)
    T = (torch.from_numpy(P).to("cuda:0") @ b.R).contiguous()
    g = torch.Generator().manual_seed(29)
    Y = torch.randn(1, b.D, generator=g).to("cuda:0")
    Z = gs.reconstruct_bind(b, T, Y, L)
    gs.stream_status()
    rows = sample_rows(N, 64, 6)
    idx = torch.from_numpy(rows).to(T.device)
    Tr, Yh, Qh = host(T[idx]), host(Y), host(b.Q)
    Zo = orc.reconstruct_bind(Tr, Qh, Yh, L)
    err = np.abs(host(Z[idx]) - Zo).reshape(len(rows), b.D // L, L).max(axis=2)
    assert np.all(err <= one_partner_bound(Tr, Qh, Yh, L, "spectral", "tensor"))


def test_bind_one_partner_full_size(gs, orc):
    """8,192 x 4,096 rows bound with one partner row in blocks of 256 (the bench's one-partner
    binding: the partner's block spectra cached per CTA), sampled rows against the oracle."""
    g = torch.Generator().manual_seed(23)
    X = torch.randn(8192, 4096, generator=g).to("cuda:0")
    Y = torch.randn(1, 4096, generator=g).to("cuda:0")
    Z = gs.bind(X, Y, 256)
    gs.stream_status()
    rows = sample_rows(8192, 32, 4)
    Xr = host(X[torch.from_numpy(rows).to(X.device)])
    Yh = host(Y)
    Zo = orc.bind(Xr, Yh, 256)
    check_bind(Z[torch.from_numpy(rows).to(X.device)], Zo, Xr, Yh, 256, method="spectral")


def test_project_similarity_rankdef_full_size(gs, orc):
    """All 16,384 rank-deficient queries (r = 922, M = 1,024) on the tensor-core path the bench
    times, three launches back to back (so every persistent CTA runs several tiles, and a stage
    left stale by the previous launch would show): the launches agree bit for bit; Y and S of a
    seeded sample of rows match the oracle run with the GPU's basis; every row's score at its
    generating codeword is within the bound of <x, c_label> computed from the codebook itself."""
    C, _ = synth.rankdef_codebook()
    b = gs.build_basis(cuda(C))
    X, labels = synth.noisy_rows(C, synth.SEEDS["rankdef"], 0, 16384, 1.0)
    Xd = cuda(X)
    outs = [gs.project_similarity(b, Xd, path="tensor", want_S=True, want_Y=True) for _ in range(3)]
    gs.stream_status()
    for o in outs[1:]:
        for k in ("Y", "S", "argmax", "maxval"):
            assert torch.equal(o[k], outs[0][k]), k
    out = outs[-1]
    rows = sample_rows(16384, 256, 5)
    idx = torch.from_numpy(rows).to(Xd.device)
    Qh, Rh, cn = host(b.Q), host(b.R), host(b.cnorm)
    ref = orc.project_similarity(X[rows], Qh, Rh, cn)
    xn = ref["xnorm"]
    assert np.all(np.abs(host(out["Y"][idx]) - ref["Y"]) <= 1e-4 * xn[:, None])
    sub = {k: out[k][idx] for k in ("S", "argmax", "maxval")}
    check_scores(sub, ref, X[rows], cn)
    # every row: S[n, label_n] against <x_n, c_label_n> (plain float64 dot products with C)
    S_lab = host(out["S"].gather(1, torch.from_numpy(labels).to(Xd.device)[:, None]))[:, 0]
    for i0 in range(0, 16384, 2048):
        Xi = X[i0:i0 + 2048].astype(np.float64)
        Ci = C[labels[i0:i0 + 2048]].astype(np.float64)
        exact = np.einsum("ij,ij->i", Xi, Ci)
        bound = 1e-4 * np.linalg.norm(Xi, axis=1) * np.linalg.norm(Ci, axis=1)
        assert np.all(np.abs(S_lab[i0:i0 + 2048] - exact) <= bound)
