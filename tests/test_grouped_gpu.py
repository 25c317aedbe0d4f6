"""GPU parity of grouped bases (gs_build_basis_grouped, gs_group_argmax) against the oracle.

Bars as for single bases: each group's Q_g within 1e-5 of the oracle's and Q_g Q_g^T = I
within 1e-5; R within 1e-5 ||c_i|| and exactly zero outside its block; scores within
1e-4 ||x|| ||c_i||; per-group argmax bit-exact wherever the oracle's top-2 margin within
the group exceeds twice the score tolerance, elsewhere scoring within tolerance of the
group's maximum.
"""
import numpy as np
import pytest
import torch

import synth
from test_parity_gpu import TOL_S, cuda, host

pytestmark = pytest.mark.gpu


def check_grouped_build(gs, b, C, off, orc):
    Qo, Ro, cno, coeff = orc.build_grouped(C, off)
    rows, coeffs = gs.basis_groups(b)
    assert rows == list(off) and coeffs == list(coeff)
    Q, R = host(b.Q), host(b.R)
    assert Q.shape == Qo.shape and R.shape == Ro.shape
    assert np.abs(Q - Qo).max() <= 1e-5
    assert np.all(np.abs(R - Ro).max(axis=1) <= 1e-5 * np.maximum(cno, 1.0))
    inside = np.zeros(R.shape, dtype=bool)
    for g in range(len(off) - 1):
        inside[off[g]:off[g + 1], coeff[g]:coeff[g + 1]] = True
    assert np.all(R[~inside] == 0.0)
    for g in range(len(off) - 1):
        Qg = Q[coeff[g]:coeff[g + 1]]
        assert np.abs(Qg @ Qg.T - np.eye(Qg.shape[0])).max() <= 1e-5
    return Qo, Ro, cno


def check_group_argmax(S_ref, off, am, mv, xn, cno):
    G = len(off) - 1
    for g in range(G):
        blk = S_ref[:, off[g]:off[g + 1]]
        bound = TOL_S * xn * cno[off[g]:off[g + 1]].max()
        assert np.all(np.abs(mv[:, g] - blk.max(axis=1)) <= bound)
        if blk.shape[1] > 1:
            top2 = np.sort(blk, axis=1)[:, -2:]
            sure = top2[:, 1] - top2[:, 0] > 2 * bound
        else:
            sure = np.ones(blk.shape[0], dtype=bool)
        assert np.array_equal(am[sure, g], np.argmax(blk, axis=1)[sure])
        chosen = blk[np.arange(blk.shape[0]), am[:, g]]
        assert np.all(chosen >= blk.max(axis=1) - 2 * bound)


def test_attribute_codebooks_in_one_handle(gs, orc):
    """The four attribute codebooks (M = 5, 6, 10, 9, D = 1024) as groups of one handle:
    every attribute's queries scored against all 30 entries in one call, then the best
    entry of each attribute."""
    cases = synth.multiattr()
    C = np.concatenate([a["C"] for a in cases])
    off = np.cumsum([0] + [a["C"].shape[0] for a in cases]).tolist()
    b = gs.build_basis_grouped(cuda(C), off)
    Qo, Ro, cno = check_grouped_build(gs, b, C, off, orc)
    X = np.concatenate([a["X"] for a in cases])
    out = gs.project_similarity(b, cuda(X), want_S=True)
    g = gs.group_argmax(out["S"], off)
    gs.stream_status()
    ref = orc.project_similarity(X, Qo, Ro, cno)
    xn = np.linalg.norm(X.astype(np.float64), axis=1)
    assert np.all(np.abs(host(out["S"]) - ref["S"]) <= TOL_S * xn[:, None] * cno[None, :])
    check_group_argmax(ref["S"], off, g["argmax"].cpu().numpy(), host(g["maxval"]), xn, cno)
    am_o, _ = orc.group_argmax(ref["S"], off)
    # each attribute's own queries: the per-group argmax of its group is its label wherever
    # the label is the clear winner
    n0 = 0
    for a_idx, a in enumerate(cases):
        n1 = n0 + a["X"].shape[0]
        agree = np.mean(am_o[n0:n1, a_idx] == a["labels"])
        assert agree > 0.95
        n0 = n1


def test_partition_when_dimension_below_entries(gs, orc):
    """D < M (Sec. 3.1): 300 bipolar entries of dimension 128 in subsets of at most 128; the
    stacked basis has r = 300 > D coordinates.  Scores equal X C^T, the reconstruction of R
    is the concatenated codebook (rounds back exactly), V = P R reconstructs to P C."""
    rng = np.random.default_rng(20260111)
    M, D = 300, 128
    off = [0, 128, 256, 300]
    C = (rng.integers(0, 2, size=(M, D)) * 2 - 1).astype(np.float32)
    b = gs.build_basis_grouped(cuda(C), off)
    Qo, Ro, cno = check_grouped_build(gs, b, C, off, orc)
    assert b.r == 300
    X, _ = synth.noisy_rows(C, 3, 0, 700, 1.0)
    out = gs.project_similarity(b, cuda(X), want_S=True)
    gs.stream_status()
    xn = np.linalg.norm(X.astype(np.float64), axis=1)
    S_ref = X.astype(np.float64) @ C.astype(np.float64).T
    assert np.all(np.abs(host(out["S"]) - S_ref) <= TOL_S * xn[:, None] * cno[None, :])
    Rp = torch.zeros((M, 304), device="cuda:0")  # 16-byte rows for the tensor-core GEMM
    Rp[:, :300] = b.R
    Xh = gs.reconstruct(b, Rp[:, :300])
    assert np.array_equal(np.rint(host(Xh)), C.astype(np.float64))
    P = synth.attention_probs(9, 1, 256, M, 1).astype(np.float32)
    V = gs.prob_vectorize(b, cuda(P))
    Vp = torch.zeros((256, 304), device="cuda:0")
    Vp[:, :300] = V
    PC = gs.reconstruct(b, Vp[:, :300])
    gs.stream_status()
    ref = P.astype(np.float64) @ C.astype(np.float64)
    bound = 2e-4 * (np.abs(P.astype(np.float64)) @ cno)
    assert np.all(np.abs(host(PC) - ref) <= bound[:, None])


def test_grouped_fused_tensor_path(gs, orc):
    """The large bipolar codebook (M = 256, D = 8192) split into four groups of 64: the
    block-diagonal R goes through the fused tensor-core kernel; the global argmax is the
    generating label and sampled scores match the oracle."""
    C = synth.large_codebook()
    off = [0, 64, 128, 192, 256]
    b = gs.build_basis_grouped(cuda(C), off)
    Qo, Ro, cno, coeff = orc.build_grouped(C, off)
    w = synth.large(rows=(0, 8192))
    X = cuda(w["X"])
    out = gs.project_similarity(b, X, path="tensor", want_S=True)
    g = gs.group_argmax(out["S"], off)
    gs.stream_status()
    assert np.array_equal(out["argmax"].cpu().numpy(), w["labels"])
    rows = np.sort(np.random.default_rng(3).choice(8192, 256, replace=False))
    ref = orc.project_similarity(w["X"][rows], Qo, Ro, cno)
    xn = ref["xnorm"]
    S = host(out["S"][torch.from_numpy(rows).to(X.device)])
    assert np.all(np.abs(S - ref["S"]) <= TOL_S * xn[:, None] * cno[None, :])
    lab = w["labels"]
    am = g["argmax"].cpu().numpy()
    assert np.array_equal(am[np.arange(8192), lab // 64], lab % 64)


def test_import_grouped_and_argument_errors(gs, orc):
    rng = np.random.default_rng(8)
    C = (rng.integers(0, 2, size=(40, 16)) * 2 - 1).astype(np.float32)
    off = [0, 16, 32, 40]
    b = gs.build_basis_grouped(cuda(C), off)
    b2 = gs.import_basis(b.Q.clone(), b.R.clone(), b.cnorm.clone())  # r = 40 > D = 16
    X = cuda(rng.normal(size=(50, 16)).astype(np.float32))
    o1 = gs.project_similarity(b, X, want_S=True)
    o2 = gs.project_similarity(b2, X, want_S=True)
    gs.stream_status()
    assert torch.equal(o1["S"], o2["S"])
    assert gs.basis_groups(b2) == ([0, 40], [0, 40])
    for bad in ([0, 16, 16, 40], [1, 16, 40], [0, 16, 39], [0]):
        with pytest.raises(gs.GramSpaceError) as ei:
            gs.build_basis_grouped(cuda(C), bad)
        assert ei.value.status == gs.GS_ERR_INVALID_ARG
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.group_argmax(torch.zeros((50, 30), device="cuda:0"), off)  # 30 columns, groups up to 40
    assert ei.value.status == gs.GS_ERR_SHAPE
    empty = gs.group_argmax(torch.zeros((0, 40), device="cuda:0"), off)
    assert empty["argmax"].shape == (0, 3)
