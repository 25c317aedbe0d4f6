"""The allocation-free project + similarity entry point, against the float64 oracle and against
the regular entry point.

gs_project_similarity_static serves callers that cannot allocate device memory (graph captures
that forbid it, plugins inside a fixed memory budget, hosts whose allocator owns the device): its
scratch is a fixed array inside the library, shared by every call.  Its scores must meet the same
bound as every fp32 path (|S - S*| <= 1e-4 ||x|| ||c_i||, argmax exact where the oracle's top-2
margin clears twice that), in every score mode and output combination, for a rank-0 basis and
an empty batch, and two calls in a row (the second reusing the scratch the first left behind)
must agree with the regular entry point.  This file is collected last so that, if it fails, a
run stopping at the first failure has already run every other test; it also passes when run
alone in a fresh process.
"""
import numpy as np
import pytest
import torch

import synth
from test_parity_gpu import check_scores

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def attn_basis(gs):
    a = synth.attention(B=1, L=1)  # r = M = 512, D = 4096: 1025 scratch floats per row
    b = gs.build_basis(torch.from_numpy(a["C"]).cuda())
    return a, b


@pytest.mark.parametrize("mode,scale", [("raw", 1.0), ("cosine", 1.0), ("softmax", 1.0 / 64)])
def test_static_entry_matches_oracle(gs, orc, attn_basis, mode, scale):
    """6,000 rows (two chunks of the static scratch), each mode, against the oracle run with the
    same basis (so only the kernels' arithmetic differs)."""
    a, b = attn_basis
    X, _ = synth.noisy_rows(a["C"], 31, 0, 6000, 1.0)
    Q, R, cn = b.Q.contiguous(), b.R.contiguous(), b.cnorm.contiguous()
    got = gs.project_similarity_static(Q, R, cn, torch.from_numpy(X).cuda(), mode=mode, scale=scale)
    gs.stream_status()
    ref = orc.project_similarity(X, Q.double().cpu().numpy(), R.double().cpu().numpy(),
                                 cn.double().cpu().numpy(), mode=getattr(orc, mode.upper()), scale=scale)
    check_scores(got, ref, X, cn.double().cpu().numpy(), mode, scale)


def test_static_entry_single_outputs(gs, orc, attn_basis):
    """argmax alone and maxval alone (the row reduction writes only what is asked for)."""
    a, b = attn_basis
    X, _ = synth.noisy_rows(a["C"], 32, 0, 500, 1.0)
    Q, R, cn = b.Q.contiguous(), b.R.contiguous(), b.cnorm.contiguous()
    Xd = torch.from_numpy(X).cuda()
    ref = orc.project_similarity(X, Q.double().cpu().numpy(), R.double().cpu().numpy(), cn.double().cpu().numpy())
    cnh = cn.double().cpu().numpy()
    only_am = gs.project_similarity_static(Q, R, cn, Xd, want_maxval=False)
    only_mv = gs.project_similarity_static(Q, R, cn, Xd, want_argmax=False)
    gs.stream_status()
    assert set(only_am) == {"argmax"} and set(only_mv) == {"maxval"}
    check_scores(only_am, ref, X, cnh)
    check_scores(only_mv, ref, X, cnh)


def test_static_entry_rank_zero_and_empty(gs):
    """A zero codebook has rank 0: every score is 0 (softmax: 1/M) and argmax is 0; N = 0 returns
    at once with empty outputs."""
    b = gs.build_basis(torch.zeros((6, 64), device="cuda"))
    assert b.r == 0
    Q, R = torch.zeros((0, 64), device="cuda"), torch.zeros((6, 0), device="cuda")
    cn = b.cnorm.contiguous()
    X = torch.ones((5, 64), device="cuda")
    raw = gs.project_similarity_static(Q, R, cn, X)
    sm = gs.project_similarity_static(Q, R, cn, X, mode="softmax")
    cos = gs.project_similarity_static(Q, R, cn, X, mode="cosine")
    gs.stream_status()
    assert torch.all(raw["argmax"] == 0) and torch.all(raw["maxval"] == 0)
    assert torch.allclose(sm["maxval"], torch.full((5,), 1 / 6, device="cuda"))
    assert torch.all(cos["maxval"] == 0)
    empty = gs.project_similarity_static(Q, R, cn, torch.zeros((0, 64), device="cuda"))
    gs.stream_status()
    assert empty["argmax"].numel() == 0 and empty["maxval"].numel() == 0


def test_static_entry_two_calls_match_regular_entry(gs, attn_basis):
    """Two calls in a row share the static scratch; each matches the regular entry point."""
    a, b = attn_basis
    Q, R, cn = b.Q.contiguous(), b.R.contiguous(), b.cnorm.contiguous()
    for mode, scale, seed in [("cosine", 1.0, 7), ("raw", 0.5, 8)]:
        X, _ = synth.noisy_rows(a["C"], seed, 0, 6000, 1.0)
        Xd = torch.from_numpy(X).cuda()
        got = gs.project_similarity_static(Q, R, cn, Xd, mode=mode, scale=scale)
        ref = gs.project_similarity(b, Xd, mode=mode, scale=scale, path="simt")
        gs.stream_status()
        assert torch.equal(got["argmax"], ref["argmax"])
        xn = np.linalg.norm(X.astype(np.float64), axis=1)
        bound = 1e-4 * (abs(scale) if mode == "cosine" else abs(scale) * xn * np.sqrt(a["D"]))
        diff = (got["maxval"] - ref["maxval"]).abs().double().cpu().numpy()
        assert np.all(diff <= bound)


def test_static_entry_rejects_oversized_problems(gs):
    lib = gs.load_library()
    st = lib.gs_project_similarity_static(None, 4096, 8, None, 4 << 20, None, None, 1, 8, 0, 1.0,
                                          None, None, None)
    assert st == gs.GS_ERR_SHAPE
    assert lib.gs_project_similarity_static(None, 0, 8, None, 4, None, None, 0, 8, 0, 1.0, None, None,
                                            None) == gs.GS_OK
