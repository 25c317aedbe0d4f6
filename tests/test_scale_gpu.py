"""Scale-free accuracy of the fp16-input tensor-core paths.

The score bound |S - S*| <= 1e-4 ||x|| ||c_i|| (and 1e-4 ||x|| for Y, 1e-4 ||t|| for a
reconstruction) is relative, so it must hold for queries of any magnitude (Sec. 3.2, Eq. 2-3:
scores on Gram-loc equal the uncompressed ones for every input).  One fp16 rounding of an input
row is accurate only while the row sits inside fp16's range and well above its subnormals; the
kernels detect the rows that do not (from their norms) and compute them again with an exact
power-of-two scale (fused kernel), in fp32 (the two-GEMM projection's rows), or scale every row
before rounding (reconstruction).  Each workload below is run at scales from 1e-6 to 1e5 on the
default path and compared with the float64 oracle on the very fp32 values the GPU received.
"""
import numpy as np
import pytest
import torch

import synth
from test_parity_gpu import TOL_S, check_scores, cuda, host

pytestmark = pytest.mark.gpu

SCALES = [1e-6, 1e-3, 1e3, 1e5]


@pytest.fixture(scope="module")
def large_basis(gs, orc):
    w = synth.large()
    b = gs.build_basis(cuda(w["C"]))
    return w, b, cuda(w["X"])


@pytest.mark.parametrize("scale", SCALES + [1.0])
def test_fused_lookup_any_scale(gs, orc, large_basis, scale):
    """All 65,536 headline queries times `scale`, argmax + maxval only (the kernel the bench
    times): every argmax equals its generating label, maxval of a seeded sample of rows meets
    the bound against the oracle, and the device reports no error."""
    w, b, X = large_basis
    Xs = X * scale
    out = gs.project_similarity(b, Xs)
    gs.stream_status()
    assert np.array_equal(out["argmax"].cpu().numpy(), w["labels"])
    rows = np.sort(np.random.default_rng(41).choice(w["N"], 256, replace=False))
    idx = torch.from_numpy(rows).to(X.device)
    Xr = host(Xs[idx])
    Qh, Rh, cn = host(b.Q), host(b.R), host(b.cnorm)
    ref = orc.project_similarity(Xr, Qh, Rh, cn)
    check_scores({"maxval": out["maxval"][idx], "argmax": out["argmax"][idx]}, ref, Xr, cn)


@pytest.mark.parametrize("scale", SCALES)
@pytest.mark.parametrize("mode,sm_scale", [("raw", 1.0), ("cosine", 1.0), ("softmax", None)])
def test_fused_full_outputs_any_scale(gs, orc, large_basis, scale, mode, sm_scale):
    """6,000 scaled queries with Y and S written (every output of the fused kernel), each mode;
    softmax takes a temperature that keeps the logits O(1) at this scale."""
    w, b, X = large_basis
    Xs = (X[:6000] * scale).contiguous()
    Xh = host(Xs)
    s = sm_scale if sm_scale is not None else 1.0 / (scale * 2048.0)
    out = gs.project_similarity(b, Xs, mode=mode, scale=s, want_Y=True, want_S=True)
    gs.stream_status()
    rows = np.sort(np.random.default_rng(42).choice(6000, 192, replace=False))
    idx = torch.from_numpy(rows).to(X.device)
    Qh, Rh, cn = host(b.Q), host(b.R), host(b.cnorm)
    ref = orc.project_similarity(Xh[rows], Qh, Rh, cn, mode=getattr(orc, mode.upper()), scale=s)
    sub = {k: out[k][idx] for k in ("S", "argmax", "maxval")}
    check_scores(sub, ref, Xh[rows], cn, mode, s)
    assert np.all(np.abs(host(out["Y"][idx]) - ref["Y"]) <= TOL_S * ref["xnorm"][:, None])


@pytest.fixture(scope="module")
def rankdef_basis(gs):
    C, _ = synth.rankdef_codebook()
    return C, gs.build_basis(cuda(C))


@pytest.mark.parametrize("scale", SCALES)
def test_two_gemm_any_scale(gs, orc, rankdef_basis, scale):
    """r = 922 > 256 (the rank-deficient codebook): the two-GEMM tensor-core projection, 1,500
    scaled queries, S and Y against the oracle."""
    C, b = rankdef_basis
    X, _ = synth.noisy_rows(C, synth.SEEDS["rankdef"], 0, 1500, 1.0)
    Xs = cuda(X) * scale
    out = gs.project_similarity(b, Xs, path="tensor", want_S=True, want_Y=True)
    gs.stream_status()
    rows = np.sort(np.random.default_rng(43).choice(1500, 128, replace=False))
    idx = torch.from_numpy(rows).to(Xs.device)
    Xr = host(Xs[idx])
    Qh, Rh, cn = host(b.Q), host(b.R), host(b.cnorm)
    ref = orc.project_similarity(Xr, Qh, Rh, cn)
    check_scores({k: out[k][idx] for k in ("S", "argmax", "maxval")}, ref, Xr, cn)
    assert np.all(np.abs(host(out["Y"][idx]) - ref["Y"]) <= TOL_S * ref["xnorm"][:, None])


@pytest.mark.parametrize("scale", SCALES)
def test_reconstruct_any_scale(gs, orc, large_basis, scale):
    """4,096 coefficient rows times `scale` back to D = 8,192 on the tensor core, with one row of
    magnitude 1e-30 and one of 1e30 among them (each row takes its own scale), against the oracle
    at 1e-4 ||t||."""
    _, b, _ = large_basis
    g = torch.Generator().manual_seed(44)
    T = (torch.randn(4096, b.r, generator=g) * scale).to("cuda:0")
    T[7] *= 1e-30 / scale
    T[8] *= 1e30 / scale
    Xh = gs.reconstruct(b, T)
    gs.stream_status()
    rows = np.concatenate([[7, 8], np.sort(np.random.default_rng(45).choice(np.arange(9, 4096), 62, False))])
    idx = torch.from_numpy(rows).to(T.device)
    Tr = host(T[idx])
    ref = orc.reconstruct(Tr, host(b.Q))
    bound = 1e-4 * np.linalg.norm(Tr, axis=1)
    assert np.all(np.abs(host(Xh[idx]) - ref).max(axis=1) <= bound)
