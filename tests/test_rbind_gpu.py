"""Reconstruct + bind with per-row partners in one kernel (gs_rbind_tc.cu) against the float64
oracle's reconstruction followed by the binding's definition (Sec. 3.3: reconstruction at the
transition into the component-wise operators; Sec. 2.2: block circular convolution / correlation).

The kernel reconstructs each 128 x 256 tile of T Q on the tensor core (one fp16 rounding of the
power-of-two-scaled T rows and of Q) and binds it through block spectra computed in tensor memory,
so its error is the tensor-core reconstruction's (1e-4 ||t||, carried through the binding as
1e-4 ||t|| sqrt(L) ||y_b||) plus the spectral method's (tests/bounds.py).  The shapes reach every
edge of the tiling: rows that do not fill the last 128-row tile, a last column tile holding fewer
than 256 columns (D % 256 = 128), ranks that end inside a 64-wide K-block, partner and output rows
with padded pitches, each block length the kernel takes (64, 128, 256), and enough tiles that
every CTA runs several (the two TMEM halves swap roles each tile).
"""
import numpy as np
import pytest
import torch

from test_bind_gpu import check_bind
from test_parity_gpu import cuda, host

pytestmark = pytest.mark.gpu


def codebook(M, D, seed):
    return np.random.default_rng(seed).normal(size=(M, D)).astype(np.float32)


def rows(n, k, seed):
    return np.sort(np.random.default_rng(seed).choice(n, min(n, k), replace=False))


@pytest.mark.parametrize("N,M,D,L,op,pad", [
    (1000, 300, 1152, 128, "bind", 0),     # ragged rows, ragged column tile, r = 300 (partial K-block)
    (777, 200, 1024, 64, "unbind", 4),     # padded partner and output pitches
    (513, 512, 4096, 256, "bind", 0),
    (513, 512, 4096, 256, "unbind", 8),
    (130, 40, 2048, 256, "unbind", 0),     # one K-block, mostly zero fill
    (300, 96, 1152, 64, "bind", 0),        # four blocks per tile row, ragged column tile
])
def test_fused_reconstruct_bind_matches_oracle(gs, orc, N, M, D, L, op, pad):
    C = codebook(M, D, 100 + N)
    b = gs.build_basis(cuda(C))
    assert b.r == min(M, D)
    rng = np.random.default_rng(N + D)
    T = rng.normal(size=(N, b.r)).astype(np.float32)
    Y = rng.normal(size=(N, D)).astype(np.float32)
    Yd = torch.zeros((N, D + pad), device="cuda:0")
    Yd[:, :D] = cuda(Y)
    Zbuf = torch.full((N, D + pad), float("nan"), device="cuda:0")
    Z = gs.reconstruct_bind(b, cuda(T), Yd[:, :D], L, op, path="tensor", out=Zbuf[:, :D])
    gs.stream_status()
    if pad:
        assert torch.isnan(Zbuf[:, D:]).all()  # nothing written past the rows' D columns
    Qh = host(b.Q)
    Xo = orc.reconstruct(T, Qh)
    Zo = orc.bind(Xo, Y, L, orc.UNBIND if op == "unbind" else orc.BIND)
    e_rec = 1e-4 * np.linalg.norm(T.astype(np.float64), axis=1)
    check_bind(Z, Zo, Xo, Y, L, e_rec, method="spectral")


@pytest.mark.parametrize("N,L,op", [(6000, 64, "unbind"), (4500, 128, "bind")])
def test_fused_reconstruct_bind_many_tiles(gs, orc, N, L, op):
    """D = 4096: 47 or 36 row tiles x 16 column tiles, several per CTA; sampled rows."""
    C = codebook(512, 4096, 7)
    b = gs.build_basis(cuda(C))
    g = torch.Generator().manual_seed(N)
    T = torch.randn(N, b.r, generator=g).to("cuda:0")
    Y = torch.randn(N, 4096, generator=g).to("cuda:0")
    Z = gs.reconstruct_bind(b, T, Y, L, op)
    gs.stream_status()
    idx = rows(N, 48, L)
    it = torch.from_numpy(idx).to(T.device)
    Tr, Yr = host(T[it]), host(Y[it])
    Xo = orc.reconstruct(Tr, host(b.Q))
    Zo = orc.bind(Xo, Yr, L, orc.UNBIND if op == "unbind" else orc.BIND)
    check_bind(Z[it], Zo, Xo, Yr, L, 1e-4 * np.linalg.norm(Tr.astype(np.float64), axis=1), method="spectral")


def test_fused_reconstruct_bind_row_scales(gs, orc):
    """Coefficient rows of magnitude 1e-30 and 1e30 (each takes its own exact scale before the
    fp16 rounding, undone before the transforms), a zero row (its output is exactly zero) and a
    zero partner row."""
    C = codebook(256, 2048, 3)
    b = gs.build_basis(cuda(C))
    rng = np.random.default_rng(4)
    N, L = 600, 256
    T = rng.normal(size=(N, b.r)).astype(np.float32)
    T[3] *= 1e-30
    T[4] *= 1e30
    T[5] = 0.0
    Y = rng.normal(size=(N, 2048)).astype(np.float32)
    Y[6] = 0.0
    for op in ("bind", "unbind"):
        Z = gs.reconstruct_bind(b, cuda(T), cuda(Y), L, op, path="tensor")
        gs.stream_status()
        Zh = host(Z)
        assert np.all(Zh[5] == 0.0) and np.all(Zh[6] == 0.0)
        Xo = orc.reconstruct(T, host(b.Q))
        Zo = orc.bind(Xo, Y, L, orc.UNBIND if op == "unbind" else orc.BIND)
        check_bind(Z, Zo, Xo, Y, L, 1e-4 * np.linalg.norm(T.astype(np.float64), axis=1), method="spectral")


def test_fused_reconstruct_bind_agrees_with_two_calls(gs):
    """The fused call against gs_reconstruct then gs_bind (the same reconstruction arithmetic,
    the spectral binding through shared memory): both within the bound, so their difference is
    within twice the binding error plus nothing from the reconstruction."""
    C = codebook(512, 4096, 9)
    b = gs.build_basis(cuda(C))
    g = torch.Generator().manual_seed(10)
    T = torch.randn(2048, b.r, generator=g).to("cuda:0")
    Y = torch.randn(2048, 4096, generator=g).to("cuda:0")
    Z1 = gs.reconstruct_bind(b, T, Y, 256, path="tensor")
    Xh = gs.reconstruct(b, T, path="tensor")
    Z2 = gs.bind(Xh, Y, 256, method="spectral")
    gs.stream_status()
    from bounds import bind_error_factor
    from test_bind_gpu import block_norms
    nx = block_norms(host(Xh), 256)
    ny = block_norms(host(Y), 256)
    bound = 2 * bind_error_factor(256, "spectral") * nx * ny
    err = np.abs(host(Z1) - host(Z2)).reshape(2048, 16, 256).max(axis=2)
    assert np.all(err <= bound)
