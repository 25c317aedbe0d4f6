"""GPU parity of binding / unbinding (gs_bind) and reconstruct-then-bind (gs_reconstruct_bind)
against the float64 oracle (the direct sums of the definition), within the per-output bounds of
tests/bounds.py (direct sum, or the transform bound of the spectral method).  For the fused call
the reconstruction error adds e_rec sqrt(L) ||y_b||, e_rec = 1e-4 ||t|| on the fp16 tensor-core
reconstruction (the reconstruct bound) and 0 on the fp32 path.
"""
import numpy as np
import pytest
import torch

import synth
from bounds import bind_error_factor
from test_parity_gpu import cuda, host

pytestmark = pytest.mark.gpu


def block_norms(A, L):
    N, D = A.shape
    return np.sqrt((A.astype(np.float64).reshape(N, D // L, L) ** 2).sum(axis=2))


def check_bind(Z, Zo, X, Y, L, e_rec=None, method="direct"):
    N, D = Zo.shape
    nx = block_norms(X, L)
    ny = block_norms(np.broadcast_to(Y, (N, D)), L)
    bound = bind_error_factor(L, method) * nx * ny
    if e_rec is not None:
        bound = bound + e_rec[:, None] * np.sqrt(L) * ny
    err = np.abs(host(Z) - Zo).reshape(N, D // L, L).max(axis=2)
    assert np.all(err <= bound + 1e-30)


@pytest.mark.parametrize("N,D,L,bcast,op", [
    (37, 1024, 1024, False, "bind"), (37, 1024, 256, False, "unbind"), (64, 1024, 8, True, "bind"),
    (50, 960, 24, False, "unbind"), (33, 1000, 10, True, "bind"), (5, 4096, 4096, False, "bind"),
    (300, 3000, 1000, False, "unbind"), (1, 64, 64, True, "bind")])
def test_bind_matches_oracle(gs, orc, N, D, L, bcast, op):
    """The direct method on all its kernels (L % 16, L % 8 == 0: shared-memory tiles; L <= 32:
    registers, here with an odd output pitch (element stores); L = 10: one output per thread),
    one partner for all rows, padded leading dimensions."""
    rng = np.random.default_rng(N + D + L)
    X = rng.normal(size=(N, D)).astype(np.float32)
    Y = rng.normal(size=(1 if bcast else N, D)).astype(np.float32)
    Xp = torch.zeros((N, D + 8), device="cuda:0")
    Xp[:, :D] = cuda(X)
    Zp = torch.zeros((N, D + 3), device="cuda:0")  # odd row pitch: element stores
    Z = gs.bind(Xp[:, :D], cuda(Y), L, op, method="direct", out=Zp[:, :D])
    gs.stream_status()
    Zo = orc.bind(X, Y, L, orc.UNBIND if op == "unbind" else orc.BIND)
    check_bind(Z, Zo, X, Y, L)


@pytest.mark.parametrize("N,D,L,bcast,op", [
    (300, 1024, 4, False, "bind"), (97, 960, 12, True, "unbind"), (300, 1024, 16, False, "unbind"),
    (33, 2048, 32, True, "bind"), (7, 640, 20, False, "bind"), (2, 8192, 8192, False, "unbind")])
def test_bind_direct_short_and_long_blocks(gs, orc, N, D, L, bcast, op):
    """The direct sum on short blocks (L <= 32: a block per thread in registers, float4 rows)
    and on a block longer than 48 KB of staging (L = 8192: the shared-memory opt-in)."""
    rng = np.random.default_rng(N + D + L + 2)
    X = rng.normal(size=(N, D)).astype(np.float32)
    Y = rng.normal(size=(1 if bcast else N, D)).astype(np.float32)
    Z = gs.bind(cuda(X), cuda(Y), L, op, method="direct")
    gs.stream_status()
    Zo = orc.bind(X, Y, L, orc.UNBIND if op == "unbind" else orc.BIND)
    check_bind(Z, Zo, X, Y, L)


@pytest.mark.parametrize("N,D,L,bcast,op", [
    (5, 192, 64, False, "bind"), (70, 64, 64, True, "unbind"), (3, 256, 128, False, "unbind"),
    (37, 1024, 256, False, "bind"), (17, 256, 256, False, "unbind"), (9, 1536, 512, True, "bind"),
    (37, 1024, 1024, False, "unbind"), (3, 4096, 2048, False, "bind"), (5, 4096, 4096, False, "unbind"),
    (2, 8192, 8192, False, "bind"), (3, 16384, 8192, True, "unbind"), (6000, 1024, 64, False, "bind"),
    (7, 4096, 1024, True, "bind"), (5, 8192, 4096, True, "unbind"), (40, 2048, 128, True, "unbind"),
    (6000, 1024, 64, True, "unbind")])
def test_bind_spectral_matches_oracle(gs, orc, N, D, L, bcast, op):
    """The spectral method at every block length it takes (L = 64 ... 8192: two and three
    Stockham passes; L = 8192 as whole-vector binding of D = 8192 rows, on 512-thread CTAs),
    partial last groups of blocks, one partner for all rows (its block spectra cached in shared
    memory, two- and three-pass plans; at L = 8192 they do not fit and every team transforms the
    partner itself), padded even row
    pitches, and 96,000 blocks (more groups than resident teams: the persistent loop)."""
    rng = np.random.default_rng(N + D + L + 1)
    X = rng.normal(size=(N, D)).astype(np.float32)
    Y = rng.normal(size=(1 if bcast else N, D)).astype(np.float32)
    Xp = torch.zeros((N, D + 6), device="cuda:0")
    Xp[:, :D] = cuda(X)
    Zp = torch.full((N, D + 2), 7.0, device="cuda:0")
    Z = gs.bind(Xp[:, :D], cuda(Y), L, op, method="spectral", out=Zp[:, :D])
    gs.stream_status()
    Zo = orc.bind(X, Y, L, orc.UNBIND if op == "unbind" else orc.BIND)
    check_bind(Z, Zo, X, Y, L, method="spectral")
    assert torch.all(Zp[:, D:] == 7.0)  # nothing written past a row's D outputs
    # the automatic choice is the spectral kernel here: identical results
    Za = gs.bind(Xp[:, :D], cuda(Y), L, op)
    gs.stream_status()
    assert torch.equal(Za, Z)


def test_unbind_recovers_unit_spectrum_binding(gs):
    rng = np.random.default_rng(7)
    L, D, N = 128, 1024, 16
    spec = np.exp(1j * rng.uniform(-np.pi, np.pi, size=(N, D // L, L)))
    spec[..., 0] = 1.0
    spec[..., L // 2] = 1.0
    spec[..., L // 2 + 1:] = np.conj(spec[..., 1:L // 2][..., ::-1])
    Y = np.real(np.fft.ifft(spec, axis=2)).reshape(N, D).astype(np.float32)
    X = rng.normal(size=(N, D)).astype(np.float32)
    Xd, Yd = cuda(X), cuda(Y)
    for method in ("direct", "spectral"):
        back = gs.bind(gs.bind(Xd, Yd, L, method=method), Yd, L, "unbind", method=method)
        gs.stream_status()
        assert np.abs(host(back) - X).max() <= 1e-4 * np.abs(X).max()


@pytest.mark.parametrize("path,method", [("simt", "direct"), ("tensor", "direct"), ("simt", "spectral"),
                                         ("tensor", "auto")])
def test_reconstruct_bind_matches_oracle(gs, orc, path, method):
    """op(T Q, Y) on the attention codebook's basis (r = 512, D = 4096, blocks of 256); against
    the oracle run with the GPU's basis, so only the kernels' arithmetic differs."""
    a = synth.attention(B=1, L=1)
    b = gs.build_basis(cuda(a["C"]))
    rng = np.random.default_rng(11)
    N = 1024 if path == "tensor" else 200
    T = synth.attention_probs(12, 1, N, b.M, 1).astype(np.float64) @ host(b.R)
    T = T.astype(np.float32)
    Y = rng.normal(size=(N, b.D)).astype(np.float32)
    for op in ("bind", "unbind"):
        Z = gs.reconstruct_bind(b, cuda(T), cuda(Y), 256, op, path=path, method=method)
        gs.stream_status()
        Zo = orc.reconstruct_bind(T, host(b.Q), Y, 256, orc.UNBIND if op == "unbind" else orc.BIND)
        Xo = orc.reconstruct(T, host(b.Q))
        e_rec = 1e-4 * np.linalg.norm(T.astype(np.float64), axis=1) if path == "tensor" else None
        check_bind(Z, Zo, Xo, Y, 256, e_rec, method="direct" if method == "direct" else "spectral")


def test_reconstruct_bind_codebook_and_broadcast(gs, orc):
    """Reconstructing R returns the codebook: binding it with one partner equals binding C."""
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Y = np.random.default_rng(3).normal(size=(1, 1024)).astype(np.float32)
    Rp = torch.zeros((b.M, 8), device="cuda:0")
    Rp[:, :b.r] = b.R
    for method in ("direct", "spectral"):
        Z = gs.reconstruct_bind(b, Rp[:, :b.r], cuda(Y), 128, method=method)
        gs.stream_status()
        Zo = orc.bind(t["C"], Y, 128)
        check_bind(Z, Zo, t["C"], Y, 128, e_rec=np.full(b.M, 1e-5 * np.sqrt(1024)), method=method)


def test_reconstruct_bind_several_chunks(gs, orc):
    """3,000 rows on the tiny basis (M = 8, D = 1024), whose scratch holds 1,024 reconstructed
    rows: three chunks, the last one partial, each reconstructed then bound before the next."""
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    rng = np.random.default_rng(5)
    N = 3000
    P = rng.dirichlet(np.ones(b.M), size=N)
    Tp = torch.zeros((N, 8), device="cuda:0")
    Tp[:, :b.r] = torch.from_numpy(P).to("cuda:0", torch.float32) @ b.R
    Y = rng.normal(size=(N, 1024)).astype(np.float32)
    Tr = host(Tp[:, :b.r])
    Xo = orc.reconstruct(Tr, host(b.Q))
    for method in ("direct", "spectral"):
        for op in ("bind", "unbind"):
            Z = gs.reconstruct_bind(b, Tp[:, :b.r], cuda(Y), 128, op, method=method)
            gs.stream_status()
            Zo = orc.bind(Xo, Y, 128, orc.UNBIND if op == "unbind" else orc.BIND)
            check_bind(Z, Zo, Xo, Y, 128, e_rec=1e-4 * np.linalg.norm(Tr, axis=1), method=method)


def one_partner_bound(T, Q, Y, L, method, path):
    """Per output of block b, for op(T Q, y) computed as T op(Q, y) (one partner row): each bound
    basis row op(q_j, y) carries the binding method's error, f ||q_j,b|| ||y_b||; the
    reconstruction from those rows adds its own rounding, one fp16 rounding each of T and of
    op(Q, y) on the tensor core (|op(q_j, y)_k| <= ||q_j,b|| ||y_b||) and the fp32 sum of r
    products.  Summed with weights |t_j|: (f + eps) ||y_b|| sum_j |t_j| ||q_j,b||."""
    r = Q.shape[0]
    eps = r * 2.0 ** -23 + (2.0 ** -10 if path == "tensor" else 0.0)
    f = bind_error_factor(L, method)
    return (f + eps) * (np.abs(T.astype(np.float64)) @ block_norms(Q, L)) * block_norms(Y, L)[0][None, :]


@pytest.mark.parametrize("path,method", [("simt", "direct"), ("simt", "spectral"), ("tensor", "direct"),
                                         ("tensor", "auto")])
def test_reconstruct_bind_one_partner(gs, orc, path, method):
    """One partner row for 2,000 rows of the attention basis (r = 512 < N): the library binds the
    basis rows once and reconstructs from them (op(t Q, y) = t op(Q, y)); against the oracle's
    reconstruction followed by binding, within the bound of that arithmetic."""
    a = synth.attention(B=1, L=1)
    b = gs.build_basis(cuda(a["C"]))
    N, L = 2000, 256
    T = (synth.attention_probs(13, 1, N, b.M, 1).astype(np.float64) @ host(b.R)).astype(np.float32)
    Y = np.random.default_rng(12).normal(size=(1, b.D)).astype(np.float32)
    Qh = host(b.Q)
    for op in ("bind", "unbind"):
        Z = gs.reconstruct_bind(b, cuda(T), cuda(Y), L, op, path=path, method=method)
        gs.stream_status()
        Zo = orc.reconstruct_bind(T, Qh, Y, L, orc.UNBIND if op == "unbind" else orc.BIND)
        err = np.abs(host(Z) - Zo).reshape(N, b.D // L, L).max(axis=2)
        bound = one_partner_bound(T, Qh, Y, L, "direct" if method == "direct" else "spectral", path)
        assert np.all(err <= bound)


def test_bind_argument_errors(gs):
    X = torch.zeros((4, 100), device="cuda:0")
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.bind(X, X, 30)
    assert ei.value.status == gs.GS_ERR_SHAPE
    assert gs.bind(torch.zeros((0, 100), device="cuda:0"), X[:1], 50).shape == (0, 100)
    with pytest.raises(ValueError):
        gs.bind(X, X[:2], 50)
    # the spectral method: block lengths it does not take, rows off an 8-byte boundary
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.bind(X, X, 50, method="spectral")
    assert ei.value.status == gs.GS_ERR_UNSUPPORTED
    W = torch.zeros((4, 131), device="cuda:0")
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.bind(W[:, :128], W[:, :128], 64, method="spectral")
    assert ei.value.status == gs.GS_ERR_ALIGNMENT
    # the fused call checks the forced method before it reconstructs anything
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Zr = torch.full((4, 1024), 5.0, device="cuda:0")
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.reconstruct_bind(b, b.R[:4], torch.zeros((4, 1024), device="cuda:0"), 32, method="spectral", out=Zr)
    assert ei.value.status == gs.GS_ERR_UNSUPPORTED
    assert torch.all(Zr == 5.0)
    # unknown op bits, or both methods at once
    lib = gs.load_library()
    p = X.data_ptr()
    for op in (8, 2 | 4, -1):
        assert lib.gs_bind(p, 4, 100, 100, p, 100, 50, op, p, 100, None) == gs.GS_ERR_INVALID_ARG
