"""GPU parity of binding / unbinding (gs_bind) and reconstruct-then-bind (gs_reconstruct_bind)
against the float64 oracle.

Bound per output of block b (fp32 sums of L products in j order, and for the fused call the
reconstruction error on top): |Z - Z*| <= L 2^-22 ||x_b|| ||y_b|| + e_rec sqrt(L) ||y_b||, with
e_rec = 1e-4 ||t|| on the fp16 tensor-core reconstruction (the reconstruct bound) and 0 on the fp32
path, where ||x_b||, ||y_b|| are the norms of the row's blocks.
"""
import numpy as np
import pytest
import torch

import synth
from test_parity_gpu import cuda, host

pytestmark = pytest.mark.gpu


def block_norms(A, L):
    N, D = A.shape
    return np.sqrt((A.astype(np.float64).reshape(N, D // L, L) ** 2).sum(axis=2))


def check_bind(Z, Zo, X, Y, L, e_rec=None):
    N, D = Zo.shape
    nx = block_norms(X, L)
    ny = block_norms(np.broadcast_to(Y, (N, D)), L)
    bound = L * 2.0 ** -22 * nx * ny
    if e_rec is not None:
        bound = bound + e_rec[:, None] * np.sqrt(L) * ny
    err = np.abs(host(Z) - Zo).reshape(N, D // L, L).max(axis=2)
    assert np.all(err <= bound + 1e-30)


@pytest.mark.parametrize("N,D,L,bcast,op", [
    (37, 1024, 1024, False, "bind"), (37, 1024, 256, False, "unbind"), (64, 1024, 8, True, "bind"),
    (50, 960, 24, False, "unbind"), (33, 1000, 10, True, "bind"), (5, 4096, 4096, False, "bind"),
    (300, 3000, 1000, False, "unbind"), (1, 64, 64, True, "bind")])
def test_bind_matches_oracle(gs, orc, N, D, L, bcast, op):
    """Block lengths on both kernels (L % 8 == 0: the shared-memory kernel, up to L = 4096;
    L = 10: one output per thread), one partner for all rows, padded leading dimensions."""
    rng = np.random.default_rng(N + D + L)
    X = rng.normal(size=(N, D)).astype(np.float32)
    Y = rng.normal(size=(1 if bcast else N, D)).astype(np.float32)
    Xp = torch.zeros((N, D + 8), device="cuda:0")
    Xp[:, :D] = cuda(X)
    Zp = torch.zeros((N, D + 3), device="cuda:0")  # odd row pitch: element stores
    Z = gs.bind(Xp[:, :D], cuda(Y), L, op, out=Zp[:, :D])
    gs.stream_status()
    Zo = orc.bind(X, Y, L, orc.UNBIND if op == "unbind" else orc.BIND)
    check_bind(Z, Zo, X, Y, L)


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
    back = gs.bind(gs.bind(Xd, Yd, L), Yd, L, "unbind")
    gs.stream_status()
    assert np.abs(host(back) - X).max() <= 1e-4 * np.abs(X).max()


@pytest.mark.parametrize("path", ["simt", "tensor"])
def test_reconstruct_bind_matches_oracle(gs, orc, path):
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
        Z = gs.reconstruct_bind(b, cuda(T), cuda(Y), 256, op, path=path)
        gs.stream_status()
        Zo = orc.reconstruct_bind(T, host(b.Q), Y, 256, orc.UNBIND if op == "unbind" else orc.BIND)
        Xo = orc.reconstruct(T, host(b.Q))
        e_rec = 1e-4 * np.linalg.norm(T.astype(np.float64), axis=1) if path == "tensor" else None
        check_bind(Z, Zo, Xo, Y, 256, e_rec)


def test_reconstruct_bind_codebook_and_broadcast(gs, orc):
    """Reconstructing R returns the codebook: binding it with one partner equals binding C."""
    t = synth.tiny()
    b = gs.build_basis(cuda(t["C"]))
    Y = np.random.default_rng(3).normal(size=(1, 1024)).astype(np.float32)
    Rp = torch.zeros((b.M, 8), device="cuda:0")
    Rp[:, :b.r] = b.R
    Z = gs.reconstruct_bind(b, Rp[:, :b.r], cuda(Y), 128)
    gs.stream_status()
    Zo = orc.bind(t["C"], Y, 128)
    check_bind(Z, Zo, t["C"], Y, 128, e_rec=np.full(b.M, 1e-5 * np.sqrt(1024)))


def test_bind_argument_errors(gs):
    X = torch.zeros((4, 100), device="cuda:0")
    with pytest.raises(gs.GramSpaceError) as ei:
        gs.bind(X, X, 30)
    assert ei.value.status == gs.GS_ERR_SHAPE
    assert gs.bind(torch.zeros((0, 100), device="cuda:0"), X[:1], 50).shape == (0, 100)
    with pytest.raises(ValueError):
        gs.bind(X, X[:2], 50)
