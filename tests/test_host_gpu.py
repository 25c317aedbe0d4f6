"""GPU tests of project + similarity from host memory (gs_project_similarity_host).

The host entry point streams the queries through the handle's two staging slots;
every row is scored by the same kernels as the device-buffer call, so on the fused
tensor-core path its argmax and maxval equal that call's bit for bit, and on every
path they meet the oracle's bar: argmax bit-exact wherever the oracle's top-2
margin exceeds twice the 1e-4 ||x|| ||c|| score tolerance, maxval within it.
"""
import numpy as np
import pytest
import torch

import synth
from test_parity_gpu import TOL_S, cuda

pytestmark = pytest.mark.gpu


def check_against_oracle(orc, X, C, am, mv):
    Qo, Ro, cno = orc.build_basis(C)
    ref = orc.project_similarity(X, Qo, Ro, cno)
    S = ref["S"]
    xn = np.linalg.norm(X.astype(np.float64), axis=1)
    bound = TOL_S * xn * cno.max()
    assert np.all(np.abs(mv.astype(np.float64) - S.max(axis=1)) <= bound)
    top2 = np.sort(S, axis=1)[:, -2:] if S.shape[1] > 1 else np.concatenate([S, S - np.inf], axis=1)
    sure = (top2[:, 1] - top2[:, 0]) > 2 * bound
    assert np.array_equal(am[sure], ref["argmax"][sure])
    # elsewhere the chosen codeword scores within tolerance of the maximum
    chosen = S[np.arange(len(am)), am]
    assert np.all(chosen >= S.max(axis=1) - 2 * bound)


@pytest.mark.parametrize("N,M,D,ld,rows,path", [
    (1000, 40, 1000, 1000, 384, "tensor"),     # three chunks, the last ragged; two slots reused
    (777, 40, 1002, 1012, 777, "tensor"),      # one chunk, ld > D, D not a multiple of 4
    (1, 40, 1000, 1000, 384, "tensor"),
    (4099, 256, 2048, 2048, 1024, "tensor"),
    (999, 40, 1000, 1000, 256, "simt"),
])
def test_host_matches_device_call(gs, orc, N, M, D, ld, rows, path):
    rng = np.random.default_rng(N + M + D + rows)
    C = (rng.integers(0, 2, size=(M, D)) * 2 - 1).astype(np.float32)
    X, _ = synth.noisy_rows(C, 7, 0, N, 1.0)
    Xp = np.zeros((N, ld), np.float32)
    Xp[:, :D] = X
    Xh = torch.from_numpy(Xp).pin_memory()[:, :D]
    b = gs.build_basis(cuda(C))
    gs.reserve_staging(b, rows)
    out = gs.project_similarity_host(b, Xh, path=path)
    dev = gs.project_similarity(b, cuda(Xp)[:, :D], path=path)  # device rows 16-byte aligned
    torch.cuda.synchronize()
    gs.stream_status()
    am = out["argmax"].numpy()
    mv = out["maxval"].numpy()
    if path == "tensor":
        assert np.array_equal(am, dev["argmax"].cpu().numpy())
        assert np.array_equal(mv, dev["maxval"].cpu().numpy())
    check_against_oracle(orc, X, C, am, mv)


def test_host_calls_back_to_back(gs):
    """Two calls on one stream, the second enqueued before the first has run: the
    second's copies into the slots must wait for the first's kernels, so each call's
    results belong to its own queries.  Also one output only (argmax or maxval)."""
    rng = np.random.default_rng(5)
    C = (rng.integers(0, 2, size=(64, 1024)) * 2 - 1).astype(np.float32)
    X1, lab1 = synth.noisy_rows(C, 8, 0, 3000, 0.5)
    X2, lab2 = synth.noisy_rows(C, 9, 0, 3000, 0.5)
    b = gs.build_basis(cuda(C))
    gs.reserve_staging(b, 512)
    # the pinned inputs stay referenced until the stream has finished: a freed pinned block
    # goes back to torch's host allocator, which may hand it to the next pin_memory() while
    # the copy out of it is still queued
    X1h, X2h = torch.from_numpy(X1).pin_memory(), torch.from_numpy(X2).pin_memory()
    o1 = gs.project_similarity_host(b, X1h, want_maxval=False)
    o2 = gs.project_similarity_host(b, X2h, want_maxval=False)
    o3 = gs.project_similarity_host(b, X1h, want_argmax=False)
    torch.cuda.synchronize()
    gs.stream_status()
    assert "maxval" not in o1 and "argmax" not in o3
    assert np.array_equal(o1["argmax"].numpy(), lab1)
    assert np.array_equal(o2["argmax"].numpy(), lab2)
    ref = gs.project_similarity(b, cuda(X1))
    torch.cuda.synchronize()
    assert np.array_equal(o3["maxval"].numpy(), ref["maxval"].cpu().numpy())


def test_host_without_staging_and_empty(gs):
    rng = np.random.default_rng(6)
    C = (rng.integers(0, 2, size=(16, 512)) * 2 - 1).astype(np.float32)
    b = gs.build_basis(cuda(C))
    X = torch.zeros(10, 512).pin_memory()
    with pytest.raises(RuntimeError):
        gs.project_similarity_host(b, X)
    gs.reserve_staging(b, 64)
    out = gs.project_similarity_host(b, torch.zeros(0, 512))
    assert out["argmax"].numel() == 0
    gs.reserve_staging(b, 0)  # released: the call is refused again
    with pytest.raises(RuntimeError):
        gs.project_similarity_host(b, X)
    with pytest.raises(TypeError):
        gs.project_similarity_host(b, X.to("cuda:0"))
