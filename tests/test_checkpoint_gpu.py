"""Basis checkpoint / restore: save Q, R and the codeword norms of a built basis,
restore a handle from them with gs_basis_import (no Gram-Schmidt), and check that
every operation of the restored handle returns bit-identical results; also the
host round trip (through numpy) and restoring without the norms."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


@pytest.mark.parametrize("which", ["tiny", "rankdef"])
def test_restored_basis_is_bit_identical(gs, which):
    if which == "tiny":
        C = synth.tiny()["C"]
        X, _ = synth.noisy_rows(C, 5, 0, 300, 0.5)
    else:
        C, _ = synth.rankdef_codebook()
        X, _ = synth.noisy_rows(C, synth.SEEDS["rankdef"], 0, 600, 1.0)
    b = gs.build_basis(cuda(C))
    # save to the host (as a checkpoint file would) and restore on the device
    saved = {k: getattr(b, k).cpu().numpy().copy() for k in ("Q", "R", "cnorm")}
    b2 = gs.import_basis(cuda(saved["Q"]), cuda(saved["R"]), cuda(saved["cnorm"]))
    assert (b2.M, b2.D, b2.r) == (b.M, b.D, b.r)
    for k in ("Q", "R", "cnorm"):
        assert torch.equal(getattr(b2, k), getattr(b, k))
    Xd = cuda(X)
    for path in ("auto", "simt"):
        o1 = gs.project_similarity(b, Xd, path=path, want_Y=True, want_S=True)
        o2 = gs.project_similarity(b2, Xd, path=path, want_Y=True, want_S=True)
        for k in o1:
            assert torch.equal(o1[k], o2[k]), (path, k)
    T = torch.randn(257, (b.r + 3) // 4 * 4, device=DEV)[:, :b.r]
    assert torch.equal(gs.reconstruct(b, T), gs.reconstruct(b2, T))
    P = torch.softmax(torch.randn(200, b.M, device=DEV), dim=1)
    assert torch.equal(gs.prob_vectorize(b, P), gs.prob_vectorize(b2, P))
    gs.stream_status()


def test_restore_without_norms_uses_coefficient_norms(gs):
    C = synth.tiny()["C"]
    b = gs.build_basis(cuda(C))
    b2 = gs.import_basis(b.Q.clone(), b.R.clone())
    cn = np.linalg.norm(C.astype(np.float64), axis=1)
    assert np.allclose(b2.cnorm.double().cpu().numpy(), cn, rtol=1e-6)


def test_restore_errors_and_rank_zero(gs):
    z = gs.import_basis(torch.zeros((0, 64), device=DEV), torch.zeros((5, 0), device=DEV))
    assert z.r == 0 and z.M == 5
    with pytest.raises(gs.GramSpaceError) as e:  # r > min(M, D)
        gs.import_basis(torch.zeros((6, 64), device=DEV), torch.zeros((5, 6), device=DEV))
    assert e.value.status == gs.GS_ERR_SHAPE
