"""The seeded input recipes (host logic, no GPU): determinism, the regeneration of any row range
on its own, and the value sets and row structure each workload's recipe states."""
import numpy as np

import synth


def test_row_ranges_regenerate_alone():
    C = synth.bipolar(np.random.default_rng(1), 16, 64)
    X, L = synth.noisy_rows(C, 7, 0, 1000, 0.5)
    for i0, i1 in ((0, 1), (255, 257), (300, 1000), (999, 1000)):
        Xr, Lr = synth.noisy_rows(C, 7, i0, i1, 0.5)
        assert np.array_equal(Xr, X[i0:i1]) and np.array_equal(Lr, L[i0:i1])
    X2, _ = synth.noisy_rows(C, 8, 0, 1000, 0.5)
    assert not np.array_equal(X2, X)  # another seed, other rows


def test_noisy_rows_are_codeword_plus_noise():
    C = synth.bipolar(np.random.default_rng(2), 8, 4096)
    X, L = synth.noisy_rows(C, 3, 0, 512, 0.5)
    noise = X.astype(np.float64) - C[L]
    assert abs(noise.mean()) < 0.01 and abs(noise.std() - 0.5) < 0.01
    assert set(np.unique(C)) == {-1.0, 1.0}
    assert np.bincount(L, minlength=8).min() > 0


def test_rankdef_codebook_structure():
    """Small instance of the rank-deficient recipe: binary independent rows, dependent rows
    that are duplicates or +-a +-b of two independent rows, rank = number of independent rows."""
    C, rank = synth.rankdef_codebook(M=60, D=200)
    assert rank == 54 and C.shape == (60, 200)
    assert np.linalg.matrix_rank(C.astype(np.float64)) == 54
    assert set(np.unique(C)) <= {-2.0, -1.0, 0.0, 1.0, 2.0}
    binary = [i for i in range(60) if set(np.unique(C[i])) <= {0.0, 1.0}]
    assert len(binary) >= 54


def test_attention_and_multiattr_probabilities():
    P = synth.attention_probs(5, 2, 8, 512, 1)
    assert P.shape == (16, 512) and np.all(P > 0)
    assert np.allclose(P.sum(axis=1), 1.0, atol=1e-5)
    for a in synth.multiattr(problems=2, panels=4):
        M = a["C"].shape[0]
        assert M in synth.MULTIATTR_M and a["X"].shape == (8, 1024) and a["P"].shape == (8, M)
        assert np.allclose(a["P"].sum(axis=1), 1.0, atol=1e-5)
        assert np.array_equal(a["labels"], np.argmax(a["P"], axis=1))
        # x = p C + N(0, 0.1^2)
        resid = a["X"].astype(np.float64) - a["P"].astype(np.float64) @ a["C"].astype(np.float64)
        assert abs(resid.std() - 0.1) < 0.01


def test_sweep_codebooks():
    for D in synth.SWEEP_D[:3]:
        w = synth.sweep(D)
        assert w["C"].shape == (40, D) and w["X"].shape == (1024, D)
        assert np.array_equal(synth.sweep(D)["X"], w["X"])
