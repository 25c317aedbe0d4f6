"""Pins of the float64 oracle against facts that do not come from the oracle itself.

Each test checks the oracle against something the paper or the mathematics fixes:
closed forms that avoid the basis altogether (S = X C^T, V Q = P C, attention
logits P_q C C^T P_k^T / sqrt(D)), the invariants of Sec. 3.2 (Eq. 2-4), the
textbook special case that Sec. 3.2 names (Householder QR, sign-fixed), exact
rational Gram-Schmidt on tiny integer codebooks, the paper's worked numbers
(tests/golden), and the generating labels of the synthetic queries.  The
planted-mistake tests show that a dropped reorthogonalisation pass or a flipped
sign does fail a pin.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- fixtures
@pytest.fixture(scope="session")
def tiny_case(orc):
    t = synth.tiny()
    return t, orc.build_basis(t["C"])


@pytest.fixture(scope="session")
def large_case(orc):
    C = synth.large_codebook()
    return C, orc.build_basis(C)


@pytest.fixture(scope="session")
def attn_case(orc):
    a = synth.attention(B=2, L=48)
    return a, orc.build_basis(a["C"])


@pytest.fixture(scope="session")
def rankdef_case(orc):
    C, rank = synth.rankdef_codebook()
    return C, rank, orc.build_basis(C)


def _check_invariants(C, Q, R, cn, tol):
    C = C.astype(np.float64)
    r = Q.shape[0]
    # Q Q^T = I_r (U^T U = I_k, Sec. 3.2)
    assert np.abs(Q @ Q.T - np.eye(r)).max() <= tol
    # C = R Q (Eq. 1 and Eq. 4: each codeword is exactly its expansion)
    norms = np.linalg.norm(C, axis=1)
    assert np.all(np.abs(R @ Q - C).max(axis=1) <= tol * np.maximum(norms, 1.0))
    # <c_i, c_j> = <R_i, R_j> (Eq. 2)
    G = C @ C.T
    assert np.abs(R @ R.T - G).max() <= tol * max(1.0, norms.max() ** 2)
    # ||R_i|| = ||c_i|| (Eq. 2 with A = B), and cnorm reports it
    assert np.allclose(np.linalg.norm(R, axis=1), norms, rtol=tol, atol=tol)
    assert np.allclose(cn, norms, rtol=1e-14, atol=0)
    # R is lower echelon with positive pivots (row order, positive normalisation)
    piv = 0
    for i in range(R.shape[0]):
        nz = np.nonzero(R[i])[0]
        last = nz.max() + 1 if nz.size else 0
        assert last <= piv + 1
        if last == piv + 1:
            assert R[i, piv] > 0
            piv += 1
    assert piv == r


# ----------------------------------------------------------------- build
def test_build_invariants_all_workloads(orc, tiny_case, large_case, attn_case):
    t, (Q, R, cn) = tiny_case
    _check_invariants(t["C"], Q, R, cn, 1e-12)
    for a in synth.multiattr():
        Qa, Ra, cna = orc.build_basis(a["C"])
        assert Qa.shape[0] == a["C"].shape[0]
        _check_invariants(a["C"], Qa, Ra, cna, 1e-12)
    C, (Q, R, cn) = large_case
    _check_invariants(C, Q, R, cn, 1e-11)
    a, (Q, R, cn) = attn_case
    _check_invariants(a["C"], Q, R, cn, 1e-11)


def test_build_rank_deficient_full_size(rankdef_case):
    """The rank-deficient binary workload: rank 922 by construction (102 of 1024
    rows are duplicates or +-1 combinations of two others)."""
    C, rank, (Q, R, cn) = rankdef_case
    assert Q.shape[0] == rank == 922
    _check_invariants(C, Q, R, cn, 1e-10)


def test_householder_crosscheck(orc, tiny_case, large_case, attn_case):
    """Sec. 3.2 computes the basis by Householder QR.  For full row rank the
    row-order Gram-Schmidt with positive pivots is the unique LQ factor, so it
    must equal LAPACK's Householder QR of C^T with signs fixed."""
    cases = [(tiny_case[0]["C"], tiny_case[1]), (large_case[0], large_case[1]),
             (attn_case[0]["C"], attn_case[1])]
    cases += [(a["C"], orc.build_basis(a["C"])) for a in synth.multiattr()]
    for C, (Q, R, _) in cases:
        Qh, Rh = np.linalg.qr(C.astype(np.float64).T)
        s = np.sign(np.diag(Rh))
        Qh = Qh * s
        Rh = Rh * s[:, None]
        assert np.abs(Q - Qh.T).max() < 1e-10
        assert np.abs(R - Rh.T).max() < 1e-10 * np.abs(Rh).max()


def _exact_gs(C):
    """Gram-Schmidt in exact rational arithmetic (orthogonal, unnormalised w_j)."""
    W = []
    for c in C:
        v = [Fraction(int(x)) for x in c]
        for w in W:
            ww = sum(a * a for a in w)
            k = sum(a * b for a, b in zip(v, w)) / ww
            v = [a - k * b for a, b in zip(v, w)]
        if any(a != 0 for a in v):
            W.append(v)
    Q = np.array([[float(a) for a in w] for w in W]) if W else np.zeros((0, C.shape[1]))
    if W:
        Q /= np.sqrt([float(sum(a * a for a in w)) for w in W])[:, None]
    return Q


@pytest.mark.parametrize("case", range(4))
def test_exact_rational_tiny(orc, case):
    """Brute force on tiny integer codebooks: rank and basis from exact rational
    Gram-Schmidt (no rounding at all, so the rank decision is exact)."""
    rng = np.random.default_rng(77 + case)
    if case == 0:   # duplicates, a zero row and a signed combination
        B = rng.integers(-1, 2, size=(4, 9))
        C = np.stack([B[0], B[1], B[0], np.zeros(9), B[2], B[0] - B[2], B[3], B[1] + B[3]])
    elif case == 1:  # more rows than dimensions (paper Sec. 3.1, D < M)
        C = rng.integers(-1, 2, size=(9, 5))
    elif case == 2:  # binary {0,1} with dependent rows
        B = rng.integers(0, 2, size=(5, 12))
        C = np.concatenate([B, B[:2] + B[2:4], B[4:5]])
    else:            # bipolar, full rank
        C = rng.integers(0, 2, size=(6, 16)) * 2 - 1
    Qx = _exact_gs(C)
    Q, R, _ = orc.build_basis(C.astype(np.float64), tau=1e-9)
    assert Q.shape[0] == Qx.shape[0] == np.linalg.matrix_rank(C)
    assert np.abs(Q - Qx).max() < 1e-12
    assert np.abs(R @ Q - C).max() < 1e-12


def test_reorthogonalisation_needed(orc):
    """An ill-conditioned codebook (rows = common vector + 1e-7 perturbations):
    with both passes Q stays orthonormal to ~1e-15; the planted single-pass
    variant loses orthogonality by orders of magnitude and fails the same pin."""
    rng = np.random.default_rng(5)
    base = rng.standard_normal(300)
    C = base + 1e-7 * rng.standard_normal((24, 300))
    Q2, _, _ = orc.build_basis(C, tau=1e-14, passes=2)
    Q1, _, _ = orc.build_basis(C, tau=1e-14, passes=1)
    assert Q2.shape[0] == 24 and Q1.shape[0] == 24
    e2 = np.abs(Q2 @ Q2.T - np.eye(24)).max()
    e1 = np.abs(Q1 @ Q1.T - np.eye(24)).max()
    assert e2 < 1e-13
    assert e1 > 1e-11


def test_planted_sign_error_fails_pin(orc, tiny_case):
    """Flipping the sign of one basis vector keeps Q orthonormal and C = R Q, but
    the positive-pivot (Householder, sign-fixed) pin catches it."""
    t, (Q, R, _) = tiny_case
    Qb, Rb = Q.copy(), R.copy()
    Qb[3] *= -1
    Rb[:, 3] *= -1
    assert np.abs(Rb @ Qb - t["C"]).max() < 1e-12
    Qh, Rh = np.linalg.qr(t["C"].astype(np.float64).T)
    s = np.sign(np.diag(Rh))
    assert np.abs(Qb - (Qh * s).T).max() > 1.0 / np.sqrt(Qb.shape[1])


def test_zero_and_degenerate_codebooks(orc):
    Q, R, cn = orc.build_basis(np.zeros((5, 32)))
    assert Q.shape == (0, 32) and R.shape == (5, 0) and np.all(cn == 0)
    X = np.random.default_rng(1).standard_normal((7, 32))
    Y, xn = orc.project(X, Q)
    S, am, mv = orc.similarity(Y, R)
    assert np.all(S == 0) and np.all(am == 0) and np.all(mv == 0)
    # a single codeword
    c = np.ones((1, 16))
    Q, R, cn = orc.build_basis(c)
    assert np.allclose(Q, 0.25) and np.allclose(R, 4.0)


def test_normalize_rows_reading(orc):
    """With atom normalisation (Sec. 3.1) the basis is unchanged and R_i scales
    by 1/||c_i||."""
    C = synth.tiny()["C"].astype(np.float64) * np.arange(1, 9)[:, None]
    Q, R, _ = orc.build_basis(C)
    Qn, Rn, cnn = orc.build_basis(C, normalize_rows=True)
    assert np.abs(Q - Qn).max() < 1e-13
    assert np.abs(Rn - R / np.linalg.norm(C, axis=1)[:, None]).max() < 1e-13
    assert np.allclose(cnn, 1.0)


# ----------------------------------------------------------------- similarity
def test_similarity_closed_form(orc, tiny_case):
    """Compressed scores equal uncompressed ones: S = scale * X C^T (Eq. 2-3)."""
    t, (Q, R, cn) = tiny_case
    X = t["X"].astype(np.float64)
    C = t["C"].astype(np.float64)
    full = X @ C.T
    xn = np.linalg.norm(X, axis=1)
    bound = 1e-12 * xn[:, None] * np.linalg.norm(C, axis=1)[None, :]
    o = orc.project_similarity(X, Q, R, cn, mode=orc.RAW, scale=0.5)
    assert np.all(np.abs(o["S"] - 0.5 * full) <= bound)
    o = orc.project_similarity(X, Q, R, cn, mode=orc.COSINE)
    cos = full / (xn[:, None] * np.linalg.norm(C, axis=1)[None, :])
    assert np.abs(o["S"] - cos).max() < 1e-13
    scale = 1.0 / 32
    o = orc.project_similarity(X, Q, R, cn, mode=orc.SOFTMAX, scale=scale)
    from scipy.special import softmax
    assert np.abs(o["S"] - softmax(scale * full, axis=1)).max() < 1e-13
    assert np.allclose(o["S"].sum(axis=1), 1.0, atol=1e-14)
    assert np.all(o["argmax"] == np.argmax(full, axis=1))
    assert np.all(o["argmax"] == t["labels"])


def test_cosine_uses_full_dimension_norm(orc, tiny_case):
    """For a query outside span(C), ||x|| > ||Q x||; the cosine reading uses the
    full-D norm so compressed cosine equals uncompressed cosine."""
    t, (Q, R, cn) = tiny_case
    X = t["X"][:4].astype(np.float64)
    o = orc.project_similarity(X, Q, R, cn, mode=orc.COSINE)
    assert np.all(np.linalg.norm(o["Y"], axis=1) < 0.99 * np.linalg.norm(X, axis=1))
    C = t["C"].astype(np.float64)
    ref = (X @ C.T) / np.linalg.norm(X, axis=1)[:, None] / np.linalg.norm(C, axis=1)[None, :]
    assert np.abs(o["S"] - ref).max() < 1e-13


def test_argmax_lowest_index_on_ties(orc):
    C = np.array([[1.0, 0, 0], [1.0, 0, 0], [0, 1.0, 0], [0, 1.0, 0]])
    Q, R, cn = orc.build_basis(C)
    X = np.array([[0, 2.0, 0], [3.0, 0, 0], [1.0, 1.0, 0]])
    o = orc.project_similarity(X, Q, R, cn)
    assert list(o["argmax"]) == [2, 0, 0]


def test_label_invariant_large_sample(orc, large_case):
    """Noisy copies of known codewords (sigma = 1, D = 8192): the margin of the
    generating label is ~8192 against score noise ~128, so the oracle's argmax
    must be the label; checked on the first 512 queries."""
    C, (Q, R, cn) = large_case
    w = synth.large(rows=(0, 512))
    o = orc.project_similarity(w["X"], Q, R, cn)
    assert np.all(o["argmax"] == w["labels"])
    full = w["X"].astype(np.float64) @ C.T.astype(np.float64)
    xn = np.linalg.norm(w["X"].astype(np.float64), axis=1)
    assert np.all(np.abs(o["S"] - full) <= 1e-11 * xn[:, None] * math.sqrt(C.shape[1]))


# ----------------------------------------------------------------- prob-vec / reconstruct / attention
def test_prob_vectorize_closed_form(orc, tiny_case):
    """V = P R is the Gram-loc of P C: V Q = P C, and V V^T = P (C C^T) P^T."""
    t, (Q, R, cn) = tiny_case
    P = t["P"].astype(np.float64)
    C = t["C"].astype(np.float64)
    V = orc.prob_vectorize(P, R)
    assert np.abs(V @ Q - P @ C).max() < 1e-12
    assert np.abs(V @ V.T - P @ C @ C.T @ P.T).max() < 1e-10
    for a in synth.multiattr():
        Qa, Ra, _ = orc.build_basis(a["C"])
        Va = orc.prob_vectorize(a["P"], Ra)
        assert np.abs(Va @ Qa - a["P"].astype(np.float64) @ a["C"]).max() < 1e-12


def test_reconstruct_round_trips_codebooks(orc, tiny_case, rankdef_case):
    """Exact reconstruction (Sec. 3.2, Table 4 "100 %"): reconstruct(R) = C, and
    integer codebooks come back bit-exact after rounding."""
    t, (Q, R, _) = tiny_case
    assert np.array_equal(np.rint(orc.reconstruct(R, Q)), t["C"])
    C, _, (Q, R, _) = rankdef_case
    sel = np.arange(0, C.shape[0], 7)
    assert np.array_equal(np.rint(orc.reconstruct(R[sel], Q)), C[sel])


def test_reconstruct_is_projector(orc, tiny_case):
    """x -> U U^T x (Eq. 4) is the orthogonal projector onto span(C): it matches
    the least-squares projection, is idempotent, and leaves a residual
    orthogonal to every codeword."""
    t, (Q, R, _) = tiny_case
    X = t["X"][:16].astype(np.float64)
    C = t["C"].astype(np.float64)
    Y, _ = orc.project(X, Q)
    Xp = orc.reconstruct(Y, Q)
    coef, *_ = np.linalg.lstsq(C.T, X.T, rcond=None)
    assert np.abs(Xp - (C.T @ coef).T).max() < 1e-12
    Y2, _ = orc.project(Xp, Q)
    assert np.abs(orc.reconstruct(Y2, Q) - Xp).max() < 1e-12
    assert np.abs((X - Xp) @ C.T).max() < 1e-9


def test_attention_closed_form(orc, attn_case):
    """Attention between compressed vectors equals full-dimension attention of
    the superposed vectors: logits = P_q (C C^T) P_k^T / sqrt(D)."""
    a, (Q, R, _) = attn_case
    B, L, D = a["B"], a["L"], a["D"]
    C = a["C"].astype(np.float64)
    Vq = orc.prob_vectorize(a["Pq"], R)
    Vk = orc.prob_vectorize(a["Pk"], R)
    scale = 1.0 / math.sqrt(D)
    logits = orc.attention(Vq, Vk, B, L, L, scale, apply_softmax=False)
    A = orc.attention(Vq, Vk, B, L, L, scale, apply_softmax=True)
    Pq = a["Pq"].astype(np.float64).reshape(B, L, -1)
    Pk = a["Pk"].astype(np.float64).reshape(B, L, -1)
    G = C @ C.T
    ref = np.einsum("bqm,mn,bkn->bqk", Pq, G, Pk) * scale
    assert np.abs(logits - ref).max() < 1e-10 * np.abs(ref).max()
    from scipy.special import softmax
    assert np.abs(A - softmax(ref, axis=2)).max() < 1e-12
    assert np.allclose(A.sum(axis=2), 1.0, atol=1e-13)


# ----------------------------------------------------------------- golden
def _golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def test_golden_memory_model(orc):
    """Sec. 3.1: M = 40, D = 256 gives D/k >= 6.4."""
    for M, D, k, ratio in _golden("memory_model.txt"):
        coef, total = orc.memory_ratios(int(M), int(D), int(k))
        assert abs(coef - float(ratio)) < 1e-12
        assert total < coef


def test_golden_table3_arithmetic():
    """Table 3's printed rows are internally consistent (transcription check of
    the context numbers quoted beside the bench)."""
    for _, orig, pipe, n, per, dec, total, speed in _golden("latency_table3.txt"):
        assert abs(int(n) * float(per) - float(dec)) < 0.006
        assert abs(float(pipe) + float(dec) - float(total)) < 0.006
        assert abs(float(orig) / float(total) - float(speed)) < 0.006


# ----------------------------------------------------------------- grouped bases (Sec. 3.1, D < M)
def test_grouped_partition_closed_forms(orc):
    """D < M: each subset of at most D entries gets its own orthonormal basis (its rank
    from an independent routine), R is block diagonal, R Q = C exactly in fp64, and scores
    through the stacked basis equal X C^T."""
    rng = np.random.default_rng(20260101)
    M, D = 40, 16
    off = [0, 16, 32, 40]
    C = (rng.integers(0, 2, size=(M, D)) * 2 - 1).astype(np.float64)
    Q, R, cn, coeff = orc.build_grouped(C, off)
    assert Q.shape[0] > D  # the stacked basis is wider than the space: only the partition fits it
    for g in range(3):
        Qg = Q[coeff[g]:coeff[g + 1]]
        assert Qg.shape[0] == np.linalg.matrix_rank(C[off[g]:off[g + 1]])
        assert np.abs(Qg @ Qg.T - np.eye(Qg.shape[0])).max() <= 1e-12
        outside = np.ones(R.shape, dtype=bool)
        outside[off[g]:off[g + 1], coeff[g]:coeff[g + 1]] = False
        assert np.all(R[off[g]:off[g + 1]][outside[off[g]:off[g + 1]]] == 0.0)
    assert np.abs(R @ Q - C).max() <= 1e-12
    assert np.allclose(cn, np.linalg.norm(C, axis=1), rtol=1e-14)
    X = rng.normal(size=(9, D))
    ref = orc.project_similarity(X, Q, R, cn)
    assert np.abs(ref["S"] - X @ C.T).max() <= 1e-10
    assert np.abs(orc.reconstruct(R, Q) - C).max() <= 1e-12


def test_grouped_single_group_is_plain_build(orc, tiny_case):
    C = tiny_case[0]["C"]
    Q, R, cn, coeff = orc.build_grouped(C, [0, C.shape[0]])
    Q1, R1, cn1 = orc.build_basis(C)
    assert coeff == [0, Q1.shape[0]]
    assert np.array_equal(Q, Q1) and np.array_equal(R, R1) and np.array_equal(cn, cn1)


def test_group_argmax_brute_force(orc):
    """Per-group argmax (first index of the maximum within the group) against plain loops,
    with ties planted inside groups."""
    rng = np.random.default_rng(5)
    S = rng.integers(-3, 4, size=(7, 12)).astype(np.float64)
    S[0, 4:9] = 3.0
    S[1, 0:3] = -1.0
    off = [0, 3, 4, 9, 12]
    am, mv = orc.group_argmax(S, off)
    for n in range(S.shape[0]):
        for g in range(len(off) - 1):
            best = off[g]
            for j in range(off[g] + 1, off[g + 1]):
                if S[n, j] > S[n, best]:
                    best = j
            assert am[n, g] == best - off[g]
            assert mv[n, g] == S[n, best]


def test_grouped_attribute_codebooks(orc):
    """The four attribute codebooks in one grouped basis: the scores of each attribute's
    columns are that attribute's own X C_a^T, and the per-group argmax is the argmax against
    each codebook alone."""
    cases = synth.multiattr()
    C = np.concatenate([a["C"] for a in cases]).astype(np.float64)
    off = np.cumsum([0] + [a["C"].shape[0] for a in cases]).tolist()
    Q, R, cn, coeff = orc.build_grouped(C, off)
    assert coeff == off  # every attribute codebook has full rank
    X = cases[2]["X"][:64].astype(np.float64)
    S = orc.project_similarity(X, Q, R, cn)["S"]
    am, _ = orc.group_argmax(S, off)
    for g, a in enumerate(cases):
        Sg = X @ a["C"].astype(np.float64).T
        assert np.abs(S[:, off[g]:off[g + 1]] - Sg).max() <= 1e-9
        assert np.array_equal(am[:, g], np.argmax(Sg, axis=1))


# ----------------------------------------------------------------- binding / unbinding (Sec. 2.2, 3.3)
def _block_fft_conv(X, Y, L, correlate):
    Z = np.zeros_like(X)
    for b0 in range(0, X.shape[1], L):
        fx = np.fft.fft(X[:, b0:b0 + L], axis=1)
        fy = np.fft.fft(Y[:, b0:b0 + L], axis=1)
        Z[:, b0:b0 + L] = np.real(np.fft.ifft(fx * (np.conj(fy) if correlate else fy), axis=1))
    return Z


@pytest.mark.parametrize("L", [48, 16, 12, 1])
def test_bind_convolution_theorem(orc, L):
    """Block circular convolution / correlation against the DFT's convolution theorem."""
    rng = np.random.default_rng(L)
    X = rng.normal(size=(5, 48))
    Y = rng.normal(size=(5, 48))
    assert np.abs(orc.bind(X, Y, L, orc.BIND) - _block_fft_conv(X, Y, L, False)).max() <= 1e-12
    assert np.abs(orc.bind(X, Y, L, orc.UNBIND) - _block_fft_conv(X, Y, L, True)).max() <= 1e-12


def test_bind_algebra(orc):
    """Identity element, commutativity, and one partner broadcast over every row."""
    rng = np.random.default_rng(2)
    L, D = 16, 64
    X = rng.normal(size=(6, D))
    Y = rng.normal(size=(6, D))
    delta = np.zeros((1, D))
    delta[0, ::L] = 1.0
    assert np.array_equal(orc.bind(X, delta, L), X)
    assert np.array_equal(orc.bind(X, delta, L, orc.UNBIND), X)
    assert np.abs(orc.bind(X, Y, L) - orc.bind(Y, X, L)).max() <= 1e-12
    y1 = Y[:1]
    assert np.array_equal(orc.bind(X, y1, L), orc.bind(X, np.repeat(y1, 6, axis=0), L))


def test_unbind_inverts_unitary_binding(orc):
    """Partners whose block spectra have unit modulus: unbinding recovers the bound vector."""
    rng = np.random.default_rng(3)
    L, D = 32, 128
    Y = np.zeros((4, D))
    for b0 in range(0, D, L):
        ph = rng.uniform(-np.pi, np.pi, size=(4, L))
        spec = np.exp(1j * ph)
        spec[:, 0] = 1.0
        spec[:, L // 2] = 1.0
        spec[:, L // 2 + 1:] = np.conj(spec[:, 1:L // 2][:, ::-1])  # Hermitian: real blocks
        Y[:, b0:b0 + L] = np.real(np.fft.ifft(spec, axis=1))
    X = rng.normal(size=(4, D))
    assert np.abs(orc.bind(orc.bind(X, Y, L), Y, L, orc.UNBIND) - X).max() <= 1e-12


def test_reconstruct_bind_of_codebook(orc, tiny_case):
    """Reconstructing R gives the codebook, so binding the reconstruction is binding C."""
    t, (Q, R, _) = tiny_case
    Y = np.random.default_rng(4).normal(size=(1, Q.shape[1]))
    Z = orc.reconstruct_bind(R, Q, Y, 256)
    assert np.abs(Z - orc.bind(t["C"], Y, 256)).max() <= 1e-9
