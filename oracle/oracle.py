"""ctypes front end of the float64 oracle (gs_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and
bench.py's cpu_baseline / reference arm.  It never imports the CUDA package
and the CUDA package never imports it.

Every function takes numpy arrays (any float dtype; converted to float64) and
returns float64 results.  See gs_oracle.c for the paper passages each step
follows and for the readings of the paper it fixes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "gs_oracle.c")
LIB = os.path.join(HERE, "_build", "liboracle.so")

RAW, COSINE, SOFTMAX = 0, 1, 2

_lib = None


def build(force=False):
    """Compile gs_oracle.c into oracle/_build/liboracle.so (OpenMP when gcc has it)."""
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", SRC, "-lm", "-o", LIB]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    return LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(LIB)
        dp = ctypes.POINTER(ctypes.c_double)
        ip = ctypes.POINTER(ctypes.c_int)
        L.orc_build_mgs.restype = ctypes.c_int
        L.orc_build_mgs.argtypes = [dp, ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_int,
                                    ctypes.c_int, dp, dp, ctypes.c_int, dp]
        L.orc_project.argtypes = [dp, ctypes.c_long, ctypes.c_int, ctypes.c_int, dp, ctypes.c_int, dp, dp]
        L.orc_similarity.argtypes = [dp, ctypes.c_long, ctypes.c_int, dp, ctypes.c_int, ctypes.c_int,
                                     ctypes.c_int, ctypes.c_double, dp, dp, dp, ip, dp]
        L.orc_prob_vectorize.argtypes = [dp, ctypes.c_long, ctypes.c_int, ctypes.c_int, dp, ctypes.c_int,
                                         ctypes.c_int, dp]
        L.orc_reconstruct.argtypes = [dp, ctypes.c_long, ctypes.c_int, ctypes.c_int, dp, ctypes.c_int, dp]
        L.orc_attention.argtypes = [dp, dp, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                    ctypes.c_double, ctypes.c_int, dp]
        L.orc_memory_ratios.argtypes = [ctypes.c_long, ctypes.c_long, ctypes.c_long, dp]
        L.orc_bind.argtypes = [dp, ctypes.c_long, ctypes.c_int, ctypes.c_int, dp, ctypes.c_long, ctypes.c_int,
                               ctypes.c_int, dp]
        L.orc_num_threads.restype = ctypes.c_int
        L.orc_set_num_threads.argtypes = [ctypes.c_int]
        _lib = L
    return _lib


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _p(a):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double)) if a is not None else None


def num_threads():
    return lib().orc_num_threads()


def set_num_threads(n):
    lib().orc_set_num_threads(int(n))


def build_basis(C, tau=1e-6, normalize_rows=False, passes=2):
    """MGS with reorthogonalisation (Sec. 3.1, Eq. 1).  Returns (Q r x D, R M x r, cnorm M)."""
    C = _f64(C)
    M, D = C.shape
    rmax = max(1, min(M, D))
    Q = np.zeros((rmax, D))
    R = np.zeros((M, rmax))
    cn = np.zeros(M)
    r = lib().orc_build_mgs(_p(C), M, D, float(tau), int(bool(normalize_rows)), int(passes),
                            _p(Q), _p(R), rmax, _p(cn))
    if r < 0:
        raise MemoryError("oracle build failed")
    return Q[:r].copy(), np.ascontiguousarray(R[:, :r]), cn


def build_grouped(C, offsets, tau=1e-6, normalize_rows=False):
    """Sec. 3.1, D < M: the entries are partitioned into subsets (rows [offsets[g],
    offsets[g+1]) of C), each subset gets its own orthonormal basis, and the
    reconstructions are concatenated.  Returns (Q, R, cnorm, coeff_offsets): Q stacks the
    subsets' bases (r = sum of their ranks rows), R is block diagonal (subset g's
    coefficients in columns [coeff_offsets[g], coeff_offsets[g+1])), so C = R Q."""
    C = _f64(C)
    M, D = C.shape
    parts = [build_basis(C[offsets[g]:offsets[g + 1]], tau, normalize_rows) for g in range(len(offsets) - 1)]
    coeff = [0]
    for Qg, _, _ in parts:
        coeff.append(coeff[-1] + Qg.shape[0])
    Q = np.zeros((coeff[-1], D))
    R = np.zeros((M, coeff[-1]))
    cn = np.zeros(M)
    for g, (Qg, Rg, cng) in enumerate(parts):
        Q[coeff[g]:coeff[g + 1]] = Qg
        R[offsets[g]:offsets[g + 1], coeff[g]:coeff[g + 1]] = Rg
        cn[offsets[g]:offsets[g + 1]] = cng
    return Q, R, cn, coeff


def group_argmax(S, offsets):
    """Best entry of each group (columns [offsets[g], offsets[g+1])) for each row of S:
    (argmax within the group, first index of the maximum; maximum), each N x G."""
    S = _f64(S)
    G = len(offsets) - 1
    am = np.zeros((S.shape[0], G), dtype=np.int32)
    mv = np.zeros((S.shape[0], G))
    for g in range(G):
        block = S[:, offsets[g]:offsets[g + 1]]
        am[:, g] = np.argmax(block, axis=1)
        mv[:, g] = block.max(axis=1)
    return am, mv


def project(X, Q):
    """Y = X Q^T (Gram-loc of each query, Sec. 3.1) and the full-D norms ||x||."""
    X = _f64(X)
    Q = _f64(Q)
    N, D = X.shape
    r = Q.shape[0]
    Y = np.zeros((N, r))
    xn = np.zeros(N)
    lib().orc_project(_p(X), N, D, D, _p(Q) if r else None, r, _p(Y), _p(xn))
    return Y, xn


def similarity(Y, R, mode=RAW, scale=1.0, xnorm=None, cnorm=None):
    """Scores in Gram-loc (Sec. 2.2, Eq. 2-3).  Returns (S, argmax, maxval)."""
    Y = _f64(Y)
    R = _f64(R)
    N, r = Y.shape
    M = R.shape[0]
    if mode == COSINE and (xnorm is None or cnorm is None):
        raise ValueError("cosine scores need xnorm and cnorm")
    xn = _f64(xnorm) if xnorm is not None else None
    cn = _f64(cnorm) if cnorm is not None else None
    S = np.zeros((N, M))
    am = np.zeros(N, dtype=np.int32)
    mv = np.zeros(N)
    Rp = R if r > 0 else np.zeros((M, 1))
    Yp = Y if r > 0 else np.zeros((N, 1))
    lib().orc_similarity(_p(Yp), N, r, _p(Rp), max(r, 1), M, int(mode), float(scale), _p(xn), _p(cn),
                         _p(S), am.ctypes.data_as(ctypes.POINTER(ctypes.c_int)), _p(mv))
    return S, am.astype(np.int64), mv


def project_similarity(X, Q, R, cnorm, mode=RAW, scale=1.0):
    Y, xn = project(X, Q)
    S, am, mv = similarity(Y, R, mode, scale, xn, cnorm)
    return {"Y": Y, "S": S, "argmax": am, "maxval": mv, "xnorm": xn}


def prob_vectorize(P, R):
    """V = P R (probability vectorization on Gram-loc, Sec. 2.2 / Sec. 3.3)."""
    P = _f64(P)
    R = _f64(R)
    N, M = P.shape
    r = R.shape[1]
    V = np.zeros((N, r))
    if r:
        lib().orc_prob_vectorize(_p(P), N, M, M, _p(R), r, r, _p(V))
    return V


def reconstruct(T, Q):
    """Xhat = T Q (x = U t, Sec. 3.1 / Sec. 3.3)."""
    T = _f64(T)
    Q = _f64(Q)
    N, r = T.shape
    D = Q.shape[1]
    X = np.zeros((N, D))
    if r:
        lib().orc_reconstruct(_p(T), N, r, r, _p(Q), D, _p(X))
    return X


def attention(Yq, Yk, B, Lq, Lk, scale, apply_softmax=True):
    """Attention scores between Gram-loc vectors (Sec. 2.2, Sec. 3.2)."""
    Yq = _f64(Yq).reshape(B * Lq, -1)
    Yk = _f64(Yk).reshape(B * Lk, -1)
    r = Yq.shape[1]
    A = np.zeros((B, Lq, Lk))
    lib().orc_attention(_p(Yq), _p(Yk), B, Lq, Lk, r, float(scale), int(bool(apply_softmax)), _p(A))
    return A


BIND, UNBIND = 0, 1


def bind(X, Y, L, op=BIND):
    """Block circular convolution (bind) or correlation (unbind) of the rows of X with the rows
    of Y (or with Y's single row for every row of X), blocks of L components (Sec. 2.2, 3.3)."""
    X = _f64(X)
    Y = _f64(Y)
    N, D = X.shape
    if D % L:
        raise ValueError("L must divide D")
    ldy = 0 if Y.shape[0] == 1 and N != 1 else D
    Z = np.zeros((N, D))
    lib().orc_bind(_p(X), N, D, D, _p(Y), ldy, int(L), int(op), _p(Z))
    return Z


def reconstruct_bind(T, Q, Y, L, op=BIND):
    """Bind (or unbind) reconstructed rows x = t Q with Y: the reconstruction at the transition
    into component-wise operators, then the operator (Sec. 3.3)."""
    return bind(reconstruct(T, Q), Y, L, op)


def memory_ratios(M, D, k):
    """(D/k, M*D/(D*k + M*k)) -- the memory model of Sec. 3.1."""
    out = np.zeros(2)
    lib().orc_memory_ratios(int(M), int(D), int(k), _p(out))
    return float(out[0]), float(out[1])
