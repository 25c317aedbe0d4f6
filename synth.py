"""Seeded synthetic inputs shaped like the paper's multi-attribute reasoning workloads.

This module only draws random numbers: it holds none of the Gram-Space
arithmetic, so both the CUDA path and the float64 oracle can take their inputs
from it.  The paper's datasets (RAVEN / I-RAVEN, Sec. 1 and Sec. 3.1) are not
available; these generators stand in for their shapes only (4 attributes of
aligned size ~10 give M = 40 in Sec. 3.1; codebooks are pseudorandom bipolar or
binary atoms, Sec. 2.1).

Large query matrices are drawn in blocks of ``BLOCK`` rows, each from its own
``numpy.random.default_rng([seed, stream, block])``, so any row range can be
regenerated on its own (the parity tests check sampled rows of the full-size
workloads against the oracle without holding the oracle's copy of everything).

Workloads (all float32 unless stated):
  tiny       M=8 bipolar, D=1024; 64 queries = codeword + N(0, 0.5^2); 64
             Dirichlet(1) probability rows.
  multiattr  4 bipolar codebooks M = 5, 6, 10, 9, D = 1024; per attribute 512
             queries (32 problems x 16 panels): p = softmax(N(0, 2^2) logits),
             x = p C + N(0, 0.1^2).
  large      M=256 bipolar, D=8192; 65,536 queries = codeword + N(0, 1).
  rankdef    M=1024, D=10,000: 922 Bernoulli(0.5) {0,1} rows and 102 dependent
             rows (half duplicates of a random independent row, half s1*a + s2*b
             with s in {-1, +1} and a != b independent), rows shuffled; rank 922.
             16,384 queries = random row + N(0, 1).
  attention  M=512 bipolar, D=4096; 64 sequences x 1024 tokens of query and key
             probability rows p = softmax(N(0, 1) logits over M) (keys from an
             independent stream).
"""
from __future__ import annotations

import numpy as np

BLOCK = 256
SEEDS = {"tiny": 20260001, "multiattr": 20260002, "large": 20260003,
         "rankdef": 20260004, "attention": 20260005, "sweep": 20260006}
SWEEP_D = (256, 512, 1024, 2048, 4096, 8192)
MULTIATTR_M = (5, 6, 10, 9)


def _rng(seed, *stream):
    return np.random.default_rng([int(seed), *[int(s) for s in stream]])


def bipolar(rng, M, D):
    """M x D matrix of i.i.d. +-1 entries (float32)."""
    return (rng.integers(0, 2, size=(M, D), dtype=np.int8) * 2 - 1).astype(np.float32)


def softmax_rows(logits):
    """Row-wise softmax in float64 (the generators' own helper for drawing
    probability vectors; not part of the method under test)."""
    z = logits - logits.max(axis=1, keepdims=True)
    e = np.exp(z)
    return e / e.sum(axis=1, keepdims=True)


# --------------------------------------------------------------------------- tiny
def tiny(seed=SEEDS["tiny"], M=8, D=1024, N=64):
    rng = _rng(seed, 0)
    C = bipolar(rng, M, D)
    labels = rng.integers(0, M, size=N)
    X = (C[labels].astype(np.float64) + rng.normal(0.0, 0.5, size=(N, D))).astype(np.float32)
    P = rng.dirichlet(np.ones(M), size=N).astype(np.float32)
    return {"C": C, "X": X, "labels": labels.astype(np.int64), "P": P}


# ---------------------------------------------------------------------- multiattr
def multiattr(seed=SEEDS["multiattr"], D=1024, problems=32, panels=16, Ms=MULTIATTR_M):
    out = []
    N = problems * panels
    for a, M in enumerate(Ms):
        rng = _rng(seed, a)
        C = bipolar(rng, M, D)
        P = softmax_rows(rng.normal(0.0, 2.0, size=(N, M)))
        X = P @ C.astype(np.float64) + rng.normal(0.0, 0.1, size=(N, D))
        out.append({"C": C, "X": X.astype(np.float32), "P": P.astype(np.float32),
                    "labels": P.argmax(axis=1).astype(np.int64)})
    return out


# --------------------------------------------------------- noisy-codeword queries
def noisy_rows(C, seed, i0, i1, sigma, stream=1):
    """Rows [i0, i1) of the query matrix x_n = C[k_n] + N(0, sigma^2), drawn block by
    block so that any range regenerates identically.  Returns (X, labels)."""
    M, D = C.shape
    b0, b1 = i0 // BLOCK, (i1 + BLOCK - 1) // BLOCK
    xs, ls = [], []
    for b in range(b0, b1):
        rng = _rng(seed, stream, b)
        lab = rng.integers(0, M, size=BLOCK)
        noise = rng.standard_normal(size=(BLOCK, D), dtype=np.float32)
        if sigma != 1.0:
            noise *= np.float32(sigma)
        noise += C[lab]
        xs.append(noise)
        ls.append(lab)
    X = np.concatenate(xs)[i0 - b0 * BLOCK:i1 - b0 * BLOCK]
    L = np.concatenate(ls)[i0 - b0 * BLOCK:i1 - b0 * BLOCK]
    return np.ascontiguousarray(X), L.astype(np.int64)


def large_codebook(seed=SEEDS["large"], M=256, D=8192):
    return bipolar(_rng(seed, 0), M, D)


def large(seed=SEEDS["large"], M=256, D=8192, N=65536, rows=None):
    """The large-batch similarity workload.  rows=(i0, i1) draws only that range."""
    C = large_codebook(seed, M, D)
    i0, i1 = rows if rows is not None else (0, N)
    X, L = noisy_rows(C, seed, i0, i1, 1.0)
    return {"C": C, "X": X, "labels": L, "N": N}


# ------------------------------------------------------------------------ rankdef
def rankdef_codebook(seed=SEEDS["rankdef"], M=1024, D=10000, n_dep=None):
    rng = _rng(seed, 0)
    if n_dep is None:
        n_dep = M // 10
    n_ind = M - n_dep
    ind = rng.integers(0, 2, size=(n_ind, D), dtype=np.int8).astype(np.float32)
    dep = np.empty((n_dep, D), dtype=np.float32)
    for t in range(n_dep):
        if rng.random() < 0.5:
            dep[t] = ind[rng.integers(0, n_ind)]
        else:
            a, b = rng.choice(n_ind, size=2, replace=False)
            s1, s2 = rng.choice([-1.0, 1.0], size=2)
            dep[t] = s1 * ind[a] + s2 * ind[b]
    C = np.concatenate([ind, dep])
    perm = rng.permutation(M)
    return np.ascontiguousarray(C[perm]), n_ind


def rankdef(seed=SEEDS["rankdef"], M=1024, D=10000, N=16384, rows=None):
    C, rank = rankdef_codebook(seed, M, D)
    i0, i1 = rows if rows is not None else (0, N)
    X, L = noisy_rows(C, seed, i0, i1, 1.0)
    return {"C": C, "X": X, "labels": L, "rank": rank, "N": N}


# ---------------------------------------------------------------------- attention
def attention_probs(seed, B, L, M, stream):
    """B*L probability rows over M codewords, p = softmax(N(0,1) logits)."""
    rng = _rng(seed, stream)
    return softmax_rows(rng.standard_normal(size=(B * L, M))).astype(np.float32)


def attention(seed=SEEDS["attention"], M=512, D=4096, B=64, L=1024):
    C = bipolar(_rng(seed, 0), M, D)
    Pq = attention_probs(seed, B, L, M, 1)
    Pk = attention_probs(seed, B, L, M, 101)
    return {"C": C, "Pq": Pq, "Pk": Pk, "B": B, "L": L, "D": D}


def sweep(D, seed=SEEDS["sweep"], M=40, N=1024, sigma=0.5):
    """Lookup-latency sweep over the original dimension: a bipolar global codebook of
    M = 40 attribute vectors (the paper's memory-model example) at dimension D, and a
    batch of N random attribute lookups x = c_k + N(0, sigma^2)."""
    C = bipolar(_rng(seed, 0, D), M, D)
    X, L = noisy_rows(C, seed + D, 0, N, sigma)
    return {"C": C, "X": X, "labels": L, "D": D}
