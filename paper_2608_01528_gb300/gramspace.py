"""Thin Python binding of libgramspace.so (include/gramspace.h).

Argument marshalling only: tensors are passed to the C ABI as raw device
pointers, outputs are allocated with torch (device memory and streams are
PyTorch's plumbing), and every step of the computation runs in the library's
CUDA kernels.  There is no CPU fallback: if the library is not built, or no
sm_103 device is present, calls raise.

Names follow the C ABI (gs_ prefix dropped): build_basis, build_basis_grouped,
basis_groups, import_basis, project_similarity, project_similarity_host (with
reserve_staging), project_similarity_static, similarity_coeffs, group_argmax,
prob_vectorize, reconstruct, reconstruct_bind, bind, attention_scores,
stream_status, selftest_wait_timeout.
"""
from __future__ import annotations

import ctypes
import os

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libgramspace.so")

GS_OK, GS_ERR_INVALID_ARG, GS_ERR_ALIGNMENT, GS_ERR_SHAPE, GS_ERR_NOMEM = 0, 1, 2, 3, 4
GS_ERR_CUDA, GS_ERR_TIMEOUT, GS_ERR_RANGE, GS_ERR_UNSUPPORTED = 5, 6, 7, 8
GS_F32, GS_BF16 = 0, 1
MODES = {"raw": 0, "cosine": 1, "softmax": 2}
PATHS = {"auto": 0, "simt": 1, "tensor": 2}
GS_BUILD_NORMALIZE_ROWS = 1

# Every symbol include/gramspace.h declares (checked by the CPU tests).
EXPORTS = ("gs_build_basis", "gs_basis_info", "gs_basis_destroy", "gs_project_similarity",
           "gs_prob_vectorize", "gs_reconstruct", "gs_attention_scores", "gs_stream_status",
           "gs_status_string", "gs_version", "gs_project_similarity_static", "gs_similarity_coeffs",
           "gs_selftest_wait_timeout", "gs_basis_import", "gs_basis_reserve_staging",
           "gs_project_similarity_host", "gs_build_basis_grouped", "gs_basis_groups", "gs_group_argmax",
           "gs_bind", "gs_reconstruct_bind")


class GramSpaceError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


_lib = None


def load_library(path=LIB_PATH):
    """Loads (once) and returns the ctypes handle of libgramspace.so."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"libgramspace.so is not built ({path}); run __graft_entry__.build()")
    L = ctypes.CDLL(path)
    vp, ip, i64, f32, u32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_longlong, ctypes.c_float, ctypes.c_uint
    L.gs_build_basis.argtypes = [vp, ip, ip, ip, f32, u32, vp, ctypes.POINTER(vp)]
    L.gs_basis_info.argtypes = [vp, ctypes.POINTER(ip), ctypes.POINTER(ip), ctypes.POINTER(ip),
                                ctypes.POINTER(vp), ctypes.POINTER(vp), ctypes.POINTER(vp)]
    L.gs_basis_destroy.argtypes = [vp]
    L.gs_basis_reserve_staging.argtypes = [vp, i64]
    L.gs_project_similarity_host.argtypes = [vp, vp, i64, ip, ip, f32, u32, vp, vp, vp]
    L.gs_basis_import.argtypes = [vp, ip, ip, ip, vp, ip, ip, vp, vp, ctypes.POINTER(vp)]
    L.gs_build_basis_grouped.argtypes = [vp, ip, ip, ip, vp, ip, f32, u32, vp, ctypes.POINTER(vp)]
    L.gs_basis_groups.argtypes = [vp, ctypes.POINTER(ip), vp, vp]
    L.gs_group_argmax.argtypes = [vp, i64, ip, vp, ip, vp, vp, vp]
    L.gs_bind.argtypes = [vp, i64, ip, ip, vp, i64, ip, ip, vp, ip, vp]
    L.gs_reconstruct_bind.argtypes = [vp, vp, ip, i64, ip, vp, i64, ip, ip, vp, ip, u32, vp]
    L.gs_project_similarity.argtypes = [vp, vp, i64, ip, ip, f32, u32, vp, ip, vp, ip, vp, vp, vp]
    L.gs_similarity_coeffs.argtypes = [vp, vp, i64, ip, ip, f32, u32, vp, ip, vp, vp, vp]
    L.gs_prob_vectorize.argtypes = [vp, vp, i64, ip, vp, ip, ip, u32, vp]
    L.gs_reconstruct.argtypes = [vp, vp, ip, i64, ip, vp, ip, u32, vp]
    L.gs_attention_scores.argtypes = [vp, vp, ip, ip, ip, ip, ip, ip, f32, ip, vp, u32, vp]
    L.gs_stream_status.argtypes = [vp]
    L.gs_selftest_wait_timeout.argtypes = [vp]
    L.gs_project_similarity_static.argtypes = [vp, ip, ip, vp, ip, vp, vp, i64, ip, ip, f32, vp, vp, vp]
    L.gs_project_similarity_static.restype = ctypes.c_int
    L.gs_status_string.argtypes = [ip]
    L.gs_status_string.restype = ctypes.c_char_p
    L.gs_version.restype = ctypes.c_int
    for name in ("gs_build_basis", "gs_basis_info", "gs_basis_destroy", "gs_project_similarity",
                 "gs_similarity_coeffs", "gs_prob_vectorize", "gs_reconstruct", "gs_attention_scores",
                 "gs_stream_status", "gs_selftest_wait_timeout", "gs_basis_import",
                 "gs_basis_reserve_staging", "gs_project_similarity_host", "gs_build_basis_grouped",
                 "gs_basis_groups", "gs_group_argmax", "gs_bind", "gs_reconstruct_bind"):
        getattr(L, name).restype = ctypes.c_int
    _lib = L
    return L


def status_string(status):
    return load_library().gs_status_string(int(status)).decode()


def _check(status, where):
    if status != GS_OK:
        raise GramSpaceError(status, where)


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def _stream(stream, device=None):
    s = stream if stream is not None else torch.cuda.current_stream(device)
    return ctypes.c_void_p(s.cuda_stream)


def _ld(t):
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("expected a 2-D tensor with unit column stride")
    return t.stride(0)


def _dtype_code(t):
    if t.dtype == torch.float32:
        return GS_F32
    if t.dtype == torch.bfloat16:
        return GS_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


class _DevArray:
    """__cuda_array_interface__ view of memory owned by a basis handle."""

    def __init__(self, ptr, shape, typestr):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr,
                                         "data": (int(ptr or 0), False), "version": 3, "strides": None}


class Basis:
    """A built Gram-Space basis (owns the C handle): Q (r x D), R (M x r), cnorm (M)."""

    def __init__(self, handle, device):
        self._h = handle
        self.device = device
        L = load_library()
        M, D, r = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
        q, rr, cn = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
        _check(L.gs_basis_info(handle, ctypes.byref(M), ctypes.byref(D), ctypes.byref(r), ctypes.byref(q),
                               ctypes.byref(rr), ctypes.byref(cn)), "gs_basis_info")
        self.M, self.D, self.r = M.value, D.value, r.value
        self._q, self._R, self._cn = q.value, rr.value, cn.value

    @property
    def handle(self):
        if self._h is None:
            raise RuntimeError("basis already destroyed")
        return self._h

    def _view(self, ptr, shape):
        if 0 in shape:
            return torch.zeros(shape, dtype=torch.float32, device=self.device)
        with torch.cuda.device(self.device):
            return torch.as_tensor(_DevArray(ptr, shape, "<f4"), device=self.device)

    @property
    def Q(self):
        return self._view(self._q, (self.r, self.D))

    @property
    def R(self):
        return self._view(self._R, (self.M, self.r))

    @property
    def cnorm(self):
        return self._view(self._cn, (self.M,))

    def destroy(self):
        if self._h is not None:
            load_library().gs_basis_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def build_basis(C, rank_tol=1e-6, normalize_rows=False, stream=None):
    """Gram-Schmidt basis of the rows of C (M x D fp32 on the GPU); see gs_build_basis."""
    if not C.is_cuda or C.dtype != torch.float32:
        raise TypeError("C must be a float32 CUDA tensor")
    L = load_library()
    h = ctypes.c_void_p()
    with torch.cuda.device(C.device):
        st = L.gs_build_basis(_ptr(C), C.shape[0], C.shape[1], _ld(C), float(rank_tol),
                              GS_BUILD_NORMALIZE_ROWS if normalize_rows else 0, _stream(stream),
                              ctypes.byref(h))
    _check(st, "gs_build_basis")
    return Basis(h, C.device)


def _offsets(group_offsets):
    off = [int(o) for o in group_offsets]
    return (ctypes.c_int * len(off))(*off), len(off) - 1


def build_basis_grouped(C, group_offsets, rank_tol=1e-6, normalize_rows=False, stream=None):
    """One Gram-Schmidt basis per group of rows of C (rows [off[g], off[g+1])), stacked in one
    handle; see gs_build_basis_grouped."""
    if not C.is_cuda or C.dtype != torch.float32:
        raise TypeError("C must be a float32 CUDA tensor")
    off, G = _offsets(group_offsets)
    L = load_library()
    h = ctypes.c_void_p()
    with torch.cuda.device(C.device):
        st = L.gs_build_basis_grouped(_ptr(C), C.shape[0], C.shape[1], _ld(C), off, G, float(rank_tol),
                                      GS_BUILD_NORMALIZE_ROWS if normalize_rows else 0, _stream(stream),
                                      ctypes.byref(h))
    _check(st, "gs_build_basis_grouped")
    return Basis(h, C.device)


def basis_groups(basis):
    """(row_offsets, coeff_offsets) of the basis' groups; see gs_basis_groups."""
    L = load_library()
    G = ctypes.c_int()
    _check(L.gs_basis_groups(basis.handle, ctypes.byref(G), None, None), "gs_basis_groups")
    rows = (ctypes.c_int * (G.value + 1))()
    coeffs = (ctypes.c_int * (G.value + 1))()
    _check(L.gs_basis_groups(basis.handle, ctypes.byref(G), rows, coeffs), "gs_basis_groups")
    return list(rows), list(coeffs)


def group_argmax(S, group_offsets, want_maxval=True, out=None, stream=None):
    """Per-row, per-group argmax (index within the group) and max of scores S (N x M fp32, CUDA);
    see gs_group_argmax.  Returns {"argmax": N x G int32, "maxval": N x G fp32}."""
    if not S.is_cuda or S.dtype != torch.float32:
        raise TypeError("S must be a float32 CUDA tensor")
    off, G = _offsets(group_offsets)
    N = S.shape[0]
    out = dict(out or {})
    if "argmax" not in out:
        out["argmax"] = torch.empty((N, G), dtype=torch.int32, device=S.device)
    if want_maxval and "maxval" not in out:
        out["maxval"] = torch.empty((N, G), dtype=torch.float32, device=S.device)
    L = load_library()
    with torch.cuda.device(S.device):
        st = L.gs_group_argmax(_ptr(S), N, _ld(S) if N else S.shape[1], off, G, _ptr(out.get("argmax")),
                               _ptr(out.get("maxval")), _stream(stream))
    _check(st, "gs_group_argmax")
    return out


def import_basis(Q, R, cnorm=None, stream=None):
    """Restore a basis saved from Basis.Q / Basis.R / Basis.cnorm (fp32 CUDA tensors, Q: r x D,
    R: M x r); see gs_basis_import.  The restored basis gives bit-identical results."""
    for t in (Q, R) + ((cnorm,) if cnorm is not None else ()):
        if not t.is_cuda or t.dtype != torch.float32:
            raise TypeError("Q, R and cnorm must be float32 CUDA tensors")
    r, D = Q.shape
    M = R.shape[0]
    L = load_library()
    h = ctypes.c_void_p()
    with torch.cuda.device(R.device):
        st = L.gs_basis_import(_ptr(Q) if r else None, r, D, _ld(Q) if r else D, _ptr(R) if r else None, M,
                               _ld(R) if r else 1, _ptr(cnorm), _stream(stream), ctypes.byref(h))
    _check(st, "gs_basis_import")
    return Basis(h, R.device)


def reserve_staging(basis, rows):
    """Device staging for project_similarity_host (rows queries); see gs_basis_reserve_staging."""
    L = load_library()
    with torch.cuda.device(basis.device):
        _check(L.gs_basis_reserve_staging(basis.handle, int(rows)), "gs_basis_reserve_staging")


def project_similarity_host(basis, X, mode="raw", scale=1.0, path="auto", want_argmax=True, want_maxval=True,
                            out=None, stream=None):
    """Project + similarity of host queries X (N x D float32 CPU tensor, ideally pinned) into host
    outputs; see gs_project_similarity_host.  Asynchronous on `stream`: synchronise before reading
    the outputs, and keep X referenced (and unchanged) until then -- a pinned tensor freed earlier
    returns its block to torch's host allocator, which can reuse it while the copy is queued."""
    if X.is_cuda or X.dtype != torch.float32:
        raise TypeError("X must be a float32 CPU tensor")
    if X.dim() != 2 or X.shape[1] != basis.D:
        raise ValueError(f"X must be N x {basis.D}")
    N = X.shape[0]
    out = dict(out or {})
    pin = X.is_pinned()
    if want_argmax and "argmax" not in out:
        out["argmax"] = torch.empty(N, dtype=torch.int32, pin_memory=pin)
    if want_maxval and "maxval" not in out:
        out["maxval"] = torch.empty(N, dtype=torch.float32, pin_memory=pin)
    L = load_library()
    with torch.cuda.device(basis.device):
        st = L.gs_project_similarity_host(basis.handle, _ptr(X), N, _ld(X), MODES[mode], float(scale),
                                          PATHS[path], _ptr(out.get("argmax")), _ptr(out.get("maxval")),
                                          _stream(stream))
    _check(st, "gs_project_similarity_host")
    return out


def project_similarity(basis, X, mode="raw", scale=1.0, path="auto", want_Y=False, want_S=False,
                       want_argmax=True, want_maxval=True, out=None, stream=None):
    """Fused Y = X Q^T and scores against the codebook in Gram-loc; see gs_project_similarity.

    Returns a dict with the requested outputs ("Y", "S", "argmax", "maxval").
    `out` may supply preallocated output tensors under the same keys.
    """
    N = X.shape[0]
    dev = X.device
    out = dict(out or {})
    if want_Y and "Y" not in out:
        out["Y"] = torch.empty((N, basis.r), dtype=torch.float32, device=dev)
    if want_S and "S" not in out:
        out["S"] = torch.empty((N, basis.M), dtype=torch.float32, device=dev)
    if want_argmax and "argmax" not in out:
        out["argmax"] = torch.empty(N, dtype=torch.int32, device=dev)
    if want_maxval and "maxval" not in out:
        out["maxval"] = torch.empty(N, dtype=torch.float32, device=dev)
    Y, S = out.get("Y"), out.get("S")
    L = load_library()
    # the handle's calls switch to the basis' device themselves: only the stream is looked up here
    st = L.gs_project_similarity(basis.handle, _ptr(X), N, _ld(X), MODES[mode], float(scale), PATHS[path],
                                 _ptr(Y), _ld(Y) if Y is not None and Y.numel() else max(basis.r, 1),
                                 _ptr(S), _ld(S) if S is not None and S.numel() else max(basis.M, 1),
                                 _ptr(out.get("argmax")), _ptr(out.get("maxval")), _stream(stream, dev))
    _check(st, "gs_project_similarity")
    return out


def similarity_coeffs(basis, Y, mode="raw", scale=1.0, path="auto", want_S=False, want_argmax=True,
                      want_maxval=True, out=None, stream=None):
    """Scores of Gram-loc queries Y (N x r fp32) against the codebook, S = Y R^T; see
    gs_similarity_coeffs.  Returns a dict with the requested outputs ("S", "argmax", "maxval")."""
    N = Y.shape[0]
    dev = Y.device
    out = dict(out or {})
    if want_S and "S" not in out:
        out["S"] = torch.empty((N, basis.M), dtype=torch.float32, device=dev)
    if want_argmax and "argmax" not in out:
        out["argmax"] = torch.empty(N, dtype=torch.int32, device=dev)
    if want_maxval and "maxval" not in out:
        out["maxval"] = torch.empty(N, dtype=torch.float32, device=dev)
    S = out.get("S")
    L = load_library()
    st = L.gs_similarity_coeffs(basis.handle, _ptr(Y) if Y.numel() else None, N,
                                _ld(Y) if Y.numel() else max(basis.r, 1), MODES[mode], float(scale),
                                PATHS[path], _ptr(S), _ld(S) if S is not None and S.numel() else max(basis.M, 1),
                                _ptr(out.get("argmax")), _ptr(out.get("maxval")), _stream(stream, dev))
    _check(st, "gs_similarity_coeffs")
    return out


def prob_vectorize(basis, P, dtype=torch.float32, path="auto", out=None, stream=None):
    """V = P R (Gram-loc of P C); see gs_prob_vectorize."""
    N = P.shape[0]
    V = out if out is not None else torch.empty((N, basis.r), dtype=dtype, device=P.device)
    L = load_library()
    with torch.cuda.device(P.device):
        st = L.gs_prob_vectorize(basis.handle, _ptr(P), N, _ld(P), _ptr(V), _dtype_code(V),
                                 _ld(V) if V.numel() else max(basis.r, 1), PATHS[path], _stream(stream))
    _check(st, "gs_prob_vectorize")
    return V


def reconstruct(basis, T, path="auto", out=None, stream=None):
    """Xhat = T Q (x = U t); see gs_reconstruct."""
    N = T.shape[0]
    X = out if out is not None else torch.empty((N, basis.D), dtype=torch.float32, device=T.device)
    L = load_library()
    with torch.cuda.device(T.device):
        st = L.gs_reconstruct(basis.handle, _ptr(T), _dtype_code(T), N, _ld(T) if T.numel() else max(basis.r, 1),
                              _ptr(X), _ld(X), PATHS[path], _stream(stream))
    _check(st, "gs_reconstruct")
    return X


BIND_OPS = {"bind": 0, "unbind": 1}
BIND_METHODS = {"auto": 0, "direct": 2, "spectral": 4}


def _partner(Y, N, D):
    if not Y.is_cuda or Y.dtype != torch.float32 or Y.dim() != 2 or Y.shape[1] != D:
        raise ValueError(f"Y must be a float32 CUDA tensor with {D} columns")
    if Y.shape[0] == 1 and N != 1:
        return 0  # one partner for every row
    if Y.shape[0] != N:
        raise ValueError("Y must have one row or one row per input row")
    return _ld(Y)


def bind(X, Y, L, op="bind", method="auto", out=None, stream=None):
    """Block circular convolution (op="bind") or correlation ("unbind") of the rows of X with
    those of Y (or with Y's single row), blocks of L; method "direct" (the sum per output),
    "spectral" (block transforms) or "auto"; see gs_bind."""
    N, D = X.shape
    ldy = _partner(Y, N, D)
    Z = out if out is not None else torch.empty((N, D), dtype=torch.float32, device=X.device)
    L_ = load_library()
    with torch.cuda.device(X.device):
        st = L_.gs_bind(_ptr(X), N, D, _ld(X) if N else D, _ptr(Y), ldy, int(L), BIND_OPS[op] | BIND_METHODS[method],
                        _ptr(Z), _ld(Z) if N else D, _stream(stream))
    _check(st, "gs_bind")
    return Z


def reconstruct_bind(basis, T, Y, L, op="bind", path="auto", method="auto", out=None, stream=None):
    """op(T Q, Y): reconstruction then binding, chunk by chunk through the basis' scratch; see gs_reconstruct_bind
    (path: the reconstruction's kernels, method: the binding's, as in bind)."""
    N = T.shape[0]
    ldy = _partner(Y, N, basis.D)
    Z = out if out is not None else torch.empty((N, basis.D), dtype=torch.float32, device=T.device)
    L_ = load_library()
    with torch.cuda.device(basis.device):
        st = L_.gs_reconstruct_bind(basis.handle, _ptr(T), _dtype_code(T), N, _ld(T) if N else basis.r, _ptr(Y),
                                    ldy, int(L), BIND_OPS[op] | BIND_METHODS[method], _ptr(Z),
                                    _ld(Z) if N else basis.D, PATHS[path], _stream(stream))
    _check(st, "gs_reconstruct_bind")
    return Z


def attention_scores(Yq, Yk, scale, apply_softmax=True, path="auto", out=None, stream=None):
    """softmax_row(scale * Yq Yk^T) per sequence; Yq: B x Lq x r, Yk: B x Lk x r."""
    B, Lq, r = Yq.shape
    Lk = Yk.shape[1]
    if Yk.shape[0] != B or Yk.shape[2] != r or Yq.dtype != Yk.dtype:
        raise ValueError("Yq and Yk must agree in batch, width and dtype")
    if not (Yq.is_contiguous() and Yk.is_contiguous()):
        raise ValueError("Yq and Yk must be contiguous (row stride r)")
    A = out if out is not None else torch.empty((B, Lq, Lk), dtype=torch.float32, device=Yq.device)
    L = load_library()
    with torch.cuda.device(Yq.device):
        st = L.gs_attention_scores(_ptr(Yq), _ptr(Yk), _dtype_code(Yq), B, Lq, Lk, r, max(r, 1), float(scale),
                                   1 if apply_softmax else 0, _ptr(A), PATHS[path], _stream(stream))
    _check(st, "gs_attention_scores")
    return A


def project_similarity_static(Q, R, cnorm, X, mode="raw", scale=1.0, want_argmax=True, want_maxval=True,
                              out=None, stream=None):
    """Project + similarity from a caller-held basis without any device allocation by the
    library; see gs_project_similarity_static.  Q: r x D, R: M x r, cnorm: M (fp32, CUDA)."""
    # the C entry takes ld(Q) = D and ld(R) = r and reads cnorm[0..M): every shape is checked here,
    # before any pointer reaches the library
    if Q.dim() != 2 or R.dim() != 2 or X.dim() != 2 or cnorm.dim() != 1:
        raise ValueError("Q, R, X must be 2-D and cnorm 1-D")
    N = X.shape[0]
    r, D = Q.shape
    M = R.shape[0]
    if R.shape[1] != r:
        raise ValueError(f"R must be M x r with r = {r} (Q's rows), got {tuple(R.shape)}")
    if X.shape[1] != D:
        raise ValueError(f"X must be N x {D} (Q's columns), got {tuple(X.shape)}")
    if cnorm.shape[0] != M:
        raise ValueError(f"cnorm must hold M = {M} entries, got {cnorm.shape[0]}")
    for t in (Q, R):
        if t.numel() and not t.is_contiguous():
            raise ValueError("Q and R must be contiguous")
    out = dict(out or {})
    for key, dt in (("argmax", torch.int32), ("maxval", torch.float32)):
        t = out.get(key)
        if t is not None and (t.dtype != dt or t.dim() != 1 or t.shape[0] != N or not t.is_contiguous()):
            raise ValueError(f"out[{key!r}] must be a contiguous {dt} vector of N = {N} entries")
    for name, t in (("Q", Q), ("R", R), ("cnorm", cnorm), ("X", X)):
        if t.dtype != torch.float32:
            raise TypeError(f"{name} must be float32, got {t.dtype}")
    tensors = [Q, R, cnorm, X] + [t for t in out.values() if t is not None]
    if any(not t.is_cuda for t in tensors) or len({t.device for t in tensors}) != 1:
        raise TypeError("Q, R, cnorm, X and the outputs must be CUDA tensors on one device")
    if want_argmax and "argmax" not in out:
        out["argmax"] = torch.empty(N, dtype=torch.int32, device=X.device)
    if want_maxval and "maxval" not in out:
        out["maxval"] = torch.empty(N, dtype=torch.float32, device=X.device)
    L = load_library()
    with torch.cuda.device(X.device):
        st = L.gs_project_similarity_static(_ptr(Q) if Q.numel() else None, r, D, _ptr(R) if R.numel() else None,
                                            M, _ptr(cnorm), _ptr(X), N, _ld(X), MODES[mode], float(scale),
                                            _ptr(out.get("argmax")), _ptr(out.get("maxval")), _stream(stream))
    _check(st, "gs_project_similarity_static")
    return out


def stream_status(stream=None):
    """Synchronises and raises GramSpaceError if the device recorded an error."""
    L = load_library()
    st = L.gs_stream_status(_stream(stream) if stream is not False else None)
    _check(st, "gs_stream_status")


def selftest_wait_timeout(stream=None):
    """Enqueue a block whose bounded wait runs out (~2 s); see gs_selftest_wait_timeout.
    stream_status() afterwards raises GramSpaceError with GS_ERR_TIMEOUT."""
    _check(load_library().gs_selftest_wait_timeout(_stream(stream)), "gs_selftest_wait_timeout")
