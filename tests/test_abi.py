"""Host-side checks of the C-ABI library that need no GPU: it loads, exports
every symbol include/gramspace.h declares, and its status strings work."""
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gramspace.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_01528_gb300 import build, gramspace
    build.build()
    return gramspace.load_library()


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"GS_API\s+[\w\s\*]*?\b(gs_\w+)\s*\(", text)))


def test_header_declares_the_five_operations():
    names = declared_symbols()
    for op in ("gs_build_basis", "gs_project_similarity", "gs_prob_vectorize", "gs_reconstruct",
               "gs_attention_scores"):
        assert op in names


def test_library_exports_every_declared_symbol(lib):
    from paper_2608_01528_gb300 import gramspace
    names = declared_symbols()
    assert sorted(gramspace.EXPORTS) == names
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings_and_version(lib):
    from paper_2608_01528_gb300 import gramspace
    assert gramspace.status_string(0) == "GS_OK"
    assert gramspace.status_string(7) == "GS_ERR_RANGE"
    assert gramspace.status_string(99) == "GS_ERR_UNKNOWN"
    assert lib.gs_version() >= 100


def test_host_side_argument_checks_need_no_device(lib):
    """Invalid arguments are rejected on the host before any CUDA call."""
    import ctypes
    from paper_2608_01528_gb300 import gramspace as g
    h = ctypes.c_void_p()
    assert lib.gs_build_basis(None, 4, 4, 4, 1e-6, 0, None, None) == g.GS_ERR_INVALID_ARG
    assert lib.gs_build_basis(None, 0, 4, 4, 1e-6, 0, None, ctypes.byref(h)) == g.GS_ERR_SHAPE
    assert lib.gs_project_similarity(None, None, 1, 1, 0, 1.0, 0, None, 0, None, 0, None, None,
                                     None) == g.GS_ERR_INVALID_ARG
    assert lib.gs_attention_scores(None, None, 5, 1, 1, 1, 1, 1, 1.0, 1, None, 0, None) == g.GS_ERR_INVALID_ARG
    assert lib.gs_attention_scores(None, None, 0, 1, 1, 1, 4, 2, 1.0, 1, None, 0, None) == g.GS_ERR_SHAPE
    assert lib.gs_attention_scores(None, None, 0, 0, 4, 4, 4, 4, 1.0, 1, None, 0, None) == g.GS_OK


def test_bind_argument_checks_need_no_device(lib):
    """gs_bind rejects unknown operator bits, both methods at once and inconsistent shapes on
    the host; N = 0 is a no-op."""
    from paper_2608_01528_gb300 import gramspace as g
    dummy = 16  # never dereferenced: every call below returns before touching memory
    for op in (8, g.BIND_METHODS["direct"] | g.BIND_METHODS["spectral"], -1):
        assert lib.gs_bind(dummy, 4, 100, 100, dummy, 100, 50, op, dummy, 100, None) == g.GS_ERR_INVALID_ARG
    assert lib.gs_bind(dummy, 4, 100, 100, dummy, 100, 30, 0, dummy, 100, None) == g.GS_ERR_SHAPE  # L | D
    assert lib.gs_bind(dummy, 4, 100, 99, dummy, 100, 50, 0, dummy, 100, None) == g.GS_ERR_SHAPE  # ldx < D
    assert lib.gs_bind(dummy, 4, 100, 100, dummy, 60, 50, 0, dummy, 100, None) == g.GS_ERR_SHAPE  # 0 < ldy < D
    assert lib.gs_bind(dummy, 0, 100, 100, dummy, 0, 50, g.BIND_METHODS["spectral"], dummy, 100,
                       None) == g.GS_OK
    assert lib.gs_bind(None, 4, 100, 100, None, 0, 50, 0, None, 100, None) == g.GS_ERR_INVALID_ARG


def test_plain_c_client(lib, tmp_path):
    """The header is plain C (C99, -pedantic, no warnings) and a C program links against the
    library and calls it: the boundary needs no C++ or torch on the caller's side."""
    import shutil
    import subprocess
    from paper_2608_01528_gb300 import build
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "client.c"
    src.write_text(
        "#include <stdio.h>\n"
        "#include \"gramspace.h\"\n"
        "int main(void) {\n"
        "    printf(\"%d %s\\n\", gs_version(), gs_status_string(GS_ERR_SHAPE));\n"
        "    /* L = 30 does not divide D = 100: rejected on the host */\n"
        "    return gs_bind(0, 4, 100, 100, 0, 0, 30, GS_BIND | GS_BIND_DIRECT, 0, 100, 0) == GS_ERR_SHAPE ? 0 : 1;\n"
        "}\n")
    exe = tmp_path / "client"
    libdir = os.path.dirname(build.LIB)
    p = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I",
                        os.path.join(ROOT, "include"), str(src), "-L", libdir, "-lgramspace",
                        f"-Wl,-rpath,{libdir}", "-o", str(exe)], capture_output=True, text=True)
    assert p.returncode == 0, p.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    assert r.stdout.split()[1] == "GS_ERR_SHAPE"


def test_static_entry_wrapper_rejects_mismatched_tensors():
    """project_similarity_static checks shapes, dtypes and devices before any pointer reaches the
    library: the C entry assumes ld(Q) = D, ld(R) = r and M norms, so a mismatch there would read
    or write past a buffer on the device.  CPU tensors reach no CUDA call."""
    import torch
    from paper_2608_01528_gb300 import gramspace as g
    r, D, M, N = 4, 16, 6, 3
    Q, R, cn, X = torch.zeros(r, D), torch.zeros(M, r), torch.zeros(M), torch.zeros(N, D)
    bad_shapes = [
        (Q, torch.zeros(M, r + 1), cn, X),   # R wider than r
        (Q, R, cn, torch.zeros(N, D - 1)),   # X narrower than D
        (Q, R, torch.zeros(M - 1), X),       # too few norms
        (Q.reshape(-1), R, cn, X),           # Q not 2-D
    ]
    for args in bad_shapes:
        with pytest.raises(ValueError):
            g.project_similarity_static(*args)
    with pytest.raises(ValueError):
        g.project_similarity_static(Q, R, cn, X, out={"argmax": torch.zeros(N - 1, dtype=torch.int32)})
    with pytest.raises(ValueError):
        g.project_similarity_static(Q, R, cn, X, out={"maxval": torch.zeros(N, dtype=torch.float64)})
    with pytest.raises(TypeError):
        g.project_similarity_static(Q, R, cn, X.to(torch.bfloat16))
    with pytest.raises(TypeError):  # right shapes and dtypes, but host tensors
        g.project_similarity_static(Q, R, cn, X)
