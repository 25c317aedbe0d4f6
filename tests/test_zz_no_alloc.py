"""The allocation-free project + similarity entry point against the regular one.

gs_project_similarity_static serves callers that cannot allocate device memory
(graph captures that forbid it, plugins inside a fixed memory budget, hosts whose
allocator owns the device): its scratch is a fixed array inside the library.
This file is collected last so that, if it fails, a run stopping at the first
failure has already run every other test; it also passes when run alone.
"""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


def test_static_scratch_entry_matches_regular_entry(gs):
    # r = M = 512: 1025 floats of scratch per row, so 6000 rows take two chunks
    a = synth.attention(B=1, L=1)
    b = gs.build_basis(torch.from_numpy(a["C"]).cuda())
    Q, R, cn = b.Q.contiguous(), b.R.contiguous(), b.cnorm.contiguous()
    calls = [("cosine", 1.0, 7), ("raw", 0.5, 8)]
    for mode, scale, seed in calls:  # two calls in a row share the static scratch
        X, _ = synth.noisy_rows(a["C"], seed, 0, 6000, 1.0)
        Xd = torch.from_numpy(X).cuda()
        got = gs.project_similarity_static(Q, R, cn, Xd, mode=mode, scale=scale)
        ref = gs.project_similarity(b, Xd, mode=mode, scale=scale, path="simt")
        gs.stream_status()
        assert torch.equal(got["argmax"], ref["argmax"])
        xn = np.linalg.norm(X.astype(np.float64), axis=1)
        bound = 1e-4 * (abs(scale) if mode == "cosine" else abs(scale) * xn * np.sqrt(a["D"]))
        diff = (got["maxval"] - ref["maxval"]).abs().double().cpu().numpy()
        assert np.all(diff <= bound)


def test_static_scratch_entry_rejects_oversized_problems(gs):
    import ctypes
    lib = gs.load_library()
    st = lib.gs_project_similarity_static(None, 4096, 8, None, 4 << 20, None, None, 1, 8, 0, 1.0,
                                          None, None, None)
    assert st == gs.GS_ERR_SHAPE
    assert lib.gs_project_similarity_static(None, 0, 8, None, 4, None, None, 0, 8, 0, 1.0, None, None,
                                            None) == gs.GS_OK
    del ctypes
