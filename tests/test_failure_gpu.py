"""Device-side failure detection, made to happen without a GPU fault.

Every wait of the tensor-core kernels on a pipeline mbarrier is bounded.  The
self-test entry point enqueues one block whose wait, through that same bounded
wait, is on a barrier that nothing ever completes.  The wait must give up, the
error must reach the host as GS_ERR_TIMEOUT through gs_stream_status, and the
CUDA context must stay usable: a normal tensor-core call right after it returns
correct results and a clean status.
"""
import time

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_context_survives(gs):
    t0 = time.perf_counter()
    gs.selftest_wait_timeout()
    with pytest.raises(gs.GramSpaceError) as e:
        gs.stream_status()
    waited = time.perf_counter() - t0
    assert e.value.status == gs.GS_ERR_TIMEOUT
    assert 1.5 < waited < 30.0  # the limit is 2 s of device time
    gs.stream_status()          # the error word was read and cleared
    # the context still runs the tensor-core path correctly
    w = synth.large(rows=(0, 4096))
    b = gs.build_basis(torch.from_numpy(w["C"]).cuda())
    out = gs.project_similarity(b, torch.from_numpy(w["X"]).cuda(), path="tensor")
    gs.stream_status()
    assert np.array_equal(out["argmax"].cpu().numpy(), w["labels"])
