"""Failure detection on a GPU, without a fault: a bounded wait that runs out.

Every kernel waits on its mbarriers with a wait that gives up after a fixed
number of SM cycles (about 1 s) and sets TGVKV_STATUS_TIMEOUT in the caller's
workspace instead of hanging.  tgvkv_check_wait_timeout makes that wait on a
barrier nothing arrives at; the host must read the timeout bit, and the context
must stay usable for the next eviction.
"""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2606_03075_gb300 import synth

import _parity as P

pytestmark = pytest.mark.gpu

STATUS_TIMEOUT = 0x20


@pytest.fixture(scope="module")
def api():
    assert torch.cuda.is_available(), "the GPU tests need a CUDA device"
    from paper_2606_03075_gb300 import build
    build.build()
    from paper_2606_03075_gb300 import api as _api
    return _api


def test_bounded_wait_runs_out_and_reports_timeout(api):
    wl = synth.WORKLOADS["tiny"]
    desc = api.desc_for_workload(wl)
    ws = api.new_workspace(desc)
    t0 = time.time()
    api.tgvkv_check_wait_timeout(ws)
    bits = api.tgvkv_status(ws)            # synchronises, reads and clears
    elapsed = time.time() - t0
    assert bits == STATUS_TIMEOUT
    assert elapsed < 10.0
    assert api.tgvkv_status(ws) == 0       # cleared
    # the context is intact: an eviction on the same device matches the oracle
    inp = synth.generate(wl, seed=0)
    g = P.run_evict(api, wl, inp, 0.25)
    assert g["status"] == 0
    ref = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"], inp["w"],
                       0.25, wl.H_kv)
    P.assert_close(g["scores"], ref["scores"], "scores after the timeout")
    assert np.array_equal(g["budgets"], np.asarray(ref["budgets"]))
