"""Failure detection on the GPU without a fault.

Every wait in the pipeline kernels (a TMA copy landing, a tensor-core commit, a
hand-off between warps) is bounded by the GPU's global timer; when one runs out the
kernel records AVTP_ERR_TIMEOUT in the workspace's status word and returns. This test
makes such a wait run out on purpose, on an mbarrier that nothing arrives on, with a
short limit, and checks that the host reads the status, that the wait lasted about
the limit, and that the context still runs the stage correctly afterwards.
"""
import time

import numpy as np
import pytest
import torch

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import DevWorkload, assert_scores_close, ensure_built

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    ensure_built()


def _timed_selftest(limit_ns, arrive, ws):
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    avtp.wait_selftest(limit_ns, arrive, ws)
    status = avtp.read_device_status(ws)  # synchronises
    return status, time.perf_counter() - t0


def test_a_wait_nothing_completes_reports_timeout_and_returns():
    ws = avtp.new_workspace(256)
    limit_ns = 20_000_000  # 20 ms
    status, secs = _timed_selftest(limit_ns, False, ws)
    assert status == avtp.ERR_TIMEOUT
    assert secs >= 0.9 * limit_ns * 1e-9  # the wait did run for its limit ...
    assert secs < 5.0  # ... and then gave up
    # the status word names the waiter that recorded first (0: one thread, 1: a warp)
    detail = int(ws[:16].view(torch.int32)[2].item())
    assert detail in (0, 1)


def test_a_wait_that_completes_reports_ok():
    ws = avtp.new_workspace(256)
    status, secs = _timed_selftest(1_000_000_000, True, ws)
    assert status == avtp.OK
    assert secs < 0.5  # nowhere near the one-second limit


def test_the_context_runs_the_stage_after_a_timeout():
    ws = avtp.new_workspace(256)
    status, _ = _timed_selftest(5_000_000, False, ws)
    assert status == avtp.ERR_TIMEOUT
    wl = synth.make_workload("tiny")
    dw = DevWorkload(wl)
    for criterion in ("hidden_variation", "text_attention"):
        scores, sums = avtp.score(dw.L, criterion, **dw.score_tensors(criterion))
        torch.cuda.synchronize()
        got = scores.cpu().numpy()
        if criterion == "hidden_variation":
            ref = O.score_hidden_variation(wl.layout, wl.h_cur, wl.h_prior)
        else:
            ref = O.score_text_attention(wl.layout, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)
        assert_scores_close(got, ref, wl.layout.visual_mask())
        assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


def test_selftest_arguments_are_checked_before_launch():
    ws = avtp.new_workspace(256)
    for bad in (0, 999, 10_000_000_001):
        with pytest.raises(avtp.AVTPError):
            avtp.wait_selftest(bad, False, ws)
