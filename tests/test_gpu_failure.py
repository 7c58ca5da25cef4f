"""Failure detection on the GPU without a fault: the device's bounded waits.

Every pipeline wait in libee (mbarrier phases in the tensor-core kernels, the
cross-CTA arrival counter of the split-KV merge) gives up after a fixed number
of SM cycles, sets EE_DEVERR_TIMEOUT in the workspace's error word and lets
the kernel return.  ee_selftest_timeout makes both kinds of wait run out (an
mbarrier nothing arrives at, a counter nothing raises); this test checks how
each ended, that the host reads the status, and that the context and the
workspace stay usable for a normal call afterwards.
"""
import time

import pytest
import torch

import paper_2506_02780_gb300 as ee

pytestmark = pytest.mark.gpu


def test_bounded_waits_time_out_and_report():
    dev = torch.device("cuda:0")
    ws = ee.new_workspace(1, 4, 4, 0, device=dev)
    assert ee.ee_read_errors(ws) == 0
    out = torch.full((7,), -1, dtype=torch.int64, device=dev)
    t0 = time.perf_counter()
    ee.ee_selftest_timeout(ws, out)
    bits = ee.ee_read_errors(ws)       # synchronises
    wall = time.perf_counter() - t0
    limit, ok_a, cyc_a, ok_b, cyc_b, ok_c, cyc_c = out.cpu().tolist()
    assert bits == ee.DEVERR_TIMEOUT
    assert limit == 2_000_000_000
    # (a) the mbarrier wait gave up at its limit
    assert ok_a == 0 and limit < cyc_a < limit * 1.05
    # (b) the later waiter left through the abort flag raised by (a), about
    # half a limit into its own wait, well before its own limit
    assert ok_b == 0 and 0.3 * limit < cyc_b < 0.8 * limit
    # (c) the global counter wait gave up at its limit
    assert ok_c == 0 and limit < cyc_c < limit * 1.05
    # two limits of SM cycles at 1-2.07 GHz, plus launch and copy overhead
    assert 1.5 < wall < 10.0
    # the error word was cleared; after re-initialising the workspace the
    # context still runs work and a second run behaves the same
    assert ee.ee_read_errors(ws) == 0
    ee.ee_workspace_init(ws)
    assert torch.arange(8, device=dev).sum().item() == 28
    ee.ee_selftest_timeout(ws, out)
    assert ee.ee_read_errors(ws) == ee.DEVERR_TIMEOUT
    assert out[1].item() == 0 and out[5].item() == 0
