"""Failure detection on the GPU without a fault: the kernels' bounded waits.

A self-check launch waits, with the library's own wait routines, on an
mbarrier that nothing arrives on and at a grid barrier that nothing
advances.  Each wait must give up after its limit, record WQ_ERR_TIMEOUT in
the device status and let the launch end; the context must stay usable (a
call after it still matches the oracle).
"""
import time

import numpy as np
import pytest
import torch

import oracle as orc
from paper_2606_04238_gb300 import synth
from tests.gpu_util import check_bf16, upload_packed

pytestmark = pytest.mark.gpu

WQ_ERR_TIMEOUT = -6


@pytest.fixture(scope="module")
def wq():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_04238_gb300 import wq as mod
    return mod


def test_bounded_waits_time_out_and_report(wq):
    assert wq.device_status() == 0
    t0 = time.time()
    wq.wait_check()
    torch.cuda.synchronize()
    elapsed = time.time() - t0
    assert wq.device_status() == WQ_ERR_TIMEOUT
    assert wq.device_status() == 0  # read and cleared
    assert 3.0 < elapsed < 30.0, f"two 2 s waits took {elapsed:.1f} s"
    # the context still works: a gate/up call against the oracle
    d, inter, group = 256, 256, 64
    w = (np.random.default_rng(1).standard_normal((inter, d)) * 0.02).astype(np.float32)
    q = orc.quantize(w, group, 2)[:3]
    g = upload_packed(*q, group, 2)
    x = synth.activations((1, d), 2)
    h = wq.gateup_w2_lora(x.cuda(), g, g, prenorm=True)
    torch.cuda.synchronize()
    assert wq.device_status() == 0
    ref, _ = orc.gateup(synth.bf16_bits(x), q, q, group, prenorm=True)
    check_bf16(h, ref, "gate/up after the timeouts")
