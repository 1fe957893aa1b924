"""A wait in the tensor-core kernels that can never complete is reported, not hung on: the
self-test kernel's wait gives up after its bounded time, the error word says so, and the
device keeps working. Nothing faults (no trap, no bad address)."""
import pytest
import torch

from gpu_helpers import gpu_step, host_inputs, to_dev
from paper_2604_11947_gb300 import resbm, synth

pytestmark = pytest.mark.gpu


def test_stuck_wait_is_reported_and_the_context_survives():
    assert resbm.resbm_device_error(clear=True) == 0
    resbm.resbm_selftest_wait_timeout()
    torch.cuda.synchronize()
    assert resbm.resbm_device_error(clear=True) == 1   # the timeout bit
    assert resbm.resbm_device_error() == 0            # cleared
    # the context is intact: a boundary step still runs and reports no timeout
    cfg = synth.BoundaryConfig("after_timeout", T=256, d=256, r=16, m=16)
    dev = {k: to_dev(v, cfg) for k, v in host_inputs(cfg).items()}
    out = gpu_step(cfg, dev)
    assert torch.isfinite(out["Y"].float()).all()
    assert resbm.resbm_device_error() == 0
