"""Failure detection without a GPU fault: a bounded device wait that is made
to run out (nothing ever arrives on its barrier) and host-side allocation
failures injected through FF_FAULT_ALLOC_FAIL_AT."""

import os
import subprocess
import sys

import numpy as np
import pytest

from tests.gpu_common import lib_ready, pair_inputs, torch_cuda

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bounded_wait_times_out_and_the_context_stays_usable():
    torch = torch_cuda()
    ff = lib_ready()
    layer = ff.Layer(784, 256, prec="bf16", init_seed=4)
    layer.selftest_wait(2000)   # 2 ms; the barrier never completes
    with pytest.raises(ff.FFError) as ei:
        layer.check()
    assert ei.value.status == 4  # FF_ERR_TIMEOUT
    layer.check()                # latched error cleared
    x2, l2 = pair_inputs(32, seed=5)
    loss = torch.empty(1, device="cuda")
    layer.train_step(torch.from_numpy(x2).cuda(), labels=torch.from_numpy(l2).cuda(), B=32, loss=loss)
    torch.cuda.synchronize()
    layer.check()
    assert np.isfinite(loss.item())


_CHILD = r"""
import sys
sys.path.insert(0, {root!r})
import torch
from paper_2404_08573_gb300 import ff
try:
    ff.Layer(784, 128, prec="bf16")
    print("created")
except ff.FFError as e:
    print("status", e.status)
layer = ff.Layer(784, 128, prec="bf16")   # later allocations succeed
print("second ok")
"""


@pytest.mark.parametrize("fail_at", [1, 2, 4])
def test_injected_allocation_failure_is_reported_and_recoverable(fail_at):
    torch_cuda()
    lib_ready()
    env = dict(os.environ, FF_FAULT_ALLOC_FAIL_AT=str(fail_at))
    r = subprocess.run([sys.executable, "-c", _CHILD.format(root=ROOT)], env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert "status 3" in r.stdout and "second ok" in r.stdout, r.stdout
