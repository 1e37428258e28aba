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


_LAUNCH_CHILD = r"""
import sys
sys.path.insert(0, {root!r})
import torch
from paper_2404_08573_gb300 import ff
from tests.gpu_common import pair_inputs
x2, l2 = pair_inputs(32, seed=5)
x, lab = torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda()
try:
    layer = ff.Layer(784, 128, prec="bf16")
    print("created")
except ff.FFError as e:
    print("create status", e.status)
    layer = ff.Layer(784, 128, prec="bf16")
try:
    layer.train_step(x, labels=lab, B=32)
    print("step ok")
except ff.FFError as e:
    print("step status", e.status)
loss = torch.zeros(1, device="cuda")
layer.train_step(x, labels=lab, B=32, loss=loss)   # later launches are made
torch.cuda.synchronize()
layer.check()
print("after", bool(torch.isfinite(loss).item()))
"""


@pytest.mark.parametrize("fail_at,expect", [(1, "create status 2"), (3, "step status 2"), (6, "step status 2")])
def test_injected_launch_failure_is_reported_and_recoverable(fail_at, expect):
    """FF_FAULT_LAUNCH_FAIL_AT=n: the n-th launch (1, 2: weight init; 3..7:
    overlay, forward, local gradient, weight gradient, Adam of the first step)
    is not made; the call that needed it returns FF_ERR_CUDA and later calls
    work."""
    torch_cuda()
    lib_ready()
    env = dict(os.environ, FF_FAULT_LAUNCH_FAIL_AT=str(fail_at))
    r = subprocess.run([sys.executable, "-c", _LAUNCH_CHILD.format(root=ROOT)], env=env, capture_output=True,
                       text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    assert expect in r.stdout and "after True" in r.stdout, r.stdout


def test_host_deadline_wait_on_a_net():
    """A net whose work waits behind a 0.5 s bounded device wait: a 20 ms
    host-side wait reports FF_ERR_TIMEOUT, a long one then completes."""
    torch = torch_cuda()
    ff = lib_ready()
    gate = ff.Layer(784, 64, prec="bf16", init_seed=1)
    layers = [ff.Layer(784, 128, prec="bf16", init_seed=2), ff.Layer(128, 64, prec="bf16", init_seed=3)]
    net = ff.Net(layers, max_B=32, depth=2)
    x2, l2 = pair_inputs(32, seed=6)
    s = torch.cuda.Stream()
    gate.selftest_wait(500000, stream=s)          # holds `s` for 0.5 s
    net.train_step(torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda(), B=32, stream=s)
    with pytest.raises(ff.FFError) as ei:
        net.wait(20)
    assert ei.value.status == 4                   # FF_ERR_TIMEOUT
    net.wait(20000)
    with pytest.raises(ff.FFError):
        gate.check()                              # the gate's own wait ran out, as intended
    for l in layers:
        l.check()
    assert all(l.get_state()["t"] == 1 for l in layers)
