"""The checked build (libff_checked.so, -DFF_DEVICE_CHECKS): every TMA
coordinate the kernels issue is checked on the device (alignment, sign), in
place of the sanitizers this pool does not run.  A mixed workload with ragged
shapes must latch no check and give bit for bit the results of the normal
build."""

import os
import subprocess
import sys

import pytest

from .gpu_common import lib_ready, torch_cuda

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_CHILD = r"""
import hashlib, sys
sys.path.insert(0, {root!r})
import numpy as np, torch
from paper_2404_08573_gb300 import ff, synth
from tests.gpu_common import pair_inputs
h = hashlib.sha1()
def take(t):
    h.update(t.detach().float().cpu().numpy().tobytes())
# a ragged forward
l0 = ff.Layer(2003, 777, prec="bf16", init_seed=1)
x = l0.new_activation(130, 2003)
x[:, :2003] = torch.from_numpy(np.maximum(synth.mnist_like(130, seed=2, features=2003), 0)).to(x.dtype)
out = l0.new_activation(130)
l0.forward(x, h_out=out)
take(out)
# a net on streams, three steps
layers = [ff.Layer(784, 256, prec="bf16", init_seed=3), ff.Layer(256, 136, prec="bf16", init_seed=4)]
net = ff.Net(layers, max_B=100, depth=2)
for t in range(3):
    x2, l2 = pair_inputs(100, seed=10 + t)
    net.train_step(torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda(), B=100)
net.sync()
torch.cuda.synchronize()
for l in layers:
    h.update(l.get_state()["W"].tobytes())
# predict, softmax head, Performance-Optimized step, chapter schedule
xs = torch.from_numpy(synth.mnist_like(300, seed=20)).cuda()
ys = torch.from_numpy(synth.labels(300, seed=21)).cuda()
G = torch.empty(300, 10, device="cuda")
pred, _ = ff.predict(layers, xs, goodness=G)
take(G)
head = ff.Head(136, lr=1e-3, max_rows=512)
head.train_step(layers, xs, ys)
take(head.predict(layers, xs)[0])
blk = ff.Head(256, lr=1e-3)
ff.po_train_step_raw(layers[0], blk, xs, ys)
torch.cuda.synchronize()
h.update(layers[0].get_state()["W"].tobytes())
x2, l2 = pair_inputs(64, seed=30)
pff = ff.Pff(layers, 64, 32, 1, 2)
pff.run(torch.from_numpy(x2).cuda(), torch.from_numpy(np.stack([l2, l2])).cuda(), 0, 2)
torch.cuda.synchronize()
for l in layers:
    h.update(l.get_state()["W"].tobytes())
# the local gradient in the forward epilogue (cluster exchange, dZ' store), ragged
lf = [ff.Layer(784, 264, prec="bf16", init_seed=40), ff.Layer(264, 136, prec="bf16", init_seed=41)]
for l in lf:
    l.set_fused_local_grad(True)
hf, sf = lf[0].new_activation(200), torch.empty(200, device="cuda")
x2, l2 = pair_inputs(100, seed=42)
lf[0].train_step(torch.from_numpy(x2).cuda(), labels=torch.from_numpy(l2).cuda(), B=100, h_out=hf, next_scale=sf)
lf[1].train_step(hf, row_scale=sf, B=100)
torch.cuda.synchronize()
for l in lf:
    h.update(l.get_state()["W"].tobytes())
# fp32 predict on the tensor cores (three TF32 products)
l32 = [ff.Layer(784, 200, prec="fp32", init_seed=50), ff.Layer(200, 136, prec="fp32", init_seed=51)]
G32 = torch.empty(300, 10, device="cuda")
ff.predict(l32, xs, goodness=G32)
take(G32)
# the softmax head's epoch call, and the persistent epoch kernel
head.train_epoch(layers, xs, ys, 128)
take(head.predict(layers, xs)[0])
le = [ff.Layer(784, 256, prec="bf16", init_seed=60), ff.Layer(256, 264, prec="bf16", init_seed=61)]
ne = ff.Net(le, max_B=128, depth=2)
parts = [pair_inputs(min(128, 296 - s0), seed=62 + s0) for s0 in range(0, 296, 128)]  # batches of 128, 128, 40 pairs
xe, le2 = np.concatenate([p[0] for p in parts]), np.concatenate([p[1] for p in parts])
ne.train_epoch(torch.from_numpy(xe).cuda(), torch.from_numpy(le2).cuda(), 296, 128)
torch.cuda.synchronize()
for l in le:
    h.update(l.get_state()["W"].tobytes())
for obj in [l0] + layers + lf + l32 + le + [head, blk]:
    obj.check()
print("digest", h.hexdigest())
"""


def test_checked_build_latches_nothing_and_matches():
    torch_cuda()
    lib_ready()
    from paper_2404_08573_gb300 import build
    build.build(checked=True)
    digests = []
    for variant in ("normal", "checked"):
        env = dict(os.environ, FF_LIB_VARIANT=variant)
        r = subprocess.run([sys.executable, "-c", _CHILD.format(root=ROOT)], env=env, capture_output=True, text=True,
                           timeout=600, cwd=ROOT)
        assert r.returncode == 0, (variant, r.stderr[-3000:])
        digests.append([l for l in r.stdout.splitlines() if l.startswith("digest")][0])
    assert digests[0] == digests[1], digests
