"""The bf16 train step's forward GEMM with the local step of §3 (Eq. 1) in
its epilogue (goodness over all column tiles through a thread-block cluster,
loss, dL/dg, next-layer scale, dZ', bias-gradient partials) against the same
step with that part in the separate local-gradient kernel: every output and
every piece of state must be bitwise equal, on a labelled first layer and on
a hidden layer fed by it, over several steps.  The separate kernel is the
one the oracle parity tests pinned first; the persistent epoch kernel
follows the same reduction orders (tests/test_gpu_epoch.py)."""

import numpy as np
import pytest

from paper_2404_08573_gb300 import synth
from tests.gpu_common import lib_ready, torch_cuda

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    torch = torch_cuda()
    ff = lib_ready()
    return torch, ff


def _pair(B, K, step, seed):
    x = synth.mnist_like(B, seed=seed, features=K, start_row=step * B)
    y = synth.labels(B, seed=seed, start=step * B)
    return synth.pair_batch(x, y, synth.negative_labels(y, seed=seed, start=step * B))


def _host(a):
    if hasattr(a, "cpu"):
        if str(a.dtype) == "torch.bfloat16":
            a = a.view(dtype=__import__("torch").int16)  # compare bf16 values bit for bit
        return a.cpu().numpy()
    return np.asarray(a)


def _same(a, b, what):
    a, b = _host(a), _host(b)
    if a.dtype != b.dtype or a.shape != b.shape:
        raise AssertionError(f"{what}: {a.dtype}{a.shape} vs {b.dtype}{b.shape}")
    eq = (a == b) | (np.isnan(a.astype(np.float64)) & np.isnan(b.astype(np.float64)))
    assert eq.all(), f"{what}: {int((~eq).sum())} of {eq.size} differ"


@pytest.mark.parametrize("K,N1,N2,B,steps", [
    (784, 256, 256, 64, 3),       # one column tile, padding rows in the last pair tile
    (784, 2000, 2000, 1024, 2),   # the benchmarked shape: four column tiles, a cluster of 8
    (784, 2000, 2000, 608, 2),    # the epoch's last, ragged batch (1216 rows)
    (300, 264, 136, 150, 3),      # partial column tiles, rows not a multiple of 32
    (136, 1536, 520, 200, 2),     # three column tiles, then two
    (40, 8, 24, 5, 2),            # a single, mostly empty tile
    (64, 2100, 64, 96, 2),        # wider than a cluster holds: the separate kernel on both sides
])
def test_fused_local_gradient_is_bitwise_the_separate_kernel(env, K, N1, N2, B, steps):
    torch, ff = env
    M = 2 * B

    def make():
        l1 = ff.Layer(K, N1, prec="bf16", theta=2.0, lr=3e-3, init_seed=50, max_rows=M, keep_grad=True)
        l2 = ff.Layer(N1, N2, prec="bf16", theta=2.0, lr=3e-3, init_seed=51, max_rows=M, keep_grad=True)
        return l1, l2

    fused, sep = make(), make()
    for l in fused:
        l.set_fused_local_grad(True)
    for l in sep:
        l.set_fused_local_grad(False)

    def outs(layers):
        l1, l2 = layers
        return dict(h1=l1.new_activation(M), s1=torch.empty(M, device="cuda"), g1=torch.empty(M, device="cuda"),
                    h2=l2.new_activation(M), s2=torch.empty(M, device="cuda"), g2=torch.empty(M, device="cuda"),
                    loss=torch.zeros(2, device="cuda"))

    # the fused form runs one kernel fewer per layer step (no separate local-
    # gradient launch) on every layer no wider than a cluster holds
    n_fusable = sum(1 for n in (N1, N2) if n <= 2048)
    for step in range(steps):
        x2, l2lab = _pair(B, K, step, seed=7)
        xg, lg = torch.from_numpy(x2).cuda(), torch.from_numpy(l2lab).cuda()
        res, launches = [], []
        for layers in (fused, sep):
            l1, l2 = layers
            o = outs(layers)
            k0 = ff.kernel_launches()
            l1.train_step(xg, labels=lg, B=B, h_out=o["h1"], next_scale=o["s1"], goodness=o["g1"],
                          loss=o["loss"][0:1])
            l2.train_step(o["h1"], row_scale=o["s1"], B=B, h_out=o["h2"], next_scale=o["s2"], goodness=o["g2"],
                          loss=o["loss"][1:2])
            launches.append(ff.kernel_launches() - k0)
            torch.cuda.synchronize()
            for l in layers:
                l.check()
            res.append(o)
        what = f"K{K} N{N1},{N2} B{B} step {step}"
        assert launches[0] == launches[1] - n_fusable, (what, launches)
        for key in ("h1", "s1", "g1", "h2", "s2", "g2", "loss"):
            _same(res[0][key], res[1][key], f"{what} {key}")
        for k, (a, b) in enumerate(zip(fused, sep)):
            sa, sb = a.get_state(), b.get_state()
            for key in ("W", "b", "mW", "vW", "mb", "vb"):
                _same(sa[key], sb[key], f"{what} layer {k + 1} {key}")
            assert sa["t"] == sb["t"] == step + 1
            assert a.stats() == b.stats(), (what, k, a.stats(), b.stats())
            for name, ga, gb in zip(("dW", "db"), a.get_grad(), b.get_grad()):
                _same(ga, gb, f"{what} layer {k + 1} {name}")
            _same(a.get_grad_operand(M), b.get_grad_operand(M), f"{what} layer {k + 1} dZ'")
    for l in fused + sep:
        l.close()
