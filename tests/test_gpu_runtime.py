"""Runtime services around the step: checkpoint files (.npz) that resume
training bit for bit."""

import os

import numpy as np
import pytest

from .gpu_common import lib_ready, pair_inputs, torch_cuda

pytestmark = pytest.mark.gpu


def test_checkpoint_file_resumes_bitwise(tmp_path):
    torch = torch_cuda()
    ff = lib_ready()
    mk = lambda: [ff.Layer(784, 96, prec="bf16", init_seed=7), ff.Layer(96, 64, prec="bf16", init_seed=8)]
    a = mk()
    head_a = ff.Head(64, lr=1e-3)
    batches = [pair_inputs(64, seed=20 + t) for t in range(6)]
    net = ff.Net(a, max_B=64, depth=2)

    def steps(net, head, layers, ts):
        for t in ts:
            x2, l2 = batches[t]
            xg, lg = torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda()
            net.train_step(xg, lg, B=64)
            net.sync()
            head.train_step(layers, xg[:64], lg[:64])
        torch.cuda.synchronize()

    steps(net, head_a, a, range(3))
    path = os.path.join(tmp_path, "ckpt.npz")
    ff.save_checkpoint(path, a, [head_a])
    steps(net, head_a, a, range(3, 6))
    b = mk()
    head_b = ff.Head(64, lr=1e-3)
    ff.load_checkpoint(path, b, [head_b])
    assert [l.get_state()["t"] for l in b] == [3, 3] and head_b.get_state()["t"] == 3
    net_b = ff.Net(b, max_B=64, depth=2)
    steps(net_b, head_b, b, range(3, 6))
    for la, lb in zip(a, b):
        sa, sb = la.get_state(), lb.get_state()
        for k in ("W", "b", "mW", "vW", "mb", "vb"):
            assert np.array_equal(sa[k], sb[k]), k
    ha, hb = head_a.get_state(), head_b.get_state()
    for k in ("V", "c", "mV", "vV"):
        assert np.array_equal(ha[k], hb[k]), k
    with pytest.raises(ValueError):
        ff.load_checkpoint(path, [ff.Layer(784, 97, prec="bf16"), b[1]], [head_b])
