"""The persistent train-epoch kernel (ff_net_train_epoch) against the same
batches through ff_net_train_step, one call per batch (which the parity tests
hold to the oracle): parameters, Adam moments, step counters, per-batch
losses and step statistics must be bitwise equal.  The first batch is also
checked against the oracle directly."""

import numpy as np
import pytest

from oracle import ff_oracle as fo
from paper_2404_08573_gb300 import synth
from tests.gpu_common import lib_ready, torch_cuda

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    torch = torch_cuda()
    ff = lib_ready()
    return torch, ff


def _pairs(n_pairs, B, K, seed):
    """Stacked pair batches (x2) and one image per pair (x1), with labels laid
    out per batch (true labels, then wrong labels)."""
    xs2, xs1, ls = [], [], []
    for start in range(0, n_pairs, B):
        b = min(B, n_pairs - start)
        x = synth.mnist_like(b, seed=seed, features=K, start_row=start)
        y = synth.labels(b, seed=seed, start=start)
        yn = synth.negative_labels(y, seed=seed, start=start)
        x2, l2 = synth.pair_batch(x, y, yn)
        xs2.append(x2)
        xs1.append(x)
        ls.append(l2)
    return np.concatenate(xs2), np.concatenate(xs1), np.concatenate(ls)


def _nets(ff, dims, B, lr, seed0):
    mk = lambda: [ff.Layer(dims[k], dims[k + 1], prec="bf16", theta=2.0, lr=lr, init_seed=seed0 + k,
                           max_rows=2 * B) for k in range(len(dims) - 1)]
    la, lb = mk(), mk()
    return la, ff.Net(la, max_B=B, depth=2), lb, ff.Net(lb, max_B=B, depth=2)


def _assert_same_state(la, lb, what):
    for k, (a, b) in enumerate(zip(la, lb)):
        sa, sb = a.get_state(), b.get_state()
        for key in ("W", "b", "mW", "vW", "mb", "vb"):
            assert np.array_equal(sa[key], sb[key]), f"{what}: layer {k + 1} {key} differs " \
                f"(max |diff| {np.max(np.abs(sa[key] - sb[key]))})"
        assert sa["t"] == sb["t"], (what, k, sa["t"], sb["t"])
        assert a.stats() == b.stats(), (what, k, a.stats(), b.stats())
        a.check()
        b.check()


@pytest.mark.parametrize("dims,B,n_pairs,images", [
    ((784, 256, 256), 128, 5 * 128 + 40, 2),        # several batches and a ragged tail
    ((784, 256, 256), 128, 5 * 128 + 40, 1),        # one image per pair
    ((784, 512, 264, 136), 256, 3 * 256, 2),        # partial column tiles, three layers, no tail
])
def test_epoch_kernel_is_bitwise_the_per_step_path(env, dims, B, n_pairs, images):
    torch, ff = env
    la, na, lb, nb_ = _nets(ff, dims, B, 0.003, 70)
    x2, x1, lab = _pairs(n_pairs, B, dims[0], seed=71)
    xg = torch.from_numpy(x2 if images == 2 else x1).cuda()
    lg = torch.from_numpy(lab).cuda()
    nbat = -(-n_pairs // B)
    L = len(dims) - 1
    loss_a = torch.zeros(nbat, L, device="cuda")
    loss_b = torch.zeros(nbat, L, device="cuda")
    na.train_epoch(xg, lg, n_pairs, B, images_per_pair_row=images, loss=loss_a)
    torch.cuda.synchronize()
    for t, start in enumerate(range(0, n_pairs, B)):
        b = min(B, n_pairs - start)
        if images == 2:
            nb_.train_step(xg[2 * start:2 * start + 2 * b], lg[2 * start:2 * start + 2 * b], B=b, loss=loss_b[t])
        else:
            nb_.train_step_images(xg[start:start + b], lg[2 * start:2 * start + 2 * b], loss=loss_b[t])
    nb_.sync()
    torch.cuda.synchronize()
    assert torch.equal(loss_a, loss_b), ("per-batch loss differences", (loss_a - loss_b).abs().cpu().numpy())
    _assert_same_state(la, lb, f"{dims} B={B}")
    # a second epoch reuses the plan and continues the same run
    na.train_epoch(xg, lg, n_pairs, B, images_per_pair_row=images, loss=loss_a)
    for t, start in enumerate(range(0, n_pairs, B)):
        b = min(B, n_pairs - start)
        if images == 2:
            nb_.train_step(xg[2 * start:2 * start + 2 * b], lg[2 * start:2 * start + 2 * b], B=b, loss=loss_b[t])
        else:
            nb_.train_step_images(xg[start:start + b], lg[2 * start:2 * start + 2 * b], loss=loss_b[t])
    nb_.sync()
    torch.cuda.synchronize()
    assert torch.equal(loss_a, loss_b)
    _assert_same_state(la, lb, f"{dims} B={B}, second epoch")
    na.close()
    nb_.close()


def test_epoch_kernel_784_2000x4_batch1024(env):
    """The benchmarked shape: four batches of 1024 pairs (the last 608) at
    lr 1e-3, bitwise against the per-step path, and the first batch's losses
    against the oracle (emulating the bf16 operands)."""
    torch, ff = env
    dims, B = (784, 2000, 2000, 2000, 2000), 1024
    n_pairs = 3 * B + 608
    la, na, lb, nb_ = _nets(ff, dims, B, 1e-3, 1000)
    init = [l.get_state() for l in la]
    x2, _, lab = _pairs(n_pairs, B, 784, seed=0)
    xg, lg = torch.from_numpy(x2).cuda(), torch.from_numpy(lab).cuda()
    loss_a = torch.zeros(4, 4, device="cuda")
    loss_b = torch.zeros(4, 4, device="cuda")
    na.train_epoch(xg, lg, n_pairs, B, loss=loss_a)
    for t, start in enumerate(range(0, n_pairs, B)):
        b = min(B, n_pairs - start)
        nb_.train_step(xg[2 * start:2 * start + 2 * b], lg[2 * start:2 * start + 2 * b], B=b, loss=loss_b[t])
    nb_.sync()
    torch.cuda.synchronize()
    assert torch.equal(loss_a, loss_b), ("per-batch loss differences", (loss_a - loss_b).abs().cpu().numpy())
    _assert_same_state(la, lb, "784-2000x4")
    states = [fo.LayerState(s["W"], s["b"]) for s in init]
    outs = fo.net_train_step(states, x2[:2 * B], lab[:2 * B], B, 2.0, fo.AdamHyper(lr=1e-3), emulate_bf16=True)
    got = loss_a[0].cpu().numpy()
    for k, o in enumerate(outs):
        assert abs(got[k] - o["loss"]) <= 1e-3 * o["loss"], (k, got[k], o["loss"])
    na.close()
    nb_.close()


def test_epoch_kernel_with_split_roles_is_bitwise_the_per_step_path(env, monkeypatch):
    """Roles split by cluster (FF_EPOCH_GEMM_CLUSTERS: that many clusters run
    only GEMM tiles, the others only the streamed tasks): the same bits."""
    torch, ff = env
    monkeypatch.setenv("FF_EPOCH_GEMM_CLUSTERS", "8")
    dims, B, n_pairs = (784, 512, 264), 256, 4 * 256 + 72
    la, na, lb, nb_ = _nets(ff, dims, B, 0.003, 90)
    x2, _, lab = _pairs(n_pairs, B, dims[0], seed=91)
    xg, lg = torch.from_numpy(x2).cuda(), torch.from_numpy(lab).cuda()
    nbat = -(-n_pairs // B)
    loss_a = torch.zeros(nbat, 2, device="cuda")
    loss_b = torch.zeros(nbat, 2, device="cuda")
    na.train_epoch(xg, lg, n_pairs, B, loss=loss_a)
    for t, start in enumerate(range(0, n_pairs, B)):
        b = min(B, n_pairs - start)
        nb_.train_step(xg[2 * start:2 * start + 2 * b], lg[2 * start:2 * start + 2 * b], B=b, loss=loss_b[t])
    nb_.sync()
    torch.cuda.synchronize()
    assert torch.equal(loss_a, loss_b), ("per-batch loss differences", (loss_a - loss_b).abs().cpu().numpy())
    _assert_same_state(la, lb, "split roles")
    na.close()
    nb_.close()
