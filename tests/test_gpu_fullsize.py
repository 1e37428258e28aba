"""Parity at the benchmarked shapes of the 784-2000-2000-2000-2000 net.

* Goodness prediction (§3 "Prediction") and AdaptiveNEG negatives (§5) over
  1200 samples: more than one sample chunk (972 + a 228-sample tail in bf16,
  524 + 524 + 152 in fp32), so the chunked layer chain, its tail and the
  forward epilogue of layers 3 and 4 that adds the previous layer's goodness
  into each label's total are all compared with the oracle, element by
  element.  Layer 1's label columns carry ten times the He-uniform scale, as
  a trained net's do: with random weights the ten label totals of a sample
  sit within 1e-5 of each other on ~0.6 % of samples, where any rounding
  order decides the argmax.
* The train step at batch 1024 (2048 rows), four layers, several steps in a
  row: each step against the oracle's step started from the GPU's own
  pre-step state (so that rounding does not compound across steps).  At
  lr 0.03 the oracle's layer 1 goes dead after the first update (every ReLU
  off: its goodness is 0, its loss softplus(2) + softplus(-2)); the GPU must
  follow it there.  At lr 0.001 every layer stays alive.
"""

import numpy as np
import pytest

from oracle import ff_oracle as fo
from paper_2404_08573_gb300 import synth
from tests.gpu_common import assert_close, lib_ready, oracle_state, rel_norm, torch_cuda

pytestmark = pytest.mark.gpu

DIMS = (784, 2000, 2000, 2000, 2000)


@pytest.fixture(scope="module")
def env():
    torch = torch_cuda()
    ff = lib_ready()
    return torch, ff


def _net(ff, prec):
    layers, states = [], []
    for i in range(len(DIMS) - 1):
        rng = np.random.default_rng(60 + i)
        W = synth.he_uniform(60 + i, DIMS[i + 1], DIMS[i])
        if i == 0:
            W[:, :10] *= 10.0
        b = (rng.standard_normal(DIMS[i + 1]) * 0.02).astype(np.float32)
        l = ff.Layer(DIMS[i], DIMS[i + 1], prec=prec)
        l.set_state(W=W, b=b)
        layers.append(l)
        states.append(fo.LayerState(W, b))
    return layers, states


def _check_labels(p, rp, rG, rel_tie):
    agree = np.mean(p == rp)
    assert agree >= 0.995, agree
    for i in np.nonzero(p != rp)[0]:   # disagreements only at near ties
        gap = abs(rG[i, p[i]] - rG[i, rp[i]])
        assert gap <= rel_tie * abs(rG[i, rp[i]]), (i, gap)


@pytest.mark.parametrize("prec", ["bf16", "fp32"])
def test_predict_784_2000x4_over_several_chunks(env, prec):
    torch, ff = env
    layers, states = _net(ff, prec)
    n = 1200
    x = synth.mnist_like(n, seed=61)
    G = torch.empty(n, 10, device="cuda")
    pred, _ = ff.predict(layers, torch.from_numpy(x).cuda(), goodness=G)
    torch.cuda.synchronize()
    layers[0].check()
    emul = prec == "bf16"
    rp, rG = fo.predict(states, x, emulate_bf16=emul)
    Gg = G.cpu().numpy()
    assert_close(Gg, rG, 1e-4 if not emul else 2e-3, 1e-6, "predict goodness")
    _check_labels(pred.cpu().numpy(), rp, rG, 1e-4 if not emul else 1e-2)
    if emul:
        _, plain_G = fo.predict(states, x)
        assert_close(Gg, plain_G, 2e-2, 1e-4, "predict goodness vs fp64")


def test_adaptive_negatives_784_2000x4_over_several_chunks(env):
    torch, ff = env
    layers, states = _net(ff, "bf16")
    n = 1200
    x = synth.mnist_like(n, seed=62)
    y = synth.labels(n, seed=62)
    G = torch.empty(n, 10, device="cuda")
    neg, _ = ff.adaptive_negatives(layers, torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda(), goodness=G)
    torch.cuda.synchronize()
    layers[0].check()
    rn, rG = fo.adaptive_negatives(states, x, y, emulate_bf16=True)
    assert_close(G.cpu().numpy(), rG, 2e-3, 1e-6, "AdaptiveNEG goodness")
    got = neg.cpu().numpy()
    assert np.all(got != y), "a negative label equals the true label"
    _check_labels(got, rn, rG, 1e-2)


@pytest.mark.parametrize("lr,steps", [(0.03, 3), (0.001, 4)])
def test_train_784_2000x4_batch1024_trace(env, lr, steps):
    torch, ff = env
    B, theta = 1024, 2.0
    L = len(DIMS) - 1
    layers = [ff.Layer(DIMS[k], DIMS[k + 1], prec="bf16", theta=theta, lr=lr, init_seed=1000 + k, max_rows=2 * B)
              for k in range(L)]
    hs = [layers[k].new_activation(2 * B) for k in range(L)]
    ss = [torch.empty(2 * B, device="cuda") for _ in range(L)]
    hp = fo.AdamHyper(lr=lr)
    for step in range(steps):
        x = synth.mnist_like(B, seed=0, start_row=step * B)
        y = synth.labels(B, seed=0, start=step * B)
        x2, l2 = synth.pair_batch(x, y, synth.negative_labels(y, seed=0, start=step * B))
        pre = [l.get_state() for l in layers]
        gs = [torch.empty(2 * B, device="cuda") for _ in range(L)]
        loss = torch.zeros(L, device="cuda")
        xg, lg = torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda()
        for k, layer in enumerate(layers):
            layer.train_step(xg if k == 0 else hs[k - 1], labels=lg if k == 0 else None,
                             row_scale=None if k == 0 else ss[k - 1], B=B, h_out=hs[k], next_scale=ss[k],
                             goodness=gs[k], loss=loss[k:k + 1])
        torch.cuda.synchronize()
        for l in layers:
            l.check()
        x_in = fo.overlay_label(x2, l2)
        for k, layer in enumerate(layers):
            st = oracle_state(pre[k])
            out = fo.layer_train_step(st, x_in, B, theta, hp, emulate_bf16=True)
            what = f"lr {lr} step {step} layer {k + 1}"
            lg_ = loss[k].item()
            assert abs(lg_ - out["loss"]) <= 1e-3 * out["loss"], (what, lg_, out["loss"])
            assert_close(gs[k].cpu().numpy(), out["g"], 1e-3, 1e-5, what + " goodness")
            act_gpu = layer.stats()[2]
            act_ref = float(np.mean(out["H"] > 0))
            assert abs(act_gpu - act_ref) <= 1e-3, (what, act_gpu, act_ref)
            post = layer.get_state()
            assert rel_norm(post["W"], st.W) <= 1e-2, (what, rel_norm(post["W"], st.W))
            if lr == 0.03 and step >= 1 and k == 0:
                # the method's own collapse at this learning rate, on both sides
                assert act_ref == 0.0 and act_gpu == 0.0, (what, act_gpu, act_ref)
                assert abs(out["loss"] - (fo.softplus(theta) + fo.softplus(-theta))) < 1e-12
            if lr == 0.001:
                assert act_gpu > 0.1, (what, act_gpu)
            x_in = out["H"]
