"""GPU parity: the CUDA path through the C ABI against the CPU oracle on the
same seeded inputs.

Tolerances.  fp32 mode: 1e-4 relative on goodness, loss and weights after
each step.  bf16-operand mode: 2e-2 relative per step; the oracle is run with
the bf16 rounding of the stored operands emulated, which lets most checks use
tighter bounds (they are stated per assertion).  Adam's first steps move a
weight by about lr*sign(g): where a gradient element is within its own
rounding bound of zero or of eps, the update is steep in g, so weights are
held to 1e-4 plus the spread of the oracle's Adam over that bound (derived in
tests/gpu_common.py), and the Adam kernel itself is checked tightly against
the GPU's own gradient.
"""

import numpy as np
import pytest

from oracle import ff_oracle as fo
from paper_2404_08573_gb300 import synth
from tests.gpu_common import (assert_adam_state, assert_close, grad_uncertainty, lib_ready, oracle_state, pair_inputs,
                              rel_norm, torch_cuda)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    torch = torch_cuda()
    ff = lib_ready()
    return torch, ff


def _rand_layer_state(N, K, seed, bias_scale=0.05):
    rng = np.random.default_rng(seed)
    W = synth.he_uniform(seed, N, K)
    b = (rng.standard_normal(N) * bias_scale).astype(np.float32)
    return W, b


# ------------------------------------------------------------------ init
@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_created_weights_equal_the_generator(env, prec):
    torch, ff = env
    layer = ff.Layer(784, 500, prec=prec, init_seed=5)
    st = layer.get_state()
    assert np.array_equal(st["W"], synth.he_uniform(5, 500, 784))
    for k in ("b", "mW", "vW", "mb", "vb"):
        assert not st[k].any()
    assert st["t"] == 0


# --------------------------------------------------------------- overlay
@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_overlay_kernel(env, prec):
    torch, ff = env
    rows, F = 37, 794
    x = synth.mnist_like(rows, seed=3, features=F)
    x[:, :10] = 0.5
    lab = synth.labels(rows, seed=3)
    lab[0], lab[1] = 0, 9
    xg = torch.from_numpy(x).cuda()
    s = torch.empty(rows, device="cuda")
    out = ff.overlay_label(xg, torch.from_numpy(lab).cuda(), prec=prec, row_scale=s)
    torch.cuda.synchronize()
    ref = fo.overlay_label(x, lab)
    got = out.float().cpu().numpy()
    assert got.shape == (rows, ff.row_stride(F))
    exp = ref if prec == "fp32" else fo.bf16_round(ref)
    assert np.array_equal(got[:, :F], exp.astype(np.float32))
    assert not got[:, F:].any()
    assert_close(s.cpu().numpy(), 1.0 / fo.row_norm(ref), 1e-6, 0, "row scale")


# --------------------------------------------------------------- forward
FWD_CASES = [
    ("fp32", 300, 784, 600), ("bf16", 300, 784, 600), ("bf16", 1, 11, 5), ("fp32", 1, 11, 5),
    ("bf16", 130, 2003, 777), ("fp32", 130, 2003, 777), ("bf16", 257, 64, 256), ("bf16", 2048, 2000, 2000),
    # the bf16 GEMM's three tile shapes: 128-column tiles (at most 76 CTAs of
    # one 128-row subtile each), 256-column tiles of one subtile, of two
    ("bf16", 1024, 300, 2000), ("bf16", 1216, 300, 2000),
]


@pytest.mark.parametrize("prec,M,K,N", FWD_CASES)
def test_forward_hidden_layer(env, prec, M, K, N):
    torch, ff = env
    rng = np.random.default_rng(M + K + N)
    xin = np.maximum(rng.standard_normal((M, K)), 0.0).astype(np.float32)
    xin[M // 2] = 0.0                                   # a dead row: s = 1/1e-12 path, g = ReLU(b)^2
    if prec == "bf16":
        xin = fo.bf16_round(xin).astype(np.float32)     # the stored activity is bf16
    W, b = _rand_layer_state(N, K, seed=K)
    layer = ff.Layer(K, N, prec=prec, init_seed=1)
    layer.set_state(W=W, b=b)
    xa = layer.new_activation(M, K)
    xa[:, :K] = torch.from_numpy(xin).to(xa.dtype)
    h = layer.new_activation(M)
    g = torch.empty(M, device="cuda")
    sn = torch.empty(M, device="cuda")
    layer.forward(xa, h_out=h, goodness=g, next_scale=sn)
    torch.cuda.synchronize()
    layer.check()
    ref = fo.layer_forward_full(fo.LayerState(W, b), xin, emulate_bf16=(prec == "bf16"))
    tol = 1e-5 if prec == "fp32" else 1e-3
    assert_close(g.cpu().numpy(), ref["g"], tol, 1e-6, "goodness")
    hg = h.float().cpu().numpy()
    assert not hg[:, N:].any()
    hrt = 1e-5 if prec == "fp32" else 2.0 ** -8 + 1e-3
    assert_close(hg[:, :N], ref["H"], hrt, 1e-5, "activity")
    assert_close(sn.cpu().numpy(), 1.0 / np.maximum(np.sqrt(ref["g"]), 1e-12), tol, 0, "next scale")


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_forward_first_layer_with_labels(env, prec):
    torch, ff = env
    B = 70
    x2, l2 = pair_inputs(B, seed=4)
    W, b = _rand_layer_state(500, 784, seed=9)
    layer = ff.Layer(784, 500, prec=prec)
    layer.set_state(W=W, b=b)
    g = torch.empty(2 * B, device="cuda")
    layer.forward(torch.from_numpy(x2).cuda(), labels=torch.from_numpy(l2).cuda(), goodness=g)
    torch.cuda.synchronize()
    ref = fo.layer_forward_full(fo.LayerState(W, b), fo.overlay_label(x2, l2), emulate_bf16=(prec == "bf16"))
    assert_close(g.cpu().numpy(), ref["g"], 1e-5 if prec == "fp32" else 1e-3, 1e-6, "goodness")
    plain = fo.layer_forward_full(fo.LayerState(W, b), fo.overlay_label(x2, l2))
    assert_close(g.cpu().numpy(), plain["g"], 1e-4 if prec == "fp32" else 2e-2, 1e-4, "goodness vs fp64")


# ------------------------------------------------------------ train step
STEP_CASES = [
    ("fp32", 64, 784, 500, True), ("bf16", 64, 784, 500, True), ("bf16", 3, 11, 5, True), ("fp32", 1, 11, 5, True),
    ("bf16", 1024, 784, 2000, True), ("bf16", 1024, 2000, 2000, False), ("fp32", 150, 2000, 300, False),
    ("bf16", 608, 2000, 2000, False),
    # two-subtile GEMMs with ragged row tiles and a partial last 32-deep K step of the
    # weight gradient (2000 batch rows)
    ("bf16", 1000, 2000, 2000, False),
    # the Adam update's element-wise form (N*K not a multiple of 8, or a padded bf16 copy of W)
    ("fp32", 33, 20, 7, False), ("bf16", 40, 20, 6, False),
]


@pytest.mark.parametrize("prec,B,K,N,first", STEP_CASES)
def test_train_step(env, prec, B, K, N, first):
    torch, ff = env
    M = 2 * B
    theta, lr = 2.0, 0.03
    W, b = _rand_layer_state(N, K, seed=B + K)
    layer = ff.Layer(K, N, prec=prec, theta=theta, lr=lr, keep_grad=True)
    layer.set_state(W=W, b=b)
    if first:
        x2, l2 = pair_inputs(B, seed=B, features=K) if K >= 784 else pair_inputs(B, seed=B, features=K)
        xin = fo.overlay_label(x2, l2)
        xg, lg = torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda()
    else:
        rng = np.random.default_rng(B)
        xin = np.maximum(rng.standard_normal((M, K)), 0).astype(np.float32)
        if prec == "bf16":
            xin = fo.bf16_round(xin).astype(np.float32)
        xg = layer.new_activation(M, K)
        xg[:, :K] = torch.from_numpy(xin).to(xg.dtype)
        lg = None
    g = torch.empty(M, device="cuda")
    loss = torch.empty(1, device="cuda")
    h = layer.new_activation(M)
    sn = torch.empty(M, device="cuda")
    layer.train_step(xg, labels=lg, B=B, h_out=h, next_scale=sn, goodness=g, loss=loss)
    torch.cuda.synchronize()
    layer.check()
    emul = prec == "bf16"
    st = fo.LayerState(W, b)
    ref = fo.layer_train_step(st, xin, B, theta, fo.AdamHyper(lr=lr), emulate_bf16=emul)
    gtol = 1e-5 if not emul else 1e-3
    assert_close(g.cpu().numpy(), ref["g"], gtol, 1e-6, "goodness")
    assert abs(loss.item() - ref["loss"]) <= (1e-5 if not emul else 1e-3) * abs(ref["loss"]) + 1e-7
    dW, db = layer.get_grad()
    assert rel_norm(dW, ref["dW"]) < (1e-5 if not emul else 1e-3), rel_norm(dW, ref["dW"])
    assert rel_norm(db, ref["db"]) < (1e-5 if not emul else 1e-3), rel_norm(db, ref["db"])
    s2 = layer.get_state()
    assert s2["t"] == 1
    dgW, dgb = grad_uncertainty(ref, W, b, xin, B, emul, tensor_cores=emul)
    assert np.all(np.abs(dW - ref["dW"]) <= dgW + 1e-6 * np.abs(ref["dW"])), "dW outside its rounding bound"
    assert np.all(np.abs(db - ref["db"]) <= dgb + 1e-6 * np.abs(ref["db"])), "db outside its rounding bound"
    hp = fo.AdamHyper(lr=lr)
    z = np.zeros_like(W, dtype=np.float64)
    zb = np.zeros_like(b, dtype=np.float64)
    # the Adam kernel applied to the GPU's own gradient, with the float32 hyper-parameters: tight
    hp32 = fo.AdamHyper(*[float(np.float32(v)) for v in (lr, 0.9, 0.999, 1e-8)])
    assert_adam_state(s2["W"], s2["mW"], s2["vW"], W, z, z, 1, dW.astype(np.float64), 0 * z, hp32, "W (own grad)",
                      rtol=1e-5, w_floor=0.05, max_band_frac=0.0)
    # against the oracle's gradient: 1e-4 plus Adam's spread over the rounding bound
    assert_adam_state(s2["W"], s2["mW"], s2["vW"], W, z, z, 1, ref["dW"], dgW, hp, "W")
    assert_adam_state(s2["b"], s2["mb"], s2["vb"], b, zb, zb, 1, ref["db"], dgb, hp, "b")
    assert rel_norm(s2["W"], st.W) <= (1e-4 if not emul else 2e-2)
    # the activity handed to the next layer and its scale
    assert_close(h.float().cpu().numpy()[:, :N], ref["H"], 1e-5 if not emul else 2.0 ** -8 + 1e-3, 1e-5, "activity")
    assert_close(sn.cpu().numpy(), 1.0 / np.maximum(np.sqrt(ref["g"]), 1e-12), gtol, 0, "next scale")
    # against the plain fp64 definition, at the tolerances of each precision
    plain = fo.layer_train_step(fo.LayerState(W, b), xin, B, theta, fo.AdamHyper(lr=lr))
    if not emul:
        assert_close(g.cpu().numpy(), plain["g"], 1e-4, 1e-4, "goodness vs fp64")
    else:
        # bf16 operands: x and W each round by at most 2^-8 of their value, so
        # |dz_ij| <= 2^-7 s_i sum_k |x_ik w_jk| and |dg_i| <= sum_j 2|h_ij||dz_ij| + dz_ij^2
        xa = np.abs(np.asarray(xin, np.float64))
        s_row = 1.0 / np.maximum(np.sqrt((xa * xa).sum(axis=1)), 1e-12)
        ez = 2.0 ** -7 * (xa * s_row[:, None]) @ np.abs(np.asarray(W, np.float64)).T
        gb = (2.0 * np.abs(plain["H"]) * ez + ez * ez).sum(axis=1)
        err = np.abs(g.cpu().numpy() - plain["g"])
        assert np.all(err <= 1e-3 * plain["g"] + gb + 1e-7), float(np.max(err / (1e-3 * plain["g"] + gb + 1e-7)))
        assert np.mean(err <= 2e-2 * plain["g"] + 1e-4) >= 0.95   # the 2e-2 tolerance, all but a few tiny rows
    assert abs(loss.item() - plain["loss"]) <= (1e-4 if not emul else 2e-2) * abs(plain["loss"])


def test_config0_sixteen_steps_fp32(env):
    """784->500->500, fp32, 16 steps of B=64: each step is compared with the
    oracle started from the GPU's state before that step."""
    torch, ff = env
    theta, lr, B = 2.0, 0.03, 64
    layers = [ff.Layer(784, 500, prec="fp32", theta=theta, lr=lr, init_seed=0, keep_grad=True),
              ff.Layer(500, 500, prec="fp32", theta=theta, lr=lr, init_seed=1, keep_grad=True)]
    h = layers[0].new_activation(2 * B)
    s1 = torch.empty(2 * B, device="cuda")
    loss = torch.empty(2, device="cuda")
    g = torch.empty(2, 2 * B, device="cuda")
    for step in range(16):
        x = synth.mnist_like(B, seed=0, start_row=step * B)
        y = synth.labels(B, seed=0, start=step * B)
        yn = synth.negative_labels(y, seed=0, start=step * B)
        x2, l2 = synth.pair_batch(x, y, yn)
        pre = [oracle_state(l.get_state()) for l in layers]
        layers[0].train_step(torch.from_numpy(x2).cuda(), labels=torch.from_numpy(l2).cuda(), B=B, h_out=h,
                             next_scale=s1, goodness=g[0], loss=loss[0:1])
        layers[1].train_step(h, row_scale=s1, B=B, goodness=g[1], loss=loss[1:2])
        torch.cuda.synchronize()
        refs = fo.net_train_step([p.copy() for p in pre], x2, l2, B, theta, fo.AdamHyper(lr=lr))
        xins = [fo.overlay_label(x2, l2), refs[0]["H"]]
        for k in range(2):
            assert_close(g[k].cpu().numpy(), refs[k]["g"], 1e-4, 1e-6, f"step {step} layer {k} goodness")
            assert abs(loss[k].item() - refs[k]["loss"]) <= 1e-4 * abs(refs[k]["loss"])
            st = layers[k].get_state()
            dgW, dgb = grad_uncertainty(refs[k], pre[k].W, pre[k].b, xins[k], B, False, tensor_cores=False)
            hp = fo.AdamHyper(lr=lr)
            p = pre[k]
            assert_adam_state(st["W"], st["mW"], st["vW"], p.W, p.mW, p.vW, step + 1, refs[k]["dW"], dgW, hp,
                              f"step {step} layer {k} W")
            assert_adam_state(st["b"], st["mb"], st["vb"], p.b, p.mb, p.vb, step + 1, refs[k]["db"], dgb, hp,
                              f"step {step} layer {k} b")
            assert st["t"] == step + 1


# ---------------------------------------------------------------- predict
@pytest.mark.parametrize("prec,dims,n", [("fp32", (784, 256, 256, 128), 300), ("bf16", (784, 256, 256, 128), 300),
                                         ("bf16", (784, 96), 40), ("bf16", (784, 200, 128), 9000),
                                         # fp32 on the tensor cores (three TF32 products) at several tile
                                         # shapes, and widths that are not multiples of 4 (CUDA-core GEMMs)
                                         ("fp32", (784, 200, 128), 3000), ("fp32", (786, 130, 66), 250)])
def test_predict(env, prec, dims, n):
    torch, ff = env
    layers, states = [], []
    for i in range(len(dims) - 1):
        W, b = _rand_layer_state(dims[i + 1], dims[i], seed=30 + i, bias_scale=0.02)
        l = ff.Layer(dims[i], dims[i + 1], prec=prec)
        l.set_state(W=W, b=b)
        layers.append(l)
        states.append(fo.LayerState(W, b))
    x = synth.mnist_like(n, seed=31, features=dims[0])
    G = torch.empty(n, 10, device="cuda")
    pred, _ = ff.predict(layers, torch.from_numpy(x).cuda(), goodness=G)
    torch.cuda.synchronize()
    layers[0].check()
    emul = prec == "bf16"
    rp, rG = fo.predict(states, x, emulate_bf16=emul)
    assert_close(G.cpu().numpy(), rG, 1e-4 if not emul else 2e-3, 1e-6, "predict goodness")
    p = pred.cpu().numpy()
    agree = np.mean(p == rp)
    assert agree >= 0.995, agree
    for i in np.nonzero(p != rp)[0]:   # disagreements only at near ties
        gap = abs(rG[i, p[i]] - rG[i, rp[i]])
        assert gap <= (1e-4 if not emul else 1e-2) * abs(rG[i, rp[i]]), (i, gap)
    plain_p, plain_G = fo.predict(states, x)
    assert_close(G.cpu().numpy(), plain_G, 1e-4 if not emul else 2e-2, 1e-4, "predict goodness vs fp64")


# ------------------------------------------------ AdaptiveNEG negatives (§5)
@pytest.mark.parametrize("prec,dims,n", [("fp32", (784, 256, 256, 128), 300), ("bf16", (784, 256, 256, 128), 300),
                                         ("bf16", (784, 96), 40), ("bf16", (784, 200, 128), 9000)])
def test_adaptive_negatives(env, prec, dims, n):
    torch, ff = env
    layers, states = [], []
    for i in range(len(dims) - 1):
        W, b = _rand_layer_state(dims[i + 1], dims[i], seed=50 + i, bias_scale=0.02)
        l = ff.Layer(dims[i], dims[i + 1], prec=prec)
        l.set_state(W=W, b=b)
        layers.append(l)
        states.append(fo.LayerState(W, b))
    x = synth.mnist_like(n, seed=51)
    y = synth.labels(n, seed=52)
    G = torch.empty(n, 10, device="cuda")
    neg, _ = ff.adaptive_negatives(layers, torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda(), goodness=G)
    torch.cuda.synchronize()
    layers[0].check()
    g = G.cpu().numpy()
    p = neg.cpu().numpy()
    # the kernel's choice is exactly the masked argmax of its own goodness
    own = g.copy()
    own[np.arange(n), y] = -np.inf
    assert np.array_equal(p, np.argmax(own, axis=1))
    assert not np.any(p == y)
    emul = prec == "bf16"
    rn, rG = fo.adaptive_negatives(states, x, y, emulate_bf16=emul)
    assert_close(g, rG, 1e-4 if not emul else 2e-3, 1e-6, "adaptive-negative goodness")
    assert np.mean(p == rn) >= 0.995
    for i in np.nonzero(p != rn)[0]:   # disagreements only at near ties
        gap = abs(rG[i, p[i]] - rG[i, rn[i]])
        assert gap <= (1e-4 if not emul else 1e-2) * abs(rG[i, rn[i]]), (i, gap)


def test_adaptive_negatives_label_outside_range_is_plain_prediction(env):
    torch, ff = env
    layers = [ff.Layer(784, 128, prec="bf16", init_seed=60), ff.Layer(128, 128, prec="bf16", init_seed=61)]
    x = torch.from_numpy(synth.mnist_like(64, seed=62)).cuda()
    y = torch.full((64,), -1, dtype=torch.int32, device="cuda")
    y[::2] = 10
    neg, _ = ff.adaptive_negatives(layers, x, y)
    pred, _ = ff.predict(layers, x)
    torch.cuda.synchronize()
    assert torch.equal(neg, pred)
    empty = torch.empty(0, 784, device="cuda")
    ff.adaptive_negatives(layers, empty, torch.empty(0, dtype=torch.int32, device="cuda"))


# ------------------------------------------------- one image per pair == stacked pairs
@pytest.mark.parametrize("prec", ["bf16", "fp32"])
def test_net_step_with_one_image_per_pair_equals_stacked_pairs(env, prec):
    torch, ff = env
    dims, Bmax = (784, 192, 160), 96
    mk = lambda: [ff.Layer(dims[i], dims[i + 1], prec=prec, init_seed=70 + i) for i in range(2)]
    a, b = mk(), mk()
    net_a, net_b = ff.Net(a, max_B=Bmax, depth=2), ff.Net(b, max_B=Bmax, depth=2)
    Bs = [96, 37, 96, 1]                                  # full and ragged batches
    la = torch.empty(len(Bs), 2, device="cuda")
    lb = torch.empty(len(Bs), 2, device="cuda")
    for t, B in enumerate(Bs):
        x2, l2 = pair_inputs(B, seed=300 + t)
        assert np.array_equal(x2[:B], x2[B:])             # the pair rows share their image
        lg = torch.from_numpy(l2).cuda()
        net_a.train_step(torch.from_numpy(x2).cuda(), lg, B=B, loss=la[t])
        net_b.train_step_images(torch.from_numpy(np.ascontiguousarray(x2[:B])).cuda(), lg, loss=lb[t])
    net_a.sync()
    net_b.sync()
    torch.cuda.synchronize()
    assert torch.equal(la, lb)
    for p, q in zip(a, b):
        sp, sq = p.get_state(), q.get_state()
        for k in ("W", "b", "mW", "vW"):
            assert np.array_equal(sp[k], sq[k]), k
    with pytest.raises(ValueError):
        net_b.train_step_images(torch.zeros(4, 784, device="cuda"), torch.zeros(4, dtype=torch.int32, device="cuda"))


# ----------------------------------------------- multi-stream net == sequential
def test_net_on_streams_is_bitwise_sequential(env):
    torch, ff = env
    dims, B, steps = (784, 256, 256, 192), 128, 6
    mk = lambda: [ff.Layer(dims[i], dims[i + 1], prec="bf16", init_seed=40 + i) for i in range(3)]
    par, seq = mk(), mk()
    net = ff.Net(par, max_B=B, depth=2)
    hs = [seq[0].new_activation(2 * B), seq[1].new_activation(2 * B)]
    ss = [torch.empty(2 * B, device="cuda") for _ in range(2)]
    lp = torch.empty(steps, 3, device="cuda")
    ls = torch.empty(steps, 3, device="cuda")
    xs = []
    for t in range(steps):
        x2, l2 = pair_inputs(B, seed=100 + t)
        xs.append((torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda()))
    for t in range(steps):
        net.train_step(xs[t][0], xs[t][1], B=B, loss=lp[t])
    net.sync()
    for t in range(steps):
        seq[0].train_step(xs[t][0], labels=xs[t][1], B=B, h_out=hs[0], next_scale=ss[0], loss=ls[t, 0:1])
        seq[1].train_step(hs[0], row_scale=ss[0], B=B, h_out=hs[1], next_scale=ss[1], loss=ls[t, 1:2])
        seq[2].train_step(hs[1], row_scale=ss[1], B=B, loss=ls[t, 2:3])
    torch.cuda.synchronize()
    assert torch.equal(lp, ls)
    for a, b in zip(par, seq):
        sa, sb = a.get_state(), b.get_state()
        for k in ("W", "b", "mW", "vW"):
            assert np.array_equal(sa[k], sb[k]), k


def test_net_on_streams_is_bitwise_sequential_full_width(env):
    """The same at the width the epoch runs: 784-2000-2000-2000, batches of
    1000 and 1024 pairs, so the layers' two-subtile GEMMs (ragged row tiles,
    a partial last K step of the weight gradient) run concurrently on the
    layer streams; every layer's loss and state bitwise equal to the layers
    stepped one after another."""
    torch, ff = env
    dims, Bs = (784, 2000, 2000, 2000), (1000, 1024, 1000)
    L = len(dims) - 1
    mk = lambda: [ff.Layer(dims[i], dims[i + 1], prec="bf16", init_seed=140 + i) for i in range(L)]
    par, seq = mk(), mk()
    net = ff.Net(par, max_B=max(Bs), depth=2)
    hs = [seq[k].new_activation(2 * max(Bs)) for k in range(L - 1)]
    ss = [torch.empty(2 * max(Bs), device="cuda") for _ in range(L - 1)]
    lp = torch.empty(len(Bs), L, device="cuda")
    ls = torch.empty(len(Bs), L, device="cuda")
    xs = []
    for t, B in enumerate(Bs):
        x2, l2 = pair_inputs(B, seed=300 + t)
        xs.append((torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda()))
    for t, B in enumerate(Bs):
        net.train_step(xs[t][0], xs[t][1], B=B, loss=lp[t])
    net.sync()
    for t, B in enumerate(Bs):
        M = 2 * B
        seq[0].train_step(xs[t][0], labels=xs[t][1], B=B, h_out=hs[0][:M], next_scale=ss[0][:M], loss=ls[t, 0:1])
        for k in range(1, L):
            last = k == L - 1
            seq[k].train_step(hs[k - 1][:M], row_scale=ss[k - 1][:M], B=B,
                              h_out=None if last else hs[k][:M], next_scale=None if last else ss[k][:M],
                              loss=ls[t, k:k + 1])
    torch.cuda.synchronize()
    assert torch.equal(lp, ls)
    for a, b in zip(par, seq):
        sa, sb = a.get_state(), b.get_state()
        for k in ("W", "b", "mW", "vW"):
            assert np.array_equal(sa[k], sb[k]), k


def test_repeat_runs_are_bitwise_equal(env):
    torch, ff = env
    B = 256
    x2, l2 = pair_inputs(B, seed=77)
    outs = []
    for _ in range(2):
        l = ff.Layer(784, 2000, prec="bf16", init_seed=3)
        loss = torch.empty(3, device="cuda")
        for t in range(3):
            l.train_step(torch.from_numpy(x2).cuda(), labels=torch.from_numpy(l2).cuda(), B=B, loss=loss[t:t + 1])
        torch.cuda.synchronize()
        outs.append((loss.cpu().numpy(), l.get_state()["W"]))
    assert np.array_equal(outs[0][0], outs[1][0]) and np.array_equal(outs[0][1], outs[1][1])


def test_dropped_gradient_lines_change_nothing(env):
    """Without keep_grad the Adam kernel drops dW's L2 lines once read (and
    the local-gradient operand's); a layer that keeps its gradient does not
    drop dW.  Both train a hidden and a first layer bit for bit alike over
    several steps, at a size whose state does not fit in L2."""
    torch, ff = env
    B = 1024
    x2, l2 = pair_inputs(B, seed=78)
    xg, lg = torch.from_numpy(x2).cuda(), torch.from_numpy(l2).cuda()
    outs = []
    for keep in (True, False):
        l1 = ff.Layer(784, 2000, prec="bf16", init_seed=5, keep_grad=keep)
        l2_ = ff.Layer(2000, 2000, prec="bf16", init_seed=6, keep_grad=keep)
        h = l1.new_activation(2 * B)
        sc = torch.empty(2 * B, device="cuda")
        loss = torch.empty(4, 2, device="cuda")
        for t in range(4):
            l1.train_step(xg, labels=lg, B=B, h_out=h, next_scale=sc, loss=loss[t, 0:1])
            l2_.train_step(h, row_scale=sc, B=B, loss=loss[t, 1:2])
        torch.cuda.synchronize()
        l1.check()
        l2_.check()
        outs.append((loss.cpu().numpy(), [l.get_state() for l in (l1, l2_)]))
    assert np.array_equal(outs[0][0], outs[1][0])
    for a, b in zip(outs[0][1], outs[1][1]):
        for k in ("W", "b", "mW", "vW", "mb", "vb"):
            assert np.array_equal(np.asarray(a[k]), np.asarray(b[k])), k


# ---------------------------------------------------------------- edges
def test_edge_cases(env):
    torch, ff = env
    l = ff.Layer(784, 300, prec="bf16", init_seed=2)
    before = l.get_state()
    x2, l2 = pair_inputs(4, seed=1)
    l.train_step(torch.from_numpy(x2).cuda(), labels=torch.from_numpy(l2).cuda(), B=0)  # empty batch: no-op
    after = l.get_state()
    assert after["t"] == 0 and np.array_equal(before["W"], after["W"])
    # misaligned activation pointer is rejected before anything runs
    buf = torch.zeros(2 * 4 * 784 + 8, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ff.FFError) as ei:
        l.forward(buf[1:1 + 8 * 784].view(8, 784), goodness=torch.empty(8, device="cuda"))
    assert ei.value.status == 1
    # a non-finite input is latched and reported by check()
    bad = x2.copy()
    bad[0, 20] = np.nan
    l.train_step(torch.from_numpy(bad).cuda(), labels=torch.from_numpy(l2).cuda(), B=4)
    with pytest.raises(ff.FFError) as ei:
        l.check()
    assert ei.value.status == 5
    l.check()  # cleared
    # a batch larger than the workspace grows it
    big = ff.Layer(784, 64, prec="bf16", max_rows=16)
    x3, l3 = pair_inputs(300, seed=2)
    loss = torch.empty(1, device="cuda")
    big.train_step(torch.from_numpy(x3).cuda(), labels=torch.from_numpy(l3).cuda(), B=300, loss=loss)
    torch.cuda.synchronize()
    assert np.isfinite(loss.item())


def test_state_round_trip_resumes_bitwise(env):
    """8 steps, save, load into a fresh layer, 8 more == 16 steps."""
    torch, ff = env
    B = 64
    batches = [pair_inputs(B, seed=200 + t) for t in range(16)]
    a = ff.Layer(784, 500, prec="bf16", init_seed=9)
    for t in range(16):
        a.train_step(torch.from_numpy(batches[t][0]).cuda(), labels=torch.from_numpy(batches[t][1]).cuda(), B=B)
    b = ff.Layer(784, 500, prec="bf16", init_seed=9)
    for t in range(8):
        b.train_step(torch.from_numpy(batches[t][0]).cuda(), labels=torch.from_numpy(batches[t][1]).cuda(), B=B)
    saved = b.get_state()
    c = ff.Layer(784, 500, prec="bf16", init_seed=123)
    c.set_state(**saved)
    for t in range(8, 16):
        c.train_step(torch.from_numpy(batches[t][0]).cuda(), labels=torch.from_numpy(batches[t][1]).cuda(), B=B)
    sa, sc = a.get_state(), c.get_state()
    for k in ("W", "b", "mW", "vW", "mb", "vb"):
        assert np.array_equal(sa[k], sc[k]), k
    assert sa["t"] == sc["t"] == 16


def test_net_steps_captured_in_a_cuda_graph_match_eager(env):
    """A synced run of ff_net steps replayed from a CUDA graph gives the same
    bits as the same steps called eagerly."""
    torch, ff = env
    dims, B = (784, 256, 128), 64
    mk = lambda: [ff.Layer(dims[i], dims[i + 1], prec="bf16", init_seed=60 + i, max_rows=2 * B) for i in range(2)]
    ga, gb = mk(), mk()
    na, nb = ff.Net(ga, max_B=B, depth=2), ff.Net(gb, max_B=B, depth=2)
    xs = [pair_inputs(B, seed=300 + t) for t in range(3)]
    X = torch.from_numpy(np.concatenate([x for x, _ in xs])).cuda()
    L = torch.from_numpy(np.concatenate([l for _, l in xs])).cuda()
    la = torch.zeros(3, 2, device="cuda")
    lb = torch.zeros(3, 2, device="cuda")
    s = torch.cuda.Stream()

    def run(net, loss):
        for t in range(3):
            net.train_step(X[2 * B * t:2 * B * (t + 1)], L[2 * B * t:2 * B * (t + 1)], B=B, loss=loss[t], stream=s)
        net.sync(s)

    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        run(na, la)
    for _ in range(2):
        g.replay()
    with torch.cuda.stream(s):
        for _ in range(2):
            run(nb, lb)
    torch.cuda.synchronize()
    assert torch.equal(la, lb)
    for a, b in zip(ga, gb):
        sa, sb = a.get_state(), b.get_state()
        assert sa["t"] == sb["t"] == 6
        for k in ("W", "b", "mW", "vW"):
            assert np.array_equal(sa[k], sb[k]), k


# ------------------------------------------------ wide net (3072-8192x4)
def test_wide_first_layer_train_step_full_size(env):
    """3072 -> 8192, B = 4096 pairs, theta = 8: the wide workload's first layer
    at full size against the bf16-emulating oracle."""
    torch, ff = env
    B, K, N, theta, lr = 4096, 3072, 8192, 8.0, 0.03
    x = synth.cifar_like(B, seed=41)
    y = synth.labels(B, seed=41)
    x2, l2 = synth.pair_batch(x, y, synth.negative_labels(y, seed=41))
    layer = ff.Layer(K, N, prec="bf16", theta=theta, lr=lr, init_seed=3000, keep_grad=True, max_rows=2 * B)
    W = layer.get_state()["W"]
    g = torch.empty(2 * B, device="cuda")
    loss = torch.empty(1, device="cuda")
    layer.train_step(torch.from_numpy(x2).cuda(), labels=torch.from_numpy(l2).cuda(), B=B, goodness=g, loss=loss)
    torch.cuda.synchronize()
    layer.check()
    st = fo.LayerState(W, np.zeros(N))
    ref = fo.layer_train_step(st, fo.overlay_label(x2, l2), B, theta, fo.AdamHyper(lr=lr), emulate_bf16=True)
    assert_close(g.cpu().numpy(), ref["g"], 1e-3, 1e-6, "goodness")
    assert abs(loss.item() - ref["loss"]) <= 1e-3 * abs(ref["loss"]) + 1e-7
    dW, db = layer.get_grad()
    assert rel_norm(dW, ref["dW"]) < 1e-3 and rel_norm(db, ref["db"]) < 1e-3
    assert rel_norm(layer.get_state()["W"], st.W) < 2e-2


def test_wide_hidden_layer_forward_sampled_rows(env):
    """8192 -> 8192 over 8192 rows (the wide workload's hidden layer, as the
    bench launches it); the oracle checks 256 sampled rows one by one."""
    torch, ff = env
    M, K, N = 8192, 8192, 8192
    layer = ff.Layer(K, N, prec="bf16", init_seed=3001, max_rows=M)
    st = layer.get_state()
    xin = torch.relu(torch.randn(M, K, device="cuda", generator=torch.Generator("cuda").manual_seed(3))).to(
        torch.bfloat16)
    xa = layer.new_activation(M, K)
    xa[:, :K] = xin
    g = torch.empty(M, device="cuda")
    h = layer.new_activation(M)
    layer.forward(xa, h_out=h, goodness=g)
    torch.cuda.synchronize()
    rows = np.sort(np.random.default_rng(4).choice(M, 256, replace=False))
    xs = xin[rows].float().cpu().numpy().astype(np.float64)
    ref = fo.layer_forward_full(fo.LayerState(st["W"], st["b"]), xs, emulate_bf16=True)
    assert_close(g.cpu().numpy()[rows], ref["g"], 1e-3, 1e-6, "sampled goodness")
    assert_close(h[rows].float().cpu().numpy()[:, :N], ref["H"], 2.0 ** -8 + 1e-3, 1e-5, "sampled activity")


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_step_statistics(env, prec):
    """ff_layer_get_stats after a train step: the mean goodness of the
    positive and of the negative rows and the active-ReLU fraction, against
    the oracle's forward of the same step."""
    torch, ff = env
    B, K, N = 96, 784, 300
    layer = ff.Layer(K, N, prec=prec, init_seed=3)
    assert layer.stats() == (0.0, 0.0, 0.0)
    W = layer.get_state()["W"]
    x2, l2 = pair_inputs(B, seed=17)
    layer.train_step(torch.from_numpy(x2).cuda(), labels=torch.from_numpy(l2).cuda(), B=B)
    gp, gn, act = layer.stats()
    emul = prec == "bf16"
    ref = fo.layer_forward_full(fo.LayerState(W, np.zeros(N)), fo.overlay_label(x2, l2), emulate_bf16=emul)
    tol = 1e-5 if not emul else 2e-3
    assert gp == pytest.approx(ref["g"][:B].mean(), rel=tol)
    assert gn == pytest.approx(ref["g"][B:].mean(), rel=tol)
    assert act == pytest.approx(float(np.mean(ref["H"] > 0)), abs=1e-3)
