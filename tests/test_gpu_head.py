"""Softmax prediction head (§3 "Prediction", Softmax method) on the GPU
against the oracle: features, logits, cross-entropy, gradient, Adam and the
prediction, through the C ABI (ff_head_*)."""

import numpy as np
import pytest

from oracle import ff_oracle as fo
from paper_2404_08573_gb300 import synth

from .gpu_common import assert_adam_state, assert_close, lib_ready, rel_norm, torch_cuda

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    torch = torch_cuda()
    ff = lib_ready()
    return torch, ff


def _net(ff, dims, prec, seed):
    layers, states = [], []
    for i in range(len(dims) - 1):
        rng = np.random.default_rng(seed + i)
        W = synth.he_uniform(seed + i, dims[i + 1], dims[i])
        b = (rng.standard_normal(dims[i + 1]) * 0.05).astype(np.float32)
        l = ff.Layer(dims[i], dims[i + 1], prec=prec)
        l.set_state(W=W, b=b)
        layers.append(l)
        states.append(fo.LayerState(W, b))
    return layers, states


def _feature_dev(states, x, safety=4.0):
    """Bound on how far the GPU's bf16 features may sit from the
    bf16-emulating oracle's, element by element.  Both round the same operands
    at the same points; they differ by fp32 against fp64 accumulation (K 2^-24
    of a pre-activation's absolute scale S = s sum|a||w| + |b|); where that
    difference crosses a bf16 rounding boundary a stored activity differs by
    one step (2^-8 |h|; expected square K 2^-24 S / (2^-8 |h|) x (2^-8 h)^2);
    and the next layers carry the deviations of their inputs.  The deviations
    have independent signs, so they are carried as root-sum-squares (a
    worst-case sum of |w| terms grows ~5x per 2000-wide layer and bounds
    nothing); the result times `safety`.  Where the oracle's ReLU output is 0
    only the pre-activation's deviation applies (the kink).  Features: the
    deviation times the row scale."""
    a = fo.overlay_neutral(x)
    E2 = np.zeros_like(a)
    devs = []
    for k, st in enumerate(states):
        f = fo.layer_forward_full(st, a, emulate_bf16=True)
        Wq = np.abs(fo.bf16_round(st.W))
        K = st.W.shape[1]
        s = f["s"][:, None]
        S = s * (np.abs(f["A"]) @ Wq.T) + np.abs(st.b)
        acc = K * 2.0 ** -24 * S
        E2k = acc ** 2 + s ** 2 * (E2 @ (Wq ** 2).T) + acc * 2.0 ** -8 * np.abs(f["H"])
        if k >= 1 or len(states) == 1:
            scale = 1.0 / np.maximum(np.sqrt(f["g"]), fo.NORM_EPS)
            devs.append(safety * scale[:, None] * np.sqrt(E2k))
        a, E2 = f["H"], E2k
    return np.concatenate(devs, axis=1)


def _grad_bound(out, A, emul, V=None, dev=None):
    """Elementwise bound on |dV_gpu - dV_exact|: the fp32 sum of |dz||a| terms,
    plus the error of dz itself (a logit error moves each probability by at
    most p times twice that error; 1e-4 of the terms p|a|/n covers fp32
    logits, and bf16 activities rounding one ulp away from the emulation).
    With the features' deviation bound dev (bf16) and the head's V: the
    features' own deviation through |dz|^T dev, and the logits' deviation
    (at most max_c sum_j dev |V_cj| per row) through dz."""
    p = fo.softmax(out["z"])
    n = A.shape[0]
    rel = 1e-4 if not emul else 4e-3
    b = rel * ((np.abs(out["dz"]) + p / n).T @ np.abs(A)) + 1e-12
    if dev is not None:
        dzl = (dev @ np.abs(np.asarray(V, dtype=np.float64)).T).max(axis=1, keepdims=True)  # [n, 1]
        ddz = 2.0 * p * dzl / n
        b = b + np.abs(out["dz"]).T @ dev + ddz.T @ (np.abs(A) + dev)
    return b


def _head_state(F, seed, scale=0.5):
    rng = np.random.default_rng(seed)
    V = (rng.standard_normal((10, F)) * scale).astype(np.float32)
    c = (rng.standard_normal(10) * 0.1).astype(np.float32)
    return V, c


CASES = [("fp32", (784, 256, 256, 128), 300), ("bf16", (784, 256, 256, 128), 300), ("bf16", (784, 96), 37),
         ("bf16", (784, 200, 136), 1000),
         # the benchmarked head: layers 2..4 of 784-2000x4 (6000 features), a 1024-row step
         ("bf16", (784, 2000, 2000, 2000, 2000), 1024)]


@pytest.mark.parametrize("prec,dims,n", CASES)
def test_head_train_step_matches_oracle(env, prec, dims, n):
    torch, ff = env
    layers, states = _net(ff, dims, prec, seed=70)
    F = ff.Head.features_of(layers)
    head = ff.Head(F, lr=1e-3, max_rows=1024)
    V, c = _head_state(F, seed=71)
    head.set_state(V=V, c=c)
    x = synth.mnist_like(n, seed=72)
    y = synth.labels(n, seed=73)
    loss = torch.zeros(1, device="cuda")
    head.train_step(layers, torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda(), loss=loss)
    torch.cuda.synchronize()
    head.check()
    emul = prec == "bf16"
    A = fo.softmax_features(states, x, emulate_bf16=emul)
    assert A.shape == (n, F)
    ref_head = fo.HeadState(V, c)
    hp = fo.AdamHyper(lr=1e-3)
    out = fo.head_train_step(ref_head, A, y, hp)
    tol = 1e-5 if not emul else 1e-3
    assert abs(loss.item() - out["loss"]) <= tol * abs(out["loss"]), (loss.item(), out["loss"])
    dV, dc = head.get_grad()
    assert rel_norm(dV, out["dV"]) < (1e-6 if not emul else 1e-3), rel_norm(dV, out["dV"])
    bound = _grad_bound(out, A, emul, V, _feature_dev(states, x) if emul else None)
    assert np.all(np.abs(dV - out["dV"]) <= bound), float(np.max(np.abs(dV - out["dV"]) / bound))
    assert_close(dc, out["dc"], 1e-4 if not emul else 2e-3, 1e-7, "dc")
    st = head.get_state()
    assert st["t"] == 1
    z = np.zeros_like(V, dtype=np.float64)
    zc = np.zeros(10)
    # the Adam update on the GPU's own gradient, tightly (link by link: the
    # gradient is held to the oracle's by the elementwise bound above)
    g_gpu = np.asarray(dV, np.float64)
    assert_adam_state(st["V"], st["mV"], st["vV"], V, z, z, 1, g_gpu, 1e-6 * np.abs(g_gpu) + 1e-12, hp,
                      "V (own gradient)", max_band_frac=1e-3)
    if n * F <= 1_000_000:
        # and on the oracle's gradient within that bound.  (At the full depth
        # of 784-2000x4, bf16 feature deviations move more than 5 % of the dV
        # elements past 1e-4 relative, each inside its bound, so the share of
        # moment elements on the band is not a useful check there.)
        assert_adam_state(st["V"], st["mV"], st["vV"], V, z, z, 1, out["dV"], bound, hp, "V")
    assert_adam_state(st["c"], st["mc"], st["vc"], c, zc, zc, 1, out["dc"], 1e-5 * np.abs(out["dc"]) + 1e-9,
                      hp, "c")


def test_head_several_steps_and_learning(env):
    """Four steps on a learnable task, each compared with the oracle started
    from the GPU's state before it; the loss goes down."""
    torch, ff = env
    dims = (784, 256, 256)
    layers, states = _net(ff, dims, "fp32", seed=80)
    F = ff.Head.features_of(layers)
    head = ff.Head(F, lr=1e-2, max_rows=512)
    x, y = synth.learnable_task(256, seed=81)
    xg, yg = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
    A = fo.softmax_features(states, x)
    hp = fo.AdamHyper(lr=1e-2)
    losses = []
    for step in range(4):
        pre = head.get_state()
        loss = torch.zeros(1, device="cuda")
        head.train_step(layers, xg, yg, loss=loss)
        torch.cuda.synchronize()
        ref = fo.HeadState(pre["V"], pre["c"], pre["mV"], pre["vV"], pre["mc"], pre["vc"], pre["t"])
        out = fo.head_train_step(ref, A, y, hp)
        assert abs(loss.item() - out["loss"]) <= 1e-5 * out["loss"]
        st = head.get_state()
        assert st["t"] == step + 1
        bound = _grad_bound(out, A, False)
        assert_adam_state(st["V"], st["mV"], st["vV"], pre["V"], pre["mV"], pre["vV"], step + 1, out["dV"], bound,
                          hp, f"V step {step}")
        losses.append(loss.item())
    assert losses[-1] < losses[0]
    head.check()


@pytest.mark.parametrize("prec,dims,n,max_rows", [("bf16", (784, 256, 256, 128), 5003, 2048),
                                                  ("fp32", (784, 128, 64), 700, 256), ("bf16", (784, 96), 1, 0),
                                                  # the benchmarked head, over two chunks and a tail
                                                  ("bf16", (784, 2000, 2000, 2000, 2000), 2500, 1024)])
def test_head_predict_matches_oracle(env, prec, dims, n, max_rows):
    torch, ff = env
    layers, states = _net(ff, dims, prec, seed=90)
    F = ff.Head.features_of(layers)
    head = ff.Head(F, max_rows=max_rows)
    V, c = _head_state(F, seed=91, scale=1.0)
    head.set_state(V=V, c=c)
    x = synth.mnist_like(n, seed=92)
    logits = torch.empty(n, 10, device="cuda")
    pred, _ = head.predict(layers, torch.from_numpy(x).cuda(), logits=logits)
    torch.cuda.synchronize()
    head.check()
    emul = prec == "bf16"
    A = fo.softmax_features(states, x, emulate_bf16=emul)
    rp, rz = fo.head_predict(fo.HeadState(V, c), A)
    scale = np.abs(A) @ np.abs(V).T.astype(np.float64) + 1e-6
    err = np.abs(logits.cpu().numpy() - rz)
    assert np.all(err <= (1e-5 if not emul else 2e-3) * scale), float(np.max(err / scale))
    p = pred.cpu().numpy()
    assert np.mean(p == rp) >= 0.995
    for i in np.nonzero(p != rp)[0]:   # disagreements only at near ties
        assert abs(rz[i, p[i]] - rz[i, rp[i]]) <= (1e-5 if not emul else 2e-3) * scale[i].max()
    # the labels of the argmax are the GPU logits' own first maximum
    assert np.array_equal(p, np.argmax(logits.cpu().numpy(), axis=1))


@pytest.mark.parametrize("prec,dims,n,B", [
    ("bf16", (784, 256, 256, 128), 5 * 512 + 100, 512),      # one forward pass, a ragged last step
    ("bf16", (784, 512, 256), 17 * 1024 + 300, 1024),        # two forward passes (16384 rows, then the rest)
    ("fp32", (784, 200, 136), 3 * 256 + 17, 256),
])
def test_head_train_epoch_is_bitwise_the_per_step_calls(env, prec, dims, n, B):
    """ff_head_train_epoch forms many steps' features in one forward pass; its
    steps must give exactly the per-step path's losses and head state."""
    torch, ff = env
    layers, _ = _net(ff, dims, prec, 40)
    F = ff.Head.features_of(layers)
    x = torch.from_numpy(synth.mnist_like(n, seed=41)).cuda()
    y = torch.from_numpy(synth.labels(n, seed=41)).cuda()
    nsteps = -(-n // B)
    ha, hb = ff.Head(F, lr=1e-3, max_rows=B), ff.Head(F, lr=1e-3, max_rows=B)
    la = torch.zeros(nsteps, device="cuda")
    lb = torch.zeros(nsteps, device="cuda")
    ha.train_epoch(layers, x, y, B, loss=la)
    for t in range(nsteps):
        r = t * B
        hb.train_step(layers, x[r:r + B], y[r:r + B], loss=lb[t:t + 1])
    torch.cuda.synchronize()
    ha.check()
    hb.check()
    assert torch.equal(la, lb), ("per-step losses differ", (la - lb).abs().max().item())
    sa, sb = ha.get_state(), hb.get_state()
    for key in sa:
        assert np.array_equal(np.asarray(sa[key]), np.asarray(sb[key])), key
    ha.close()
    hb.close()


def test_head_features_are_unit_norm_segments(env):
    """With V = a selector of one feature per class, the logits are those
    features of A: checks the neutral label, the layer order and the
    per-layer normalisation directly."""
    torch, ff = env
    dims = (784, 64, 48, 32)
    layers, states = _net(ff, dims, "fp32", seed=95)
    F = ff.Head.features_of(layers)
    assert F == 80
    head = ff.Head(F)
    pick = [0, 5, 47, 48, 49, 60, 70, 79, 10, 30]
    V = np.zeros((10, F), np.float32)
    V[np.arange(10), pick] = 1.0
    head.set_state(V=V, c=np.zeros(10, np.float32))
    x = synth.mnist_like(40, seed=96)
    logits = torch.empty(40, 10, device="cuda")
    head.predict(layers, torch.from_numpy(x).cuda(), logits=logits)
    torch.cuda.synchronize()
    A = fo.softmax_features(states, x)
    assert_close(logits.cpu().numpy(), A[:, pick], 1e-5, 1e-7, "selected features")


def test_head_argument_errors(env):
    torch, ff = env
    layers, _ = _net(ff, (784, 64, 32), "bf16", seed=97)
    head = ff.Head(31)                       # wrong feature count for this chain
    x = torch.zeros(4, 784, device="cuda")
    y = torch.zeros(4, dtype=torch.int32, device="cuda")
    with pytest.raises(ff.FFError):
        head.train_step(layers, x, y)
    head2 = ff.Head(32, max_rows=2)
    with pytest.raises(ff.FFError):
        head2.train_step(layers, x, y)       # more rows than max_rows
    head2.train_step(layers, x[:0], y[:0])   # n == 0: no-op
    assert head2.get_state()["t"] == 0
    mixed = [layers[0], ff.Layer(64, 32, prec="fp32")]
    with pytest.raises(ff.FFError):
        head2.predict(mixed, x)
