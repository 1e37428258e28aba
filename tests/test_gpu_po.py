"""Performance-Optimized PFF layer (§4): a layer and its own softmax block
trained together by two-layer backpropagation on the GPU, against the
oracle's step, through the C ABI (ff_po_*)."""

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


def _layer(ff, K, N, prec, seed, lr=0.01):
    rng = np.random.default_rng(seed)
    W = synth.he_uniform(seed, N, K)
    b = (rng.standard_normal(N) * 0.05).astype(np.float32)
    l = ff.Layer(K, N, prec=prec, lr=lr, keep_grad=True)
    l.set_state(W=W, b=b)
    return l, W, b


def _block(ff, N, seed, lr=1e-3):
    rng = np.random.default_rng(seed)
    V = (rng.standard_normal((10, N)) * 0.3).astype(np.float32)
    c = (rng.standard_normal(10) * 0.1).astype(np.float32)
    h = ff.Head(N, lr=lr, max_rows=2048)
    h.set_state(V=V, c=c)
    return h, V, c


def _bounds(out, x_in, V, emul):
    """Elementwise bounds on the GPU's gradients: rel times the sum of the
    absolute terms of each product, where a dz term also carries the error of
    dz itself (p/n per logit error).  fp32: 1e-4 covers the sums.  bf16: a
    stored operand (h, s*dZ) may round one bf16 ulp -- at most 2^-7 of its
    value -- away from the emulation, plus 1e-3 for the fp32 sums."""
    rel = 1e-4 if not emul else 2.0 ** -7 + 1e-3
    p = fo.softmax(out["z"])
    n = p.shape[0]
    dzs = np.abs(out["dz"]) + p / n
    H = out["H"]
    s = out["s"]
    xh = s[:, None] * np.abs(fo.bf16_round(x_in) if emul else np.asarray(x_in, np.float64))
    dH = (dzs @ np.abs(np.asarray(V, np.float64))) * (H > 0)
    bW = rel * (dH.T @ xh) + 1e-12
    bb = rel * dH.sum(axis=0) + 1e-12
    bV = rel * (dzs.T @ np.abs(H)) + 1e-12
    return bW, bb, bV


@pytest.mark.parametrize("prec,raw,K,N,n", [("fp32", True, 784, 256, 300), ("bf16", True, 784, 256, 300),
                                            ("bf16", False, 256, 136, 257), ("fp32", False, 200, 96, 64),
                                            # a full-size hidden layer: the forward GEMM's logits
                                            # epilogue on two 128-row subtiles per CTA
                                            ("bf16", False, 2000, 2000, 2048)])
def test_po_step_matches_oracle(env, prec, raw, K, N, n):
    torch, ff = env
    layer, W, b = _layer(ff, K, N, prec, seed=K + N)
    block, V, c = _block(ff, N, seed=N)
    y = synth.labels(n, seed=5)
    emul = prec == "bf16"
    if raw:
        x = synth.mnist_like(n, seed=6, features=K)
        xg = torch.from_numpy(x).cuda()
        x_in = fo.overlay_neutral(x)
    else:
        rng = np.random.default_rng(7)
        x_in = np.maximum(rng.standard_normal((n, K)), 0.0)
        if emul:
            x_in = fo.bf16_round(x_in)
        xg = layer.new_activation(n, K)
        xg[:, :K] = torch.from_numpy(x_in.astype(np.float32)).to(xg.dtype)
    h = layer.new_activation(n)
    sn = torch.empty(n, device="cuda")
    loss = torch.zeros(1, device="cuda")
    yg = torch.from_numpy(y).cuda()
    if raw:
        ff.po_train_step_raw(layer, block, xg, yg, h_out=h, next_scale=sn, loss=loss)
    else:
        ff.po_train_step_act(layer, block, xg, yg, h_out=h, next_scale=sn, loss=loss)
    torch.cuda.synchronize()
    layer.check()
    block.check()
    hpl, hpb = fo.AdamHyper(lr=0.01), fo.AdamHyper(lr=1e-3)
    st, hd = fo.LayerState(W, b), fo.HeadState(V, c)
    out = fo.po_layer_train_step(st, hd, x_in, y, hpl, hpb, emulate_bf16=emul)
    tol = 1e-5 if not emul else 1e-3
    assert abs(loss.item() - out["loss"]) <= tol * out["loss"], (loss.item(), out["loss"])
    # the activity and the next layer's scale handed on (pre-update weights)
    assert_close(h.float().cpu().numpy()[:, :N], out["H"], 1e-5 if not emul else 2.0 ** -8 + 1e-3, 1e-5, "activity")
    assert_close(sn.cpu().numpy(), 1.0 / np.maximum(np.sqrt(out["g"]), 1e-12), 1e-5 if not emul else 2e-3, 0,
                 "next scale")
    bW, bb, bV = _bounds(out, x_in, V, emul)
    dW, db = layer.get_grad()
    dV, dc = block.get_grad()
    for name, got, ref, bd in (("dW", dW, out["dW"], bW), ("db", db, out["db"], bb), ("dV", dV, out["dV"], bV)):
        err = np.abs(got - ref)
        assert np.all(err <= bd), (name, float(np.max(err / bd)))
        assert rel_norm(got, ref) < (1e-5 if not emul else 2e-3), (name, rel_norm(got, ref))
    assert_close(dc, out["dc"], 1e-4 if not emul else 2e-3, 1e-7, "dc")
    ls, bs = layer.get_state(), block.get_state()
    assert ls["t"] == 1 and bs["t"] == 1
    z = np.zeros_like(W, dtype=np.float64)
    # the Adam kernels applied to the GPU's own gradients, with the float32 hyper-parameters: tight
    f32 = lambda hp: fo.AdamHyper(*[float(np.float32(v)) for v in (hp.lr, hp.beta1, hp.beta2, hp.eps)])
    assert_adam_state(ls["W"], ls["mW"], ls["vW"], W, z, z, 1, dW.astype(np.float64), 0 * z, f32(hpl), "W (own grad)",
                      rtol=1e-5, w_floor=0.05, max_band_frac=0.0)
    # The weight gradient is the contraction dW = G^T A of the stored operand G = s*dZ.  In
    # bf16 mode G rounds to a neighbouring bf16 value wherever the GPU's fp32 dz and the
    # oracle's fp64 dz straddle a rounding boundary, which over a 2048-row contraction moves
    # a few % of dW elements past 1e-4 relative of the oracle's own dW (each inside bW, checked
    # above).  So the step is checked link by link instead:
    #  (1) the GPU's G against the oracle's, element by element, within one bf16 rounding plus
    #      the rounding bound of its ten-term dot product (apart from a few elements at ReLU
    #      kinks, where the mask itself may differ);
    #  (2) the GPU's dW against the oracle's contraction of the GPU's own G (fp32 sums);
    #  (3) the Adam state against the oracle's Adam fed that gradient, at most 5 % of the
    #      elements needing the spread of its rounding bound.
    G = layer.get_grad_operand(n)[:, :N]
    sdz = out["s"][:, None] * out["dZ"]
    Gref = fo.bf16_round(sdz) if emul else sdz
    # dZ_j = sum_c dz_c V_cj sums ten terms whose dz_c add up to zero, so its error is relative
    # to sum_c |dz_c V_cj| (with dz's own error, p/n per logit), not to |dZ_j| (as in _bounds)
    p = fo.softmax(out["z"])
    dHs = ((np.abs(out["dz"]) + p / n) @ np.abs(np.asarray(V, np.float64))) * (out["H"] > 0)
    rel = 2.0 ** -7 + 1e-3 if emul else 1e-4
    gtol = (2.0 ** -7 if emul else 1e-4) * np.abs(Gref) + rel * out["s"][:, None] * dHs + 1e-30
    off = np.abs(G - Gref) > gtol
    # beyond that only where the ReLU mask may differ: z within rounding of 0, i.e. an activity
    # that is (nearly) zero on the oracle's side, and rarely
    assert off.mean() <= 1e-3, ("G elements off", off.mean())
    assert np.all(out["H"][off] <= 1e-4 * float(np.max(out["H"]))), "G differs away from a ReLU kink"
    if emul:
        assert np.mean(G != Gref) <= 0.05, ("G elements a rounding away from the oracle's", np.mean(G != Gref))
    # G carries the row scale, so its contraction partner is the raw layer input (as stored)
    A = fo.bf16_round(x_in) if emul else np.asarray(x_in, np.float64)
    dW_own = G.T @ A
    own_bound = (n + 16) * 2.0 ** -23 * (np.abs(G).T @ np.abs(A)) + 1e-30
    assert np.all(np.abs(dW - dW_own) <= own_bound), ("dW vs own G", float(np.max(np.abs(dW - dW_own) / own_bound)))
    assert_adam_state(ls["W"], ls["mW"], ls["vW"], W, z, z, 1, dW_own, own_bound, hpl, "W", max_band_frac=0.05)
    assert_adam_state(ls["b"], ls["mb"], ls["vb"], b, np.zeros(N), np.zeros(N), 1, out["db"], bb, hpl, "b",
                      max_band_frac=0.05)
    zv = np.zeros_like(V, dtype=np.float64)
    assert_adam_state(bs["V"], bs["mV"], bs["vV"], V, zv, zv, 1, out["dV"], bV, hpb, "V", max_band_frac=0.05)


def test_po_net_learns_and_predicts(env):
    """Two Performance-Optimized layers, fp32, eight steps on a learnable
    task: each step against the oracle started from the GPU's states, the
    loss falls, and the prediction matches the oracle's on the final net."""
    torch, ff = env
    n, dims = 256, (784, 128, 64)
    x, y = synth.learnable_task(n, seed=31)
    xg, yg = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
    layers = [_layer(ff, dims[i], dims[i + 1], "fp32", seed=40 + i, lr=0.003)[0] for i in range(2)]
    blocks = [_block(ff, dims[i + 1], seed=50 + i, lr=0.01)[0] for i in range(2)]
    h1 = layers[0].new_activation(n)
    s1 = torch.empty(n, device="cuda")
    hpl, hpb = fo.AdamHyper(lr=0.003), fo.AdamHyper(lr=0.01)
    first, last = None, None
    for step in range(8):
        pre_l = [l.get_state() for l in layers]
        pre_b = [bk.get_state() for bk in blocks]
        loss = torch.zeros(2, device="cuda")
        ff.po_train_step_raw(layers[0], blocks[0], xg, yg, h_out=h1, next_scale=s1, loss=loss[0:1])
        ff.po_train_step_act(layers[1], blocks[1], h1, yg, row_scale=s1, loss=loss[1:2])
        torch.cuda.synchronize()
        a = fo.overlay_neutral(x)
        for k in range(2):
            st = fo.LayerState(pre_l[k]["W"], pre_l[k]["b"], pre_l[k]["mW"], pre_l[k]["vW"], pre_l[k]["mb"],
                               pre_l[k]["vb"], pre_l[k]["t"])
            hd = fo.HeadState(pre_b[k]["V"], pre_b[k]["c"], pre_b[k]["mV"], pre_b[k]["vV"], pre_b[k]["mc"],
                              pre_b[k]["vc"], pre_b[k]["t"])
            out = fo.po_layer_train_step(st, hd, a, y, hpl, hpb)
            assert abs(loss[k].item() - out["loss"]) <= 1e-4 * out["loss"], (step, k, loss[k].item(), out["loss"])
            a = out["H"]
        if first is None:
            first = loss.cpu().numpy().copy()
        last = loss.cpu().numpy()
    assert np.all(last < first)
    logits = torch.empty(n, 10, device="cuda")
    pred, _ = ff.po_predict(layers, blocks[1], xg, logits=logits)
    torch.cuda.synchronize()
    states = [fo.LayerState(l.get_state()["W"], l.get_state()["b"]) for l in layers]
    bst = blocks[1].get_state()
    rp, rz = fo.po_predict(states, [None, fo.HeadState(bst["V"], bst["c"])], x)
    assert_close(logits.cpu().numpy(), rz, 1e-4, 1e-5, "block logits")
    assert np.mean(pred.cpu().numpy() == rp) >= 0.995


def test_po_argument_errors(env):
    torch, ff = env
    layer, _, _ = _layer(ff, 784, 64, "bf16", seed=9)
    wrong = ff.Head(63)
    x = torch.zeros(4, 784, device="cuda")
    y = torch.zeros(4, dtype=torch.int32, device="cuda")
    with pytest.raises(ff.FFError):
        ff.po_train_step_raw(layer, wrong, x, y)          # block width != layer width
    block = ff.Head(64)
    ff.po_train_step_raw(layer, block, x[:0], y[:0])      # n == 0: no-op
    assert layer.get_state()["t"] == 0
    with pytest.raises(ff.FFError):
        ff.po_predict([layer], wrong, x)


def test_po_net_on_streams_is_bitwise_sequential(env):
    """ff_net_create_po: three Performance-Optimized layers on their own
    streams over five batches (one ragged) give bit for bit the states and
    losses of the same steps issued layer after layer on one stream."""
    torch, ff = env
    dims, rows = (784, 128, 96, 64), [200, 200, 173, 200, 200]

    def make():
        ls = [ff.Layer(dims[i], dims[i + 1], prec="bf16", init_seed=60 + i, lr=0.003) for i in range(3)]
        bs = [ff.Head(dims[i + 1], lr=0.01, max_rows=256) for i in range(3)]
        for i, b in enumerate(bs):
            b.set_state(V=_block(ff, dims[i + 1], seed=70 + i)[1], c=np.zeros(10, np.float32))
        return ls, bs
    data = [(torch.from_numpy(synth.mnist_like(n, seed=80 + t)).cuda(), torch.from_numpy(synth.labels(n, seed=90 + t)).cuda())
            for t, n in enumerate(rows)]
    la, ba = make()
    net = ff.PoNet(la, ba, max_rows=200, depth=2)
    lp = torch.zeros(len(rows), 3, device="cuda")
    for t, (x, y) in enumerate(data):
        net.train_step(x, y, loss=lp[t])
    net.sync()
    lb, bb = make()
    ls = torch.zeros(len(rows), 3, device="cuda")
    for t, (x, y) in enumerate(data):
        n = x.shape[0]
        hs = [lb[k].new_activation(n) for k in range(2)]
        ss = [torch.empty(n, device="cuda") for _ in range(2)]
        ff.po_train_step_raw(lb[0], bb[0], x, y, h_out=hs[0], next_scale=ss[0], loss=ls[t, 0:1])
        ff.po_train_step_act(lb[1], bb[1], hs[0], y, row_scale=ss[0], h_out=hs[1], next_scale=ss[1], loss=ls[t, 1:2])
        ff.po_train_step_act(lb[2], bb[2], hs[1], y, row_scale=ss[1], loss=ls[t, 2:3])
    torch.cuda.synchronize()
    assert torch.equal(lp, ls)
    for a, b in zip(la + ba, lb + bb):
        sa, sb = a.get_state(), b.get_state()
        for k in sa:
            assert np.array_equal(np.asarray(sa[k]), np.asarray(sb[k])), k
    with pytest.raises(ff.FFError):
        net.train_step(data[0][0][:0].new_zeros(300, 784), torch.zeros(300, dtype=torch.int32, device="cuda"))
