"""Pins of the CPU oracle against facts fixed by the paper and by mathematics.

None of these compares the oracle with itself: each checks a closed form, an
invariant, a library routine, finite differences, or brute force on tiny
inputs, chosen so that a dropped term, a wrong sign or index, or a transposed
operand in the oracle fails at least one of them.
"""

import json
import math
import os

import numpy as np
import pytest

from oracle import ff_oracle as fo
from paper_2404_08573_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ------------------------------------------------------------ bf16 rounding
def test_bf16_round_matches_torch_conversion():
    """RNE to bfloat16 equals PyTorch's float32 -> bfloat16 conversion."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(1)
    vals = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(5000) * 1e-20).astype(np.float32),
        (rng.standard_normal(5000) * 1e20).astype(np.float32),
    ])
    # exact ties: 8 significant bits plus a half ulp
    base = (rng.integers(128, 256, 2000) * 2 + 1).astype(np.float64)   # odd 9-bit ints
    ties = (base * 2.0 ** rng.integers(-20, 20, 2000)).astype(np.float32)
    vals = np.concatenate([vals, ties, -ties, np.zeros(3, np.float32)])
    ref = torch.from_numpy(vals).to(torch.bfloat16).to(torch.float64).numpy()
    got = fo.bf16_round(vals.astype(np.float64))
    assert np.array_equal(got, ref)


# ------------------------------------------------------------------ overlay
def test_overlay_is_exact_one_hot_and_leaves_rest_untouched():
    x = synth.mnist_like(64, seed=3).astype(np.float64)
    x[:, :10] = 0.37   # nonzero under the label area: overlay must replace
    y = synth.labels(64, seed=3)
    o = fo.overlay_label(x, y)
    assert np.array_equal(o[:, :10], np.eye(10)[y])
    assert np.array_equal(o[:, 10:], x[:, 10:])
    assert np.array_equal(x[:, :10], np.full((64, 10), 0.37))   # input not mutated


# -------------------------------------------------------------- normalise
def test_normalise_unit_norm_zero_row_and_scale_invariance():
    x = synth.mnist_like(200, seed=5).astype(np.float64)
    x[7] = 0.0
    xh = fo.normalise(x)
    n = np.sqrt(np.sum(xh ** 2, axis=1))
    nz = np.arange(200) != 7
    assert np.max(np.abs(n[nz] - 1.0)) <= 4 * np.finfo(np.float64).eps
    assert np.all(xh[7] == 0.0)
    assert np.allclose(fo.normalise(3.5 * x), xh, rtol=0, atol=1e-15)


# --------------------------------------------------------------- goodness
def test_goodness_of_hand_built_layers():
    K = 6
    x = np.abs(np.random.default_rng(2).standard_normal((5, K))) * 3.0   # x >= 0, not unit norm
    st = fo.LayerState(np.eye(K), np.zeros(K))
    f = fo.layer_forward_full(st, x)
    assert np.allclose(f["g"], 1.0, atol=1e-14)           # W = I: g = ||x_hat||^2 = 1
    st = fo.LayerState(-np.eye(K), np.zeros(K))
    assert np.all(fo.layer_forward_full(st, x)["g"] == 0.0)  # W = -I: all units off
    # one active unit: g = z^2
    W = np.zeros((3, 2)); W[1, 0] = 2.0
    b = np.array([-1.0, 0.25, -3.0])
    xx = np.array([[3.0, 4.0]])                           # x_hat = (0.6, 0.8)
    g = fo.layer_forward_full(fo.LayerState(W, b), xx)["g"]
    assert g[0] == pytest.approx((2.0 * 0.6 + 0.25) ** 2, abs=1e-15)


# ------------------------------------------------------------------- loss
def test_loss_closed_forms():
    gold = _golden("closed_forms.json")
    B, theta = 7, 2.0
    g = np.full(2 * B, theta)
    assert fo.ff_loss(g, theta, B) == pytest.approx(gold["loss_at_threshold"], abs=1e-15)
    d = fo.dloss_dg(g, theta, B)
    assert np.allclose(d[:B], -0.5 / B, atol=1e-17) and np.allclose(d[B:], 0.5 / B, atol=1e-17)
    # p(real) at the threshold is 1/2 (Eq. 1)
    assert fo.p_real(theta, theta) == 0.5
    # large margins: positives far above, negatives far below -> loss ~ 0
    g2 = np.concatenate([np.full(B, theta + 60.0), np.full(B, theta - 60.0)])
    assert 0.0 < fo.ff_loss(g2, theta, B) < 2 * math.exp(-59)
    # wrong-way margins: loss ~ 2 * 60 per pair
    g3 = np.concatenate([np.full(B, theta - 60.0), np.full(B, theta + 60.0)])
    assert fo.ff_loss(g3, theta, B) == pytest.approx(120.0, rel=1e-12)
    # mirror: swapping the pos/neg halves and reflecting g about theta keeps L
    rng = np.random.default_rng(4)
    g4 = theta + rng.standard_normal(2 * B)
    g5 = np.concatenate([2 * theta - g4[B:], 2 * theta - g4[:B]])
    assert fo.ff_loss(g5, theta, B) == pytest.approx(fo.ff_loss(g4, theta, B), rel=1e-14)
    # -log p(real) definition for one positive pair member, written out
    p = 1.0 / (1.0 + math.exp(-(g4[0] - theta)))
    q = 1.0 / (1.0 + math.exp(-(g4[B] - theta)))
    one = fo.ff_loss(np.array([g4[0], g4[B]]), theta, 1)
    assert one == pytest.approx(-math.log(p) - math.log(1.0 - q), rel=1e-13)


def test_softplus_stable_branch_agrees_with_naive():
    t = np.linspace(-30, 30, 601)
    assert np.allclose(fo.softplus(t), np.log1p(np.exp(t)), rtol=1e-14, atol=1e-300)
    assert fo.softplus(np.array([800.0]))[0] == 800.0


# -------------------------------------------------------------- gradients
def _layer_loss(W, b, x_in, B, theta):
    f = fo.layer_forward_full(fo.LayerState(W, b), x_in)
    return fo.ff_loss(f["g"], theta, B)


def _fd_check(K, N, B, seed, theta):
    rng = np.random.default_rng(seed)
    for _ in range(100):
        x = np.abs(rng.standard_normal((2 * B, K)))
        W = rng.standard_normal((N, K)) * (1.5 / math.sqrt(K))
        b = rng.standard_normal(N) * 0.3
        z = fo.normalise(x) @ W.T + b
        if np.min(np.abs(z)) > 1e-3:
            break
    else:
        pytest.fail("no kink-free draw")
    st = fo.LayerState(W, b)
    out = fo.layer_train_step(st, x, B, theta, fo.AdamHyper(lr=0.0))
    h = 1e-6
    num_W = np.zeros_like(W)
    for i in range(N):
        for j in range(K):
            Wp = W.copy(); Wp[i, j] += h
            Wm = W.copy(); Wm[i, j] -= h
            num_W[i, j] = (_layer_loss(Wp, b, x, B, theta) - _layer_loss(Wm, b, x, B, theta)) / (2 * h)
    num_b = np.zeros_like(b)
    for i in range(N):
        bp = b.copy(); bp[i] += h
        bm = b.copy(); bm[i] -= h
        num_b[i] = (_layer_loss(W, bp, x, B, theta) - _layer_loss(W, bm, x, B, theta)) / (2 * h)
    scale_W = np.max(np.abs(num_W))
    scale_b = np.max(np.abs(num_b))
    assert np.max(np.abs(out["dW"] - num_W)) <= 1e-6 * scale_W
    assert np.max(np.abs(out["db"] - num_b)) <= 1e-6 * scale_b


def test_gradient_matches_finite_differences_4_to_3():
    _fd_check(K=4, N=3, B=3, seed=10, theta=0.4)


def test_gradient_matches_finite_differences_784_to_16():
    _fd_check(K=784, N=16, B=2, seed=11, theta=0.05)


# ------------------------------------------------------------------- Adam
def test_adam_first_step_closed_form_and_zero_gradient():
    hp = fo.AdamHyper(lr=0.03)
    rng = np.random.default_rng(6)
    w = rng.standard_normal(1000)
    g = rng.standard_normal(1000) * 10.0 ** rng.integers(-9, 2, 1000)
    g[:10] = 0.0
    w1, m1, v1 = fo.adam_update(w, g, np.zeros(1000), np.zeros(1000), 1, hp)
    # w1 - w cancels: allow a few ulps of |w| absolute
    assert np.allclose(w1 - w, -hp.lr * g / (np.abs(g) + hp.eps), rtol=1e-12, atol=1e-15)
    assert np.all(w1[:10] == w[:10])
    # a constant gradient keeps the bias-corrected step at -lr*g/(|g|+eps)
    w_t, m_t, v_t = w1, m1, v1
    for t in range(2, 6):
        w_n, m_t, v_t = fo.adam_update(w_t, g, m_t, v_t, t, hp)
        assert np.allclose(w_n - w_t, -hp.lr * g / (np.abs(g) + hp.eps), rtol=1e-9, atol=1e-14)
        w_t = w_n


def test_adam_two_steps_with_different_gradients_pin_both_decay_rates():
    """Two steps with g1 != g2 (a constant gradient hides beta1 and beta2,
    since then m_hat = g and v_hat = g^2 for any rates).  The expected values
    are worked out by hand with beta1 = 0.9, beta2 = 0.999, lr = 0.03,
    eps = 1e-8 and written as decimals:
      element 0: w0 = 0.5, g1 = 2, g2 = -1
        m1 = 0.2, v1 = 0.004, w1 = 0.5 - 0.06/(2 + 1e-8)
        m2 = 0.08, v2 = 0.004996, m_hat2 = 8/19, v_hat2 = 4996/1999
      element 1: w0 = 0, g1 = 1, g2 = 3
        m1 = 0.1, v1 = 0.001, w1 = -0.03/(1 + 1e-8)
        m2 = 0.39, v2 = 0.009999, m_hat2 = 39/19, v_hat2 = 9999/1999
    (w2 to 40 digits by decimal arithmetic)."""
    hp = fo.AdamHyper(lr=0.03, beta1=0.9, beta2=0.999, eps=1e-8)
    w0 = np.array([0.5, 0.0])
    z = np.zeros(2)
    w1, m1, v1 = fo.adam_update(w0, np.array([2.0, 1.0]), z, z, 1, hp)
    assert np.allclose(m1, [0.2, 0.1], rtol=1e-15, atol=0)
    assert np.allclose(v1, [0.004, 0.001], rtol=1e-14, atol=0)
    assert np.allclose(w1, [0.47000000014999999925, -0.02999999970000000300], rtol=1e-15, atol=1e-16)
    w2, m2, v2 = fo.adam_update(w1, np.array([-1.0, 3.0]), m1, v1, 2, hp)
    assert np.allclose(m2, [0.08, 0.39], rtol=1e-14, atol=0)
    assert np.allclose(v2, [0.004996, 0.009999], rtol=1e-14, atol=0)
    assert np.allclose(w2, [0.46200988901072940735, -0.05753343314630051164], rtol=1e-14, atol=1e-16)


# ---------------------------------------------------------------- predict
def _brute_predict(Ws, bs, x, n_classes=10):
    """Pure-Python loops, no NumPy algebra: overlay, normalise, ReLU layers,
    goodness of layers 2..L, first maximum wins."""
    preds, Gs = [], []
    L = len(Ws)
    for row in x:
        G = [0.0] * n_classes
        for c in range(n_classes):
            a = [0.0] * n_classes + [float(v) for v in row[n_classes:]]
            a[c] = 1.0
            for k in range(L):
                nrm = math.sqrt(sum(v * v for v in a))
                nrm = max(nrm, 1e-12)
                xh = [v / nrm for v in a]
                W, b = Ws[k], bs[k]
                h = []
                for i in range(len(b)):
                    z = b[i]
                    for j in range(len(xh)):
                        z += W[i][j] * xh[j]
                    h.append(z if z > 0 else 0.0)
                if k >= 1 or L == 1:
                    G[c] += sum(v * v for v in h)
                a = h
        best = 0
        for c in range(1, n_classes):
            if G[c] > G[best]:
                best = c
        preds.append(best)
        Gs.append(G)
    return np.array(preds), np.array(Gs)


@pytest.mark.parametrize("dims", [(12, 5, 4, 3), (12, 6)])
def test_predict_matches_brute_force(dims):
    rng = np.random.default_rng(7)
    Ws = [rng.standard_normal((dims[i + 1], dims[i])) for i in range(len(dims) - 1)]
    bs = [rng.standard_normal(dims[i + 1]) * 0.2 for i in range(len(dims) - 1)]
    x = rng.random((50, dims[0]))
    states = [fo.LayerState(W, b) for W, b in zip(Ws, bs)]
    pred, G = fo.predict(states, x)
    bp, bG = _brute_predict([W.tolist() for W in Ws], [b.tolist() for b in bs], x)
    assert np.allclose(G, bG, rtol=1e-12, atol=1e-12)
    assert np.array_equal(pred, bp)


def test_predict_hand_built_label_column_dominates():
    # layer 1 copies the label area; layer 2 squares unit c strongly
    K = 14
    W1 = np.zeros((10, K)); W1[np.arange(10), np.arange(10)] = 1.0
    W2 = np.eye(10) * 1.0
    for c in (0, 3, 9):
        W2c = W2.copy(); W2c[c, c] = 5.0
        x = np.random.default_rng(c).random((4, K))
        pred, G = fo.predict([fo.LayerState(W1, np.zeros(10)), fo.LayerState(W2c, np.zeros(10))], x)
        assert np.all(pred == c)


def test_predict_ties_go_to_lowest_label():
    K = 12
    W = np.zeros((3, K)); W[:, 10:] = 1.0          # ignores the label area
    st = [fo.LayerState(W, np.zeros(3)), fo.LayerState(np.eye(3), np.zeros(3))]
    pred, G = fo.predict(st, np.random.default_rng(0).random((5, K)))
    assert np.all(pred == 0) and np.allclose(G, G[:, :1])


def test_layer1_overlay_identity_used_by_predict():
    """X^c W^T = X0 W^T + W[:, c] and ||x^c||^2 = ||x0||^2 + 1, where x0 is x
    with the label area zeroed: the identity the GPU predict relies on."""
    x = synth.mnist_like(30, seed=8).astype(np.float64)
    W = synth.he_uniform(8, 20, 784).astype(np.float64)
    x0 = x.copy(); x0[:, :10] = 0.0
    for c in range(10):
        xc = fo.overlay_label(x, np.full(30, c))
        assert np.allclose(xc @ W.T, x0 @ W.T + W[:, c], rtol=0, atol=1e-12)
        assert np.allclose(np.sum(xc ** 2, 1), np.sum(x0 ** 2, 1) + 1.0, rtol=1e-15)


# ------------------------------------------------------- init statistic
def test_he_uniform_goodness_expectation():
    """Unit-norm input, He-uniform W, b = 0: E[g] = N/K (Var w = 2/K, E relu(z)^2 = Var z / 2)."""
    gold = _golden("closed_forms.json")
    for (K, N) in ((784, 2000), (2000, 2000), (784, 500)):
        W = synth.he_uniform(21, N, K)
        lo, hi = W.min(), W.max()
        bound = math.sqrt(6.0 / K)
        assert -bound <= lo < -0.99 * bound and 0.99 * bound < hi <= bound
        x = synth.mnist_like(4000 if K == 784 else 1000, seed=22, features=784)
        if K != 784:
            x = np.abs(np.random.default_rng(23).standard_normal((1000, K)))
        f = fo.layer_forward_full(fo.LayerState(W, np.zeros(N)), x)
        key = f"E_g_he_uniform_{K}_{N}"
        expect = gold[key]
        assert expect == pytest.approx(N / K, rel=1e-3)
        # g is a sum over N units for one row; rows share W, so allow 3%
        assert np.mean(f["g"]) == pytest.approx(expect, rel=0.03)


# -------------------------------------------------------- bf16 emulation
def test_emulation_with_identity_rounding_is_the_plain_definition():
    rng = np.random.default_rng(9)
    B, K, N = 6, 40, 17
    x = rng.random((2 * B, K))
    W = rng.standard_normal((N, K)) * 0.3
    b = rng.standard_normal(N) * 0.1
    a = fo.layer_train_step(fo.LayerState(W, b), x, B, 1.0, fo.AdamHyper())
    e = fo.layer_train_step(fo.LayerState(W, b), x, B, 1.0, fo.AdamHyper(), rounding=lambda v: np.asarray(v, np.float64))
    for k in ("g", "dW", "db"):
        assert np.allclose(a[k], e[k], rtol=1e-12, atol=1e-15)


def test_emulation_rounds_operands_to_bf16():
    rng = np.random.default_rng(12)
    B, K, N = 4, 32, 9
    x = rng.random((2 * B, K))
    W = rng.standard_normal((N, K)) * 0.3
    st = fo.LayerState(W, np.zeros(N))
    f = fo.layer_forward_full(st, x, emulate_bf16=True)
    assert np.array_equal(f["A"], fo.bf16_round(x))
    # the product uses the rounded W and the exact norm of the unrounded input
    s = 1.0 / np.sqrt(np.sum(x ** 2, 1))
    assert np.allclose(f["Z"], s[:, None] * (fo.bf16_round(x) @ fo.bf16_round(W).T), rtol=1e-14)


# ------------------------------------------------ whole-step consistency
def test_net_step_layer_inputs_are_previous_activities():
    B = 8
    x = synth.mnist_like(B, seed=1)
    y = synth.labels(B, seed=1)
    yn = synth.negative_labels(y, seed=1)
    x2, l2 = synth.pair_batch(x, y, yn)
    dims = [784, 30, 20]
    states = [fo.LayerState(synth.he_uniform(100 + i, dims[i + 1], dims[i]), np.zeros(dims[i + 1])) for i in range(2)]
    before = [s.copy() for s in states]
    outs = fo.net_train_step(states, x2, l2, B, 2.0, fo.AdamHyper())
    # layer 2's forward used layer 1's pre-update activity
    f1 = fo.layer_forward_full(before[0], fo.overlay_label(x2, l2))
    f2 = fo.layer_forward_full(before[1], f1["H"])
    assert np.allclose(outs[0]["H"], f1["H"], rtol=1e-14, atol=1e-15)
    assert np.allclose(outs[1]["g"], f2["g"], rtol=1e-14, atol=1e-15)
    assert all(s.t == 1 for s in states)


def test_negative_labels_are_wrong_and_cover_all_offsets():
    y = synth.labels(20000, seed=2)
    yn = synth.negative_labels(y, seed=2)
    assert np.all(yn != y)
    off = (yn - y - 1) % 10
    assert set(np.unique(off)) == set(range(9))
    assert np.all(np.abs(np.bincount(y, minlength=10) / 20000 - 0.1) < 0.01)


def test_adaptive_negatives_are_the_strongest_wrong_label():
    """Brute force: for each sample the strongest of the 9 wrong labels, never
    the true one; with hand-built nets the dominated label is chosen."""
    rng = np.random.default_rng(13)
    dims = (12, 5, 4)
    Ws = [rng.standard_normal((dims[i + 1], dims[i])) for i in range(2)]
    bs = [rng.standard_normal(dims[i + 1]) * 0.2 for i in range(2)]
    x = rng.random((40, 12))
    y = rng.integers(0, 10, 40)
    states = [fo.LayerState(W, b) for W, b in zip(Ws, bs)]
    neg, G = fo.adaptive_negatives(states, x, y)
    _, bG = _brute_predict([W.tolist() for W in Ws], [b.tolist() for b in bs], x)
    for i in range(40):
        assert neg[i] != y[i]
        best = max((c for c in range(10) if c != y[i]), key=lambda c: (bG[i][c], -c))
        assert neg[i] == best
    # the true label dominates: the negative is the runner-up
    K = 14
    W1 = np.zeros((10, K)); W1[np.arange(10), np.arange(10)] = 1.0
    W2 = np.eye(10); W2[3, 3] = 5.0; W2[7, 7] = 3.0
    xx = np.random.default_rng(0).random((6, K))
    st = [fo.LayerState(W1, np.zeros(10)), fo.LayerState(W2, np.zeros(10))]
    neg, _ = fo.adaptive_negatives(st, xx, np.full(6, 3))
    assert np.all(neg == 7)



# ------------------------------------------------------- softmax head (§3)
def _brute_features(Ws, bs, x, n_classes=10):
    """Pure-Python loops: neutral label (0.1 in each label feature), normalise,
    ReLU layers; each of layers 2..L (layer 1 if L == 1) contributes its
    activity divided by its own norm."""
    out = []
    L = len(Ws)
    for row in x:
        a = [0.1] * n_classes + [float(v) for v in row[n_classes:]]
        feats = []
        for k in range(L):
            nrm = max(math.sqrt(sum(v * v for v in a)), 1e-12)
            xh = [v / nrm for v in a]
            W, b = Ws[k], bs[k]
            h = []
            for i in range(len(b)):
                z = b[i]
                for j in range(len(xh)):
                    z += W[i][j] * xh[j]
                h.append(z if z > 0 else 0.0)
            if k >= 1 or L == 1:
                hn = max(math.sqrt(sum(v * v for v in h)), 1e-12)
                feats += [v / hn for v in h]
            a = h
        out.append(feats)
    return np.array(out)


@pytest.mark.parametrize("dims", [(12, 5), (12, 6, 4), (14, 7, 5, 3)])
def test_softmax_features_match_brute_force(dims):
    rng = np.random.default_rng(len(dims))
    Ws = [rng.standard_normal((dims[i + 1], dims[i])) for i in range(len(dims) - 1)]
    bs = [rng.standard_normal(dims[i + 1]) * 0.3 for i in range(len(dims) - 1)]
    x = rng.random((9, dims[0]))
    x[3] = 0.0                                    # a zero image still carries the neutral label
    A = fo.softmax_features([fo.LayerState(W, b) for W, b in zip(Ws, bs)], x)
    ref = _brute_features([W.tolist() for W in Ws], [b.tolist() for b in bs], x)
    assert A.shape == ref.shape == (9, sum(dims[2:]) if len(dims) > 2 else dims[1])
    np.testing.assert_allclose(A, ref, rtol=1e-12, atol=1e-14)


def test_neutral_overlay_writes_point_one():
    x = np.arange(24, dtype=np.float64).reshape(2, 12)
    o = fo.overlay_neutral(x)
    assert np.all(o[:, :10] == 0.1) and np.array_equal(o[:, 10:], x[:, 10:])
    assert x[0, 0] == 0.0                          # the input is not modified


def test_cross_entropy_closed_forms():
    y = np.array([0, 3, 9, 9])
    z0 = np.zeros((4, 10))
    assert fo.cross_entropy(z0, y) == pytest.approx(math.log(10.0), rel=0, abs=1e-15)
    dz = fo.dce_dz(z0, y)
    exp = np.full((4, 10), 0.1 / 4)
    exp[np.arange(4), y] -= 1.0 / 4
    np.testing.assert_allclose(dz, exp, rtol=0, atol=1e-17)
    # a logit margin m on the right class: -log(e^m / (e^m + 9))
    z = np.zeros((4, 10))
    z[np.arange(4), y] = 3.0
    assert fo.cross_entropy(z, y) == pytest.approx(math.log(1.0 + 9.0 * math.exp(-3.0)), rel=1e-14)
    # shift invariance, probabilities sum to one, gradient rows sum to zero
    rng = np.random.default_rng(3)
    z = rng.standard_normal((6, 10)) * 4
    yy = rng.integers(0, 10, 6)
    assert fo.cross_entropy(z + 7.5, yy) == pytest.approx(fo.cross_entropy(z, yy), rel=1e-13)
    np.testing.assert_allclose(fo.softmax(z).sum(axis=1), 1.0, rtol=1e-15)
    np.testing.assert_allclose(fo.dce_dz(z, yy).sum(axis=1), 0.0, atol=1e-16)
    # huge logits stay finite (no overflow in the exponent)
    assert np.isfinite(fo.cross_entropy(z * 1e3, yy))


def test_head_gradient_matches_finite_differences():
    rng = np.random.default_rng(5)
    n, F = 7, 6
    A = rng.standard_normal((n, F))
    y = rng.integers(0, 10, n)
    V = rng.standard_normal((10, F)) * 0.5
    c = rng.standard_normal(10) * 0.1
    z = fo.head_logits(A, V, c)
    dz = fo.dce_dz(z, y)
    dV, dc = dz.T @ A, dz.sum(axis=0)
    h = 1e-6
    for (i, j) in [(0, 0), (3, 2), (9, 5), (5, 1)]:
        Vp, Vm = V.copy(), V.copy()
        Vp[i, j] += h
        Vm[i, j] -= h
        fd = (fo.cross_entropy(fo.head_logits(A, Vp, c), y) - fo.cross_entropy(fo.head_logits(A, Vm, c), y)) / (2 * h)
        assert fd == pytest.approx(dV[i, j], rel=1e-6, abs=1e-9)
    for i in (0, 4, 9):
        cp, cm = c.copy(), c.copy()
        cp[i] += h
        cm[i] -= h
        fd = (fo.cross_entropy(fo.head_logits(A, V, cp), y) - fo.cross_entropy(fo.head_logits(A, V, cm), y)) / (2 * h)
        assert fd == pytest.approx(dc[i], rel=1e-6, abs=1e-9)


def test_head_train_step_first_adam_step_and_prediction():
    rng = np.random.default_rng(8)
    n, F = 20, 9
    A = rng.standard_normal((n, F))
    y = rng.integers(0, 10, n)
    head = fo.HeadState(np.zeros((10, F)), np.zeros(10))
    hp = fo.AdamHyper(lr=1e-4)
    out = fo.head_train_step(head, A, y, hp)
    assert out["loss"] == pytest.approx(math.log(10.0), abs=1e-15)   # zero start: uniform softmax
    # first Adam step: -lr * g / (|g| + eps) elementwise
    np.testing.assert_allclose(head.V, -1e-4 * out["dV"] / (np.abs(out["dV"]) + 1e-8), rtol=1e-12, atol=1e-20)
    np.testing.assert_allclose(head.c, -1e-4 * out["dc"] / (np.abs(out["dc"]) + 1e-8), rtol=1e-12, atol=1e-20)
    assert head.t == 1
    # prediction = first maximum of the logits (brute force)
    V = rng.standard_normal((10, F))
    c = rng.standard_normal(10)
    hs = fo.HeadState(V, c)
    pred, z = fo.head_predict(hs, A)
    for i in range(n):
        zi = [float(c[k] + sum(V[k][j] * A[i][j] for j in range(F))) for k in range(10)]
        best = 0
        for k in range(1, 10):
            if zi[k] > zi[best]:
                best = k
        assert pred[i] == best
    # a selector head predicts the class whose feature is largest
    Fs = 10
    A2 = rng.random((5, Fs))
    hsel = fo.HeadState(np.eye(10), np.zeros(10))
    assert np.array_equal(fo.head_predict(hsel, A2)[0], np.argmax(A2, axis=1))


# ------------------------------------------------- chapter schedule (§4)
def test_lr_cooldown_closed_forms():
    assert fo.lr_at(0.01, 0, 100, 0.5) == 0.01
    assert fo.lr_at(0.01, 49, 100, 0.5) == 0.01
    assert fo.lr_at(0.01, 50, 100, 0.5) == pytest.approx(0.01)
    assert fo.lr_at(0.01, 75, 100, 0.5) == pytest.approx(0.005)
    assert fo.lr_at(0.01, 99, 100, 0.5) == pytest.approx(0.0002)
    assert fo.lr_at(0.01, 99, 100, 1.0) == 0.01
    assert fo.lr_at(0.03, 3, 4, 0.0) == pytest.approx(0.0075)


def test_pair_batches_cover_the_set_once():
    bl = fo.pair_batches(10, 4)
    assert bl == [(0, 4), (8, 4), (16, 2)]
    assert sum(2 * b for _, b in bl) == 20


def _schedule_inputs(P, seed):
    x = synth.mnist_like(P, seed=seed, features=24)
    y = synth.labels(P, seed=seed)
    xs, ls = [], []
    for r0, b in fo.pair_batches(P, 4):
        s0 = r0 // 2
        x2, l2 = synth.pair_batch(x[s0:s0 + b], y[s0:s0 + b], synth.negative_labels(y[s0:s0 + b], seed=seed, start=s0))
        xs.append(x2)
        ls.append(l2)
    return np.concatenate(xs), np.concatenate(ls), y


def _fresh_states(dims, seed):
    rng = np.random.default_rng(seed)
    return [fo.LayerState(rng.standard_normal((dims[i + 1], dims[i])) * 0.4, rng.standard_normal(dims[i + 1]) * 0.05)
            for i in range(len(dims) - 1)]


def test_chapter_schedule_matches_a_wavefront_replay():
    """The schedule's dependency order (layer i, chapter c after layer i-1,
    chapter c and layer i, chapter c-1), replayed along the diagonals
    t = i + c with every layer's published output kept per chapter, gives
    the same weights and losses as the chapter-major definition."""
    dims = (24, 6, 5, 4)
    P, B, C, S, theta = 10, 4, 2, 3, 0.5
    x2, l2, y = _schedule_inputs(P, seed=3)
    rng = np.random.default_rng(4)
    labs = np.stack([np.concatenate([y, (y + 1 + rng.integers(0, 9, P)) % 10]).astype(np.int32) for _ in range(S)])
    # the batch-major layout: rebuild per chapter from the per-chapter negatives
    def chapter_labels(c):
        out = np.empty(2 * P, np.int32)
        for r0, b in fo.pair_batches(P, B):
            s0 = r0 // 2
            out[r0:r0 + b] = labs[c, s0:s0 + b]
            out[r0 + b:r0 + 2 * b] = labs[c, P + s0:P + s0 + b]
        return out
    lab_pc = np.stack([chapter_labels(c) for c in range(S)])
    hp = fo.AdamHyper(lr=0.02)
    ref_states = _fresh_states(dims, 5)
    losses = fo.chapter_schedule(ref_states, x2, lab_pc, B, C, theta, hp, cooldown_start=0.5)
    # wavefront replay, written independently
    st = _fresh_states(dims, 5)
    L = len(st)
    published = {}
    wl = np.zeros_like(losses)
    E = C * S
    for t in range(L + S - 1):
        for i in range(L):
            c = t - i
            if not (0 <= c < S):
                continue
            inp = fo.overlay_label(x2, lab_pc[c]) if i == 0 else published[(i - 1, c)]
            k = 0
            for m in range(C):
                lr = hp.lr if c * C + m < 0.5 * E else hp.lr * (E - (c * C + m)) / (0.5 * E)
                for r0, b in fo.pair_batches(P, B):
                    o = fo.layer_train_step(st[i], inp[r0:r0 + 2 * b], b, theta, fo.AdamHyper(lr=lr))
                    wl[c, i, k] = o["loss"]
                    k += 1
            published[(i, c)] = fo.layer_forward_full(st[i], inp)["H"]
    np.testing.assert_allclose(wl, losses, rtol=0, atol=0)
    for a, b in zip(st, ref_states):
        np.testing.assert_array_equal(a.W, b.W)
        np.testing.assert_array_equal(a.b, b.b)
        assert a.t == b.t == S * C * len(fo.pair_batches(P, B))


def test_chapter_schedule_without_updates_is_a_fixed_forward():
    """lr = 0: no weight moves, so every step's loss is the loss of the fixed
    net on its batch -- computed here from plain forwards."""
    dims = (24, 6, 5)
    P, B, theta = 8, 4, 0.3
    x2, l2, _ = _schedule_inputs(P, seed=6)
    st = _fresh_states(dims, 7)
    W0 = [s.W.copy() for s in st]
    losses = fo.chapter_schedule(st, x2, np.stack([l2, l2]), B, 1, theta, fo.AdamHyper(lr=0.0))
    assert all(np.array_equal(s.W, w) for s, w in zip(st, W0))
    a = fo.overlay_label(x2, l2)
    for i, s in enumerate(st):
        for j, (r0, b) in enumerate(fo.pair_batches(P, B)):
            g = fo.goodness(fo.layer_forward(fo.normalise(a[r0:r0 + 2 * b]), s.W, s.b)[1])
            exp = fo.ff_loss(g, theta, b)
            assert losses[0, i, j] == pytest.approx(exp, rel=1e-12)
            assert losses[1, i, j] == pytest.approx(exp, rel=1e-12)
        a = fo.layer_forward(fo.normalise(a), s.W, s.b)[1]


# --------------------------------- Performance-Optimized PFF layer (§4)
def _po_loss(W, b, V, c, x_in, y):
    xh = fo.normalise(x_in)
    H = np.maximum(xh @ W.T + b, 0.0)
    return fo.cross_entropy(H @ V.T + c, y)


def test_po_layer_gradients_match_finite_differences():
    rng = np.random.default_rng(21)
    n, K, N = 9, 14, 7
    x = rng.random((n, K))
    y = rng.integers(0, 10, n)
    W = rng.standard_normal((N, K))
    b = rng.standard_normal(N) * 0.2
    V = rng.standard_normal((10, N))
    c = rng.standard_normal(10) * 0.1
    st, hd = fo.LayerState(W, b), fo.HeadState(V, c)
    out = fo.po_layer_train_step(st, hd, x, y, fo.AdamHyper(lr=0.0), fo.AdamHyper(lr=0.0))
    assert out["loss"] == pytest.approx(_po_loss(W, b, V, c, x, y), rel=1e-13)
    h = 1e-6
    for (i, j) in [(0, 0), (3, 5), (6, 13), (2, 7)]:
        Wp, Wm = W.copy(), W.copy()
        Wp[i, j] += h
        Wm[i, j] -= h
        fd = (_po_loss(Wp, b, V, c, x, y) - _po_loss(Wm, b, V, c, x, y)) / (2 * h)
        assert fd == pytest.approx(out["dW"][i, j], rel=1e-5, abs=1e-9)
    for i in (0, 3, 6):
        bp, bm = b.copy(), b.copy()
        bp[i] += h
        bm[i] -= h
        fd = (_po_loss(W, bp, V, c, x, y) - _po_loss(W, bm, V, c, x, y)) / (2 * h)
        assert fd == pytest.approx(out["db"][i], rel=1e-5, abs=1e-9)
    for (i, j) in [(0, 0), (9, 6), (4, 2)]:
        Vp, Vm = V.copy(), V.copy()
        Vp[i, j] += h
        Vm[i, j] -= h
        fd = (_po_loss(W, b, Vp, c, x, y) - _po_loss(W, b, Vm, c, x, y)) / (2 * h)
        assert fd == pytest.approx(out["dV"][i, j], rel=1e-5, abs=1e-9)
    np.testing.assert_allclose(out["dc"], fo.dce_dz(out["z"], y).sum(axis=0), rtol=1e-14)


def test_po_layer_special_cases():
    rng = np.random.default_rng(22)
    n, K, N = 6, 12, 5
    x = rng.random((n, K))
    y = rng.integers(0, 10, n)
    W = rng.standard_normal((N, K))
    # a zero block: nothing reaches the layer, its Adam step is zero, the loss is log 10
    st, hd = fo.LayerState(W, np.zeros(N)), fo.HeadState(np.zeros((10, N)), np.zeros(10))
    out = fo.po_layer_train_step(st, hd, x, y, fo.AdamHyper(), fo.AdamHyper(lr=1e-4))
    assert out["loss"] == pytest.approx(math.log(10.0), abs=1e-15)
    assert not out["dW"].any() and not out["db"].any()
    np.testing.assert_array_equal(st.W, W)
    # identity rounding reproduces the plain definition
    V = rng.standard_normal((10, N))
    a = fo.po_layer_train_step(fo.LayerState(W, np.zeros(N)), fo.HeadState(V, np.zeros(10)), x, y,
                               fo.AdamHyper(), fo.AdamHyper())
    b = fo.po_layer_train_step(fo.LayerState(W, np.zeros(N)), fo.HeadState(V, np.zeros(10)), x, y,
                               fo.AdamHyper(), fo.AdamHyper(), rounding=lambda v: np.asarray(v, np.float64))
    np.testing.assert_allclose(b["dW"], a["dW"], rtol=1e-12, atol=1e-15)
    # a dead unit (all pre-activations negative) gets no gradient
    Wd = W.copy()
    Wd[2] = -np.abs(Wd[2]) - 1.0
    o = fo.po_layer_train_step(fo.LayerState(Wd, np.zeros(N)), fo.HeadState(V, np.zeros(10)), x, y,
                               fo.AdamHyper(), fo.AdamHyper())
    assert not o["dW"][2].any() and o["db"][2] == 0.0


def _brute_po_predict(Ws, bs, V, c, x):
    """The last block's argmax with explicit loops: neutral label (0.1 in the
    10 label features), each layer's input scaled to unit length (1e-12
    floor), ReLU layers, logits V h + c on the last raw activity, lowest
    class on ties."""
    preds = []
    for row in x:
        a = [0.1] * 10 + [float(v) for v in row[10:]]
        for W, b in zip(Ws, bs):
            nrm = math.sqrt(sum(v * v for v in a))
            s = 1.0 / max(nrm, 1e-12)
            h = []
            for j in range(len(W)):
                z = b[j] + sum(W[j][k] * a[k] * s for k in range(len(a)))
                h.append(z if z > 0 else 0.0)
            a = h
        z = [c[k] + sum(V[k][j] * a[j] for j in range(len(a))) for k in range(10)]
        best = 0
        for k in range(1, 10):
            if z[k] > z[best]:
                best = k
        preds.append(best)
    return np.array(preds)


@pytest.mark.parametrize("dims", [(14, 6, 5), (14, 7)])
def test_po_predict_matches_brute_force(dims):
    rng = np.random.default_rng(31)
    Ws = [rng.standard_normal((dims[i + 1], dims[i])) for i in range(len(dims) - 1)]
    bs = [rng.standard_normal(dims[i + 1]) * 0.2 for i in range(len(dims) - 1)]
    V = rng.standard_normal((10, dims[-1]))
    c = rng.standard_normal(10) * 0.1
    x = rng.random((40, dims[0]))
    states = [fo.LayerState(W, b) for W, b in zip(Ws, bs)]
    heads = [fo.HeadState(rng.standard_normal((10, d)), np.zeros(10)) for d in dims[1:-1]] + [fo.HeadState(V, c)]
    pred, z = fo.po_predict(states, heads, x)
    bp = _brute_po_predict([W.tolist() for W in Ws], [b.tolist() for b in bs], V.tolist(), c.tolist(), x)
    assert np.array_equal(pred, bp)
    # only the last layer's block decides: the earlier blocks are ignored
    heads2 = [fo.HeadState(np.zeros((10, d)), np.ones(10)) for d in dims[1:-1]] + [fo.HeadState(V, c)]
    assert np.array_equal(fo.po_predict(states, heads2, x)[0], pred)


def test_po_predict_hand_built_block_selects_the_class():
    # one layer copying features 10..19 through the ReLU; the block maps unit j to class j
    K = 24
    W = np.zeros((10, K)); W[np.arange(10), 10 + np.arange(10)] = 1.0
    V = np.eye(10)
    x = np.zeros((10, K))
    for k in range(10):
        x[k, 10 + k] = 1.0          # the only nonzero image feature of sample k
    pred, z = fo.po_predict([fo.LayerState(W, np.zeros(10))], [fo.HeadState(V, np.zeros(10))], x)
    assert np.array_equal(pred, np.arange(10))
    # the neutral label area (10 x 0.1) only enters through the input norm: z_k = 1 / sqrt(1.1)
    np.testing.assert_allclose(z[np.arange(10), np.arange(10)], 1.0 / math.sqrt(1.1), rtol=1e-14)
