"""Forward-Forward CPU oracle.  TEST INFRASTRUCTURE ONLY.

A plain, slow, obviously-correct fp64 NumPy statement of what the FF train
step and FF goodness prediction compute, written from "Going Forward-Forward
in Distributed Deep Learning" (arXiv 2404.08573).  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py`` (its CPU-baseline and reference
legs) may import this module.  The CUDA library never calls it, and it shares
no code, header, table or constant with the CUDA path.

What each function follows:

* ``overlay_label``   -- §3 "Negative Data": a 1-of-C label written into a
  10-feature area; correct label for positive rows, wrong label for negative.
* ``normalise``       -- x / max(||x||_2, 1e-12) per row, applied to each
  layer's input (the normalisation of Hinton's FF, cited in §2/§3; the paper
  itself does not restate it).
* ``layer_forward``   -- §3 "Goodness Function": rectified linear neurons,
  y = ReLU(x_hat W^T + b); §4 notation L_i(x).
* ``goodness``        -- Eq. 1: sum_j y_j^2.
* ``p_real``          -- Eq. 1: sigma(sum_j y_j^2 - theta).
* ``ff_loss``/``dloss_dg`` -- the negative log-likelihood of Eq. 1: -log p for
  positive rows, -log(1-p) for negative rows, i.e. softplus(theta - g_pos) +
  softplus(g_neg - theta), averaged over the B pairs.
* ``layer_train_step`` -- one local (layer-wise, §2/§3) update: the gradient of
  the layer's own loss w.r.t. its own W, b only (no gradient crosses layers),
  then Adam (§5.1).
* ``net_train_step``  -- §4: x is the concatenation of the positive and the
  negative data; layer i trains on L_{i-1}(x) computed with the weights that
  layer i-1 had before this step's update.
* ``predict``         -- §3 "Prediction", Goodness method: run the input with
  each of the 10 labels, accumulate goodness over all but the first hidden
  layer, pick the label with the largest total.
* ``adaptive_negatives`` -- AdaptiveNEG of §5: the negative label of a sample
  is the incorrect label the network currently predicts most strongly, i.e.
  the goodness-prediction argmax over the 9 wrong labels.
* ``lr_at``/``chapter_schedule`` -- §3 "Sequential Training" and §4
  (Algorithm 1, Single-Layer PFF; Algorithm 2 runs the same dependency
  order on other nodes): the E epochs are cut into S chapters of C = E/S
  epochs; in chapter c layer i trains C epochs on the output of layer i-1
  as it stands after that layer's chapter c, then publishes its own output.
* ``po_layer_train_step``/``po_predict`` -- Performance-Optimized PFF (§4,
  "PFF with a new goodness function"): each layer gets its own softmax block
  and the two are trained together by backpropagation through these two
  layers only, on the block's cross-entropy; no negative data.
* ``overlay_neutral``/``softmax_features``/``head_*`` -- §3 "Prediction",
  Softmax method: the input carries a neutral label (0.1 in each of the 10
  label features), the activities of all but the first hidden layer feed a
  linear softmax layer trained by backpropagation through that layer only
  (cross-entropy, Adam with the head's own learning rate, §5.1); the
  prediction is the class with the largest logit.

Readings of points the paper leaves open (the paper states none of them):

1. Loss = mean over the B pairs of softplus(theta-g_pos) + softplus(g_neg-theta).
2. Normalisation x/max(||x||,1e-12) of every layer input, after the overlay.
3. Overlay *replaces* features 0..9 with a one-hot of value 1.0.
4. Adam with beta1=0.9, beta2=0.999, eps=1e-8, bias-corrected, eps outside
   the square root, no weight decay; the step counter t starts at 1.
5. ReLU derivative at 0 is 0.
6. Prediction sums goodness of layers 2..L (layer 1 when L == 1); ties go to
   the lowest label.
7. The layer input fed to the next layer is the ReLU activity computed with
   the pre-update weights of the same step.
8. Softmax head: its input is the concatenation, over layers 2..L (layer 1
   when L == 1), of each layer's activity normalised like a layer input,
   h / max(||h||, 1e-12); cross-entropy averaged over the rows; weights and
   biases start at zero; ties of the logits go to the lowest class.
9. Learning-rate cooldown (named, not given, in §5.1): constant until epoch
   f*E, then falling linearly to 0 at epoch E (f = 0.5: the "after the 50th
   of 100 epochs" of §5.1); f >= 1 keeps it constant.  The epoch of a step is
   the layer's own epoch count.  Batches run in dataset order every epoch;
   the negative labels of a chapter are an input (Random/Fixed/AdaptiveNEG
   choose them).
10. Performance-Optimized layer: the input of layer 1 carries the neutral
   label; the layer's block reads its raw activity h (z = h V^T + c); the
   gradient reaching the layer is dz V, masked by the ReLU; the layer and its
   block each keep their own Adam state and learning rate; the input of the
   next layer is h from the pre-update weights, as in FF; prediction is the
   last layer's block's argmax.

``emulate_bf16=True`` rounds (round-to-nearest-even) the operands that the
bf16-operand mode stores in bfloat16 -- the layer's input activity, W, the
activity used in the local gradient, and the weight-gradient operand s*dZ --
and keeps every sum in fp64.  With the rounding replaced by the identity it
reduces to the plain definition (a test pins that).
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

N_CLASSES = 10
NORM_EPS = 1e-12


# ----------------------------------------------------------------- rounding
def bf16_round(a):
    """Round to the nearest bfloat16 (8 significant bits), ties to even.

    Written from the format's definition: a = m * 2**e with 0.5 <= |m| < 1;
    keep 8 significant bits of m by rounding m * 2**8 to an integer (numpy's
    ``rint`` rounds halves to even).  Finite, normal-range values only.
    """
    a = np.asarray(a, dtype=np.float64)
    m, e = np.frexp(a)
    return np.ldexp(np.rint(m * 256.0), e - 8)


def _identity(a):
    return np.asarray(a, dtype=np.float64)


# ---------------------------------------------------------------- §3 pieces
def overlay_label(x, labels, n_classes: int = N_CLASSES):
    """§3 Negative Data: write one-hot(label) into features 0..n_classes-1."""
    out = np.array(x, dtype=np.float64, copy=True)
    labels = np.asarray(labels, dtype=np.int64)
    out[:, :n_classes] = 0.0
    out[np.arange(out.shape[0]), labels] = 1.0
    return out


def row_norm(x):
    x = np.asarray(x, dtype=np.float64)
    return np.sqrt(np.sum(x * x, axis=1))


def normalise(x):
    """x_hat = x / max(||x||_2, 1e-12), row by row (a zero row stays zero)."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.maximum(row_norm(x), NORM_EPS)[:, None]


def layer_forward(x_hat, W, b):
    """§3: activities of rectified linear neurons, y = ReLU(x_hat W^T + b).

    Returns (Z, H): the pre-activation and the activity."""
    Z = np.asarray(x_hat, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T + np.asarray(b, dtype=np.float64)
    return Z, np.maximum(Z, 0.0)


def goodness(H):
    """Eq. 1: g = sum_j y_j^2 for each row."""
    H = np.asarray(H, dtype=np.float64)
    return np.sum(H * H, axis=1)


def sigmoid(t):
    t = np.asarray(t, dtype=np.float64)
    e = np.exp(-np.abs(t))
    return np.where(t >= 0, 1.0 / (1.0 + e), e / (1.0 + e))


def softplus(t):
    """log(1 + e^t), as max(t, 0) + log1p(e^-|t|)."""
    t = np.asarray(t, dtype=np.float64)
    return np.maximum(t, 0.0) + np.log1p(np.exp(-np.abs(t)))


def p_real(g, theta):
    """Eq. 1: p(real) = sigma(g - theta)."""
    return sigmoid(np.asarray(g, dtype=np.float64) - theta)


def ff_loss(g, theta, B):
    """-log p(real) on the B positive rows plus -log(1 - p(real)) on the B
    negative rows (Eq. 1), averaged over the B pairs."""
    g = np.asarray(g, dtype=np.float64)
    pos, neg = g[:B], g[B:2 * B]
    return float((np.sum(softplus(theta - pos)) + np.sum(softplus(neg - theta))) / B)


def dloss_dg(g, theta, B):
    """d ff_loss / d g_i: -sigma(theta - g)/B on positive rows,
    +sigma(g - theta)/B on negative rows."""
    g = np.asarray(g, dtype=np.float64)
    d = np.empty_like(g)
    d[:B] = -sigmoid(theta - g[:B]) / B
    d[B:2 * B] = sigmoid(g[B:2 * B] - theta) / B
    return d


# ------------------------------------------------------------------- §5.1 Adam
@dataclass
class AdamHyper:
    lr: float = 0.03
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-8


def adam_update(w, grad, m, v, t, hp: AdamHyper):
    """Adam (Kingma & Ba), step t >= 1, bias-corrected.  Returns (w, m, v)."""
    grad = np.asarray(grad, dtype=np.float64)
    m = hp.beta1 * np.asarray(m, dtype=np.float64) + (1.0 - hp.beta1) * grad
    v = hp.beta2 * np.asarray(v, dtype=np.float64) + (1.0 - hp.beta2) * grad * grad
    m_hat = m / (1.0 - hp.beta1 ** t)
    v_hat = v / (1.0 - hp.beta2 ** t)
    w = np.asarray(w, dtype=np.float64) - hp.lr * m_hat / (np.sqrt(v_hat) + hp.eps)
    return w, m, v


# ------------------------------------------------------------ one FF layer
@dataclass
class LayerState:
    W: np.ndarray          # [out, in]
    b: np.ndarray          # [out]
    mW: np.ndarray = None
    vW: np.ndarray = None
    mb: np.ndarray = None
    vb: np.ndarray = None
    t: int = 0

    def __post_init__(self):
        self.W = np.array(self.W, dtype=np.float64)
        self.b = np.array(self.b, dtype=np.float64)
        for name, like in (("mW", self.W), ("vW", self.W), ("mb", self.b), ("vb", self.b)):
            cur = getattr(self, name)
            setattr(self, name, np.zeros_like(like) if cur is None else np.array(cur, dtype=np.float64))

    def copy(self):
        return LayerState(self.W.copy(), self.b.copy(), self.mW.copy(), self.vW.copy(),
                          self.mb.copy(), self.vb.copy(), self.t)


def layer_forward_full(state: LayerState, x_in, emulate_bf16=False):
    """L_i(x) of §4 for one layer, on the raw (un-normalised) layer input.

    Returns dict(s, A, Z, H, g): s = 1/max(||x_in||, eps) per row, A the GEMM
    operand (x_in, rounded to bf16 when emulating), Z = s*(A W^T) + b, H, g.
    """
    rnd = bf16_round if emulate_bf16 else _identity
    x_in = np.asarray(x_in, dtype=np.float64)
    s = 1.0 / np.maximum(row_norm(x_in), NORM_EPS)
    A = rnd(x_in)
    x_hat = s[:, None] * A                       # the normalised input
    Z, H = layer_forward(x_hat, rnd(state.W), state.b)
    return dict(s=s, A=A, x_hat=x_hat, Z=Z, H=H, g=goodness(H))


def layer_train_step(state: LayerState, x_in, B: int, theta: float, hp: AdamHyper,
                     emulate_bf16: bool = False, rounding=None):
    """One local FF update of one layer (§3, Eq. 1; Adam of §5.1).

    x_in: [2B, in] raw layer input (rows 0..B-1 positive, B..2B-1 negative;
    for layer 1 already label-overlaid).  Mutates ``state``; returns a dict
    with the forward quantities (H, g, s), the loss and the gradients.
    ``rounding`` overrides the bf16 rounding function (tests use the identity).
    """
    rnd = rounding if rounding is not None else (bf16_round if emulate_bf16 else _identity)
    emul = emulate_bf16 or rounding is not None
    x_in = np.asarray(x_in, dtype=np.float64)
    assert x_in.shape[0] == 2 * B
    s = 1.0 / np.maximum(row_norm(x_in), NORM_EPS)
    A = rnd(x_in)
    x_hat = s[:, None] * A
    Z, H = layer_forward(x_hat, rnd(state.W), state.b)
    g = goodness(H)
    loss = ff_loss(g, theta, B)
    c = dloss_dg(g, theta, B)
    # local gradient dL/dz = dL/dg * 2h * [z > 0]   (no gradient leaves the layer)
    Hg = rnd(H) if emul else H
    dZ = 2.0 * c[:, None] * Hg * (Z > 0)
    if emul:
        G = rnd(s[:, None] * dZ)               # weight-gradient operand, as stored
        gL, gR = G, A
    else:
        gL, gR = dZ, x_hat                     # dL/dW = dZ^T x_hat
    dW = gL.T @ gR
    db = np.sum(dZ, axis=0)
    state.t += 1
    state.W, state.mW, state.vW = adam_update(state.W, dW, state.mW, state.vW, state.t, hp)
    state.b, state.mb, state.vb = adam_update(state.b, db, state.mb, state.vb, state.t, hp)
    # gL, gR: the two operands of the weight-gradient product dW = gL^T gR
    return dict(H=H, g=g, s=s, loss=loss, dW=dW, db=db, c=c, dZ=dZ, gL=gL, gR=gR)


def net_train_step(states, x_raw, labels, B: int, theta: float, hp: AdamHyper,
                   emulate_bf16: bool = False):
    """§4: one batch through every layer; layer k+1 trains on layer k's
    activity from the same step (pre-update weights).  Returns per-layer dicts."""
    x_in = overlay_label(x_raw, labels)
    outs = []
    for st in states:
        o = layer_train_step(st, x_in, B, theta, hp, emulate_bf16=emulate_bf16)
        outs.append(o)
        x_in = o["H"]
    return outs


# ------------------------------------------------------------------ predict
def predict(states, x_raw, emulate_bf16: bool = False, n_classes: int = N_CLASSES):
    """§3 Prediction (Goodness): for every label c, overlay c, run all layers,
    sum the goodness of layers 2..L (layer 1 if L == 1); argmax over c, the
    lowest label winning ties.  Returns (pred [n] int64, G [n, n_classes])."""
    x_raw = np.asarray(x_raw, dtype=np.float64)
    n = x_raw.shape[0]
    L = len(states)
    G = np.zeros((n, n_classes), dtype=np.float64)
    for c in range(n_classes):
        a = overlay_label(x_raw, np.full(n, c))
        for k, st in enumerate(states):
            f = layer_forward_full(st, a, emulate_bf16=emulate_bf16)
            if k >= 1 or L == 1:
                G[:, c] += f["g"]
            a = f["H"]
    return np.argmax(G, axis=1), G


def adaptive_negatives(states, x_raw, labels, emulate_bf16: bool = False, n_classes: int = N_CLASSES):
    """AdaptiveNEG (§5): for each sample, the wrong label with the largest
    accumulated goodness (the lowest such label on ties).  Returns
    (neg [n] int64, G [n, n_classes])."""
    labels = np.asarray(labels, dtype=np.int64)
    _, G = predict(states, x_raw, emulate_bf16=emulate_bf16, n_classes=n_classes)
    masked = G.copy()
    masked[np.arange(G.shape[0]), labels] = -np.inf
    return np.argmax(masked, axis=1), G


# --------------------------------------------------------- softmax head (§3)
NEUTRAL_LABEL = 0.1


def overlay_neutral(x, n_classes: int = N_CLASSES, value: float = NEUTRAL_LABEL):
    """§3 Softmax prediction: the unlabelled input gets the neutral label,
    ``value`` (0.1) in each of the 10 label features (written, as the overlay)."""
    out = np.array(x, dtype=np.float64, copy=True)
    out[:, :n_classes] = value
    return out


def softmax_features(states, x_raw, emulate_bf16: bool = False):
    """§3 Softmax prediction: run the neutral-labelled input through every
    layer and concatenate the normalised activities of layers 2..L (layer 1
    when L == 1).  In bf16 mode the stored activity is rounded and its scale
    comes from the unrounded goodness, as the layers hand it on."""
    a = overlay_neutral(x_raw)
    L = len(states)
    feats = []
    for k, st in enumerate(states):
        f = layer_forward_full(st, a, emulate_bf16=emulate_bf16)
        if k >= 1 or L == 1:
            h = bf16_round(f["H"]) if emulate_bf16 else f["H"]
            scale = 1.0 / np.maximum(np.sqrt(f["g"]), NORM_EPS)
            feats.append(scale[:, None] * h)
        a = f["H"]
    return np.concatenate(feats, axis=1)


@dataclass
class HeadState:
    V: np.ndarray          # [classes, features]
    c: np.ndarray          # [classes]
    mV: np.ndarray = None
    vV: np.ndarray = None
    mc: np.ndarray = None
    vc: np.ndarray = None
    t: int = 0

    def __post_init__(self):
        self.V = np.array(self.V, dtype=np.float64)
        self.c = np.array(self.c, dtype=np.float64)
        for name, like in (("mV", self.V), ("vV", self.V), ("mc", self.c), ("vc", self.c)):
            v = getattr(self, name)
            setattr(self, name, np.zeros_like(like) if v is None else np.array(v, dtype=np.float64))


def head_logits(A, V, c):
    """z = A V^T + c."""
    return np.asarray(A, dtype=np.float64) @ np.asarray(V, dtype=np.float64).T + np.asarray(c, dtype=np.float64)


def softmax(z):
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - np.max(z, axis=1, keepdims=True))
    return e / np.sum(e, axis=1, keepdims=True)


def cross_entropy(z, labels):
    """Mean over rows of -log softmax(z)[label] = logsumexp(z) - z[label]."""
    z = np.asarray(z, dtype=np.float64)
    labels = np.asarray(labels, dtype=np.int64)
    m = np.max(z, axis=1)
    lse = m + np.log(np.sum(np.exp(z - m[:, None]), axis=1))
    return float(np.mean(lse - z[np.arange(z.shape[0]), labels]))


def dce_dz(z, labels):
    """d(cross_entropy)/dz = (softmax(z) - onehot(label)) / n."""
    p = softmax(z)
    n = p.shape[0]
    p[np.arange(n), np.asarray(labels, dtype=np.int64)] -= 1.0
    return p / n


def head_train_step(head: HeadState, A, labels, hp: AdamHyper):
    """One backpropagation step of the softmax layer alone (the gradient does
    not reach the FF layers); Adam on V and c.  Mutates ``head``."""
    A = np.asarray(A, dtype=np.float64)
    z = head_logits(A, head.V, head.c)
    loss = cross_entropy(z, labels)
    dz = dce_dz(z, labels)
    dV = dz.T @ A
    dc = np.sum(dz, axis=0)
    head.t += 1
    head.V, head.mV, head.vV = adam_update(head.V, dV, head.mV, head.vV, head.t, hp)
    head.c, head.mc, head.vc = adam_update(head.c, dc, head.mc, head.vc, head.t, hp)
    return dict(z=z, loss=loss, dz=dz, dV=dV, dc=dc)


def head_predict(head: HeadState, A):
    """The class with the largest logit (the lowest class on ties).
    Returns (pred [n] int64, z [n, classes])."""
    z = head_logits(A, head.V, head.c)
    return np.argmax(z, axis=1), z


# ------------------------------------------------------ chapter schedule (§4)
def lr_at(lr0: float, epoch: int, total_epochs: int, cooldown_start: float) -> float:
    """The learning rate of (0-based) epoch ``epoch`` of ``total_epochs``:
    lr0 until epoch cooldown_start*E, then linearly down to 0 at epoch E."""
    if cooldown_start >= 1.0:
        return lr0
    e0 = cooldown_start * total_epochs
    if epoch < e0:
        return lr0
    return lr0 * (total_epochs - epoch) / (total_epochs - e0)


def pair_batches(n_pairs: int, B: int):
    """(first row, pairs) of each batch of the batch-major pair layout:
    batch j occupies rows 2*j*B .. 2*j*B + 2*b (b positive rows, then the
    same b images with wrong labels)."""
    out, done = [], 0
    while done < n_pairs:
        b = min(B, n_pairs - done)
        out.append((2 * done, b))
        done += b
    return out


def chapter_schedule(states, x_pairs, labels_per_chapter, B: int, C: int, theta: float, hp: AdamHyper,
                     emulate_bf16: bool = False, cooldown_start: float = 1.0):
    """Chapters c = 1..S of §4 (Single-Layer PFF, Algorithm 1): layer i trains
    C epochs over the batches of the output of layer i-1 after its chapter c
    (layer 1: the raw pairs overlaid with chapter c's labels), then its own
    output with the updated weights is published for layer i+1.  Mutates the
    states; returns losses [S, L, C * batches] (each train step's loss)."""
    x_pairs = np.asarray(x_pairs, dtype=np.float64)
    labels_per_chapter = np.asarray(labels_per_chapter)
    S = labels_per_chapter.shape[0]
    L = len(states)
    bl = pair_batches(x_pairs.shape[0] // 2, B)
    E = C * S
    losses = np.zeros((S, L, C * len(bl)))
    for c in range(S):
        a = overlay_label(x_pairs, labels_per_chapter[c])
        for i, st in enumerate(states):
            for m in range(C):
                e = c * C + m
                hpe = AdamHyper(lr_at(hp.lr, e, E, cooldown_start), hp.beta1, hp.beta2, hp.eps)
                for j, (r0, b) in enumerate(bl):
                    o = layer_train_step(st, a[r0:r0 + 2 * b], b, theta, hpe, emulate_bf16=emulate_bf16)
                    losses[c, i, m * len(bl) + j] = o["loss"]
            a = layer_forward_full(st, a, emulate_bf16=emulate_bf16)["H"]
    return losses


# ------------------------------------- Performance-Optimized PFF layer (§4)
def po_layer_train_step(state: LayerState, head: HeadState, x_in, labels, hp_layer: AdamHyper, hp_head: AdamHyper,
                        emulate_bf16: bool = False, rounding=None):
    """One step of a Performance-Optimized PFF layer and its softmax block
    (§4): z = h V^T + c on the layer's activity h = ReLU(x_hat W^T + b),
    cross-entropy averaged over the n rows, backpropagation through the block
    and the layer only, then Adam on W, b and on V, c.  x_in [n, in] is the
    raw layer input (layer 1: the neutral-labelled image).  Mutates both
    states; returns the forward quantities, the loss and the gradients."""
    rnd = rounding if rounding is not None else (bf16_round if emulate_bf16 else _identity)
    emul = emulate_bf16 or rounding is not None
    x_in = np.asarray(x_in, dtype=np.float64)
    s = 1.0 / np.maximum(row_norm(x_in), NORM_EPS)
    A = rnd(x_in)
    x_hat = s[:, None] * A
    Z, H = layer_forward(x_hat, rnd(state.W), state.b)
    Hs = rnd(H) if emul else H                   # the activity as stored, read by the block
    z = head_logits(Hs, head.V, head.c)
    loss = cross_entropy(z, labels)
    dz = dce_dz(z, labels)
    dV = dz.T @ Hs
    dc = np.sum(dz, axis=0)
    dZ = (dz @ head.V) * (Z > 0)                 # through the block (pre-update V) and the ReLU
    if emul:
        G = rnd(s[:, None] * dZ)
        dW = G.T @ A
    else:
        dW = dZ.T @ x_hat
    db = np.sum(dZ, axis=0)
    state.t += 1
    state.W, state.mW, state.vW = adam_update(state.W, dW, state.mW, state.vW, state.t, hp_layer)
    state.b, state.mb, state.vb = adam_update(state.b, db, state.mb, state.vb, state.t, hp_layer)
    head.t += 1
    head.V, head.mV, head.vV = adam_update(head.V, dV, head.mV, head.vV, head.t, hp_head)
    head.c, head.mc, head.vc = adam_update(head.c, dc, head.mc, head.vc, head.t, hp_head)
    return dict(H=H, g=goodness(H), s=s, z=z, loss=loss, dz=dz, dW=dW, db=db, dV=dV, dc=dc, dZ=dZ)


def po_predict(states, heads, x_raw, emulate_bf16: bool = False):
    """The last layer's block's prediction on the neutral-labelled input.
    Returns (pred [n] int64, z [n, classes])."""
    a = overlay_neutral(x_raw)
    H = None
    for st in states:
        f = layer_forward_full(st, a, emulate_bf16=emulate_bf16)
        H = f["H"]
        a = H
    Hs = bf16_round(H) if emulate_bf16 else H
    return head_predict(heads[-1], Hs)

