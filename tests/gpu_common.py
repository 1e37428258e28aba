"""Shared helpers of the GPU parity tests (inputs from synth, references from
the oracle; nothing here computes any part of the method)."""

import numpy as np
import pytest

from oracle import ff_oracle as fo
from paper_2404_08573_gb300 import synth


def torch_cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch


def lib_ready():
    from paper_2404_08573_gb300 import build, ff
    build.build()
    ff.lib()
    return ff


def pair_inputs(B, seed, features=784, kind="mnist"):
    x = synth.mnist_like(B, seed=seed, features=features) if kind == "mnist" else synth.cifar_like(
        B, seed=seed, features=features)
    y = synth.labels(B, seed=seed)
    yn = synth.negative_labels(y, seed=seed)
    return synth.pair_batch(x, y, yn)


def rel_norm(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    d = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (d if d > 0 else 1.0))


def assert_close(got, ref, rtol, atol, what, max_bad_frac=0.0):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    bad = np.abs(got - ref) > atol + rtol * np.abs(ref)
    frac = bad.mean() if bad.size else 0.0
    if frac > max_bad_frac:
        idx = np.argwhere(bad)[:5]
        samples = [(tuple(i), got[tuple(i)], ref[tuple(i)]) for i in idx]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside rtol={rtol} atol={atol}; e.g. {samples}")


U32 = 2.0 ** -24


def grad_uncertainty(ref, W, b, x_in, B, emulate_bf16, tensor_cores):
    """First-order bound on |dW_gpu - dW_exact| (and for db) for one FF step
    computed with fp32 arithmetic, element by element.

    Forward: z = s * (x . w) + b has absolute error dh <= gamma_K * s|x||w|
    + u|b| (ReLU is 1-Lipschitz, so h inherits it, whatever the size of h).
    Goodness g = sum h^2 then errs by sum 2h dh + gamma_N g, and dL/dg =
    +-sigma/B by at most dg/(4B).  Each term 2c h s x of the weight gradient
    therefore errs by 2|c| dh + 2 dc |h| plus the gamma_R of the R-term sum;
    in bf16-operand mode the stored h and s*dZ may also round one bf16 ulp
    (2^-7 relative) away from the emulation where fp32 and fp64 straddle a
    rounding boundary.  Tensor-core sums get twice the fp32 gamma."""
    u = U32 * (2.0 if tensor_cores else 1.0)
    H, c, s = ref["H"], ref["c"], ref["s"]
    M, N = H.shape
    K = W.shape[1]
    from oracle import ff_oracle as fo
    Wop = fo.bf16_round(W) if emulate_bf16 else np.asarray(W, np.float64)
    Aop = fo.bf16_round(x_in) if emulate_bf16 else np.asarray(x_in, np.float64)
    xh = s[:, None] * np.abs(Aop)
    dh = (K + 8) * u * (xh @ np.abs(Wop).T) + 2 * U32 * np.abs(np.asarray(b, np.float64))
    gerr = np.sum(2 * H * dh, axis=1) + (N + 8) * U32 * ref["g"]
    dc = 0.25 * gerr / B + 8 * U32 * np.abs(c)
    op = 2.0 ** -6 if emulate_bf16 else 0.0
    T = 2 * np.abs(c)[:, None] * (dh + (op + (M + 16) * u) * H) + 2 * dc[:, None] * (H + dh)
    return T.T @ xh, T.sum(axis=0)


def assert_adam_state(got_w, got_m, got_v, pre_w, pre_m, pre_v, t, g_ref, dg, hp, what, rtol=1e-4,
                      w_floor=1e-2, max_band_frac=0.05, max_flip_frac=0.0):
    """Parameters and moments after one Adam step (§5.1) against the oracle.

    Adam maps the gradient through m/(sqrt(v)+eps); at the first steps this is
    about lr*sign(g), so where |g| is comparable to eps or to its own rounding
    error the update is steep in g.  Each element may therefore differ from
    the reference by rtol relative plus the spread of the oracle's own update
    over gradients g_ref +- dg (dg = the fp32 rounding bound of that gradient
    element).  Elements that need the spread must be a small fraction; in
    bf16-operand mode a few elements may also differ by a whole sign flip
    (operand roundings at ties that the emulation does not reproduce)."""
    from oracle import ff_oracle as fo
    ref = fo.adam_update(pre_w, g_ref, pre_m, pre_v, t, hp)
    hi = fo.adam_update(pre_w, g_ref + dg, pre_m, pre_v, t, hp)
    lo = fo.adam_update(pre_w, g_ref - dg, pre_m, pre_v, t, hp)
    for i, (name, got) in enumerate((("param", got_w), ("m", got_m), ("v", got_v))):
        r = ref[i]
        band = np.maximum(np.abs(hi[i] - r), np.abs(lo[i] - r))
        floor = w_floor if i == 0 else 1e-3 * float(np.max(np.abs(r)) or 1.0)
        tol = rtol * np.maximum(np.abs(r), floor)
        err = np.abs(np.asarray(got, np.float64) - r)
        plain = err <= tol
        ok = err <= tol + band
        nbad = int((~ok).sum())
        if nbad > max_flip_frac * err.size:
            j = tuple(np.argwhere(~ok)[0])
            raise AssertionError(f"{what} {name}: {nbad} of {err.size} off (e.g. {j}: {np.asarray(got)[j]} vs "
                                 f"{r[j]}, g={g_ref[j]}, dg={dg[j]})")
        assert (~plain).mean() <= max_band_frac, f"{what} {name}: {(~plain).sum()} need the rounding band"


def oracle_state(st):
    return fo.LayerState(st["W"], st["b"], st["mW"], st["vW"], st["mb"], st["vb"], st["t"])
