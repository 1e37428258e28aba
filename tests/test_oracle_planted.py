"""Mistakes planted in the CPU oracle are caught by its pins.

Each case swaps one oracle function (or one line of it, in a copy) for a
plausible wrong version -- a dropped term, a wrong sign or index, a
transposed operand, a missing floor or bias correction -- and runs the pins
of tests/test_oracle_pins.py that cover it: every such run must fail.  The
planted versions live only here and only for the duration of one test
(monkeypatch restores the module), so the oracle itself is untouched.
"""

import numpy as np
import pytest

from oracle import ff_oracle as fo
from tests import test_oracle_pins as pins


def _caught(pin, *args, errors=(AssertionError,)):
    with pytest.raises(errors):
        pin(*args)


# ------------------------------------------------------------ §3 pieces
def test_overlay_with_an_off_by_one_label_is_caught(monkeypatch):
    def bad(x, labels, n_classes=fo.N_CLASSES):
        out = np.array(x, dtype=np.float64, copy=True)
        out[:, :n_classes] = 0.0
        out[np.arange(out.shape[0]), (np.asarray(labels) + 1) % n_classes] = 1.0
        return out
    monkeypatch.setattr(fo, "overlay_label", bad)
    _caught(pins.test_overlay_is_exact_one_hot_and_leaves_rest_untouched)


def test_overlay_that_adds_instead_of_replacing_is_caught(monkeypatch):
    def bad(x, labels, n_classes=fo.N_CLASSES):
        out = np.array(x, dtype=np.float64, copy=True)
        out[np.arange(out.shape[0]), np.asarray(labels)] += 1.0
        return out
    monkeypatch.setattr(fo, "overlay_label", bad)
    _caught(pins.test_overlay_is_exact_one_hot_and_leaves_rest_untouched)


def test_normalise_without_the_norm_floor_is_caught(monkeypatch):
    def bad(x):
        x = np.asarray(x, dtype=np.float64)
        with np.errstate(invalid="ignore", divide="ignore"):
            return x / fo.row_norm(x)[:, None]
    monkeypatch.setattr(fo, "normalise", bad)
    _caught(pins.test_normalise_unit_norm_zero_row_and_scale_invariance)


def test_l1_row_norm_is_caught(monkeypatch):
    monkeypatch.setattr(fo, "row_norm", lambda x: np.sum(np.abs(np.asarray(x, dtype=np.float64)), axis=1))
    _caught(pins.test_goodness_of_hand_built_layers)
    _caught(pins.test_normalise_unit_norm_zero_row_and_scale_invariance)


def test_goodness_without_the_square_is_caught(monkeypatch):
    monkeypatch.setattr(fo, "goodness", lambda H: np.sum(np.asarray(H, dtype=np.float64), axis=1))
    _caught(pins.test_goodness_of_hand_built_layers)


def test_layer_without_its_bias_is_caught(monkeypatch):
    def bad(x_hat, W, b):
        Z = np.asarray(x_hat, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T
        return Z, np.maximum(Z, 0.0)
    monkeypatch.setattr(fo, "layer_forward", bad)
    _caught(pins.test_goodness_of_hand_built_layers)


def test_layer_without_its_relu_is_caught(monkeypatch):
    def bad(x_hat, W, b):
        Z = np.asarray(x_hat, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T + b
        return Z, Z
    monkeypatch.setattr(fo, "layer_forward", bad)
    _caught(pins.test_goodness_of_hand_built_layers)


# -------------------------------------------------------- loss, gradient
def test_loss_summed_over_pairs_instead_of_averaged_is_caught(monkeypatch):
    def bad(g, theta, B):
        g = np.asarray(g, dtype=np.float64)
        return float(np.sum(fo.softplus(theta - g[:B])) + np.sum(fo.softplus(g[B:2 * B] - theta)))
    monkeypatch.setattr(fo, "ff_loss", bad)
    _caught(pins.test_loss_closed_forms)


def test_loss_with_the_negative_margin_mirrored_is_caught(monkeypatch):
    def bad(g, theta, B):
        g = np.asarray(g, dtype=np.float64)
        return float((np.sum(fo.softplus(theta - g[:B])) + np.sum(fo.softplus(theta - g[B:2 * B]))) / B)
    monkeypatch.setattr(fo, "ff_loss", bad)
    _caught(pins.test_loss_closed_forms)


def test_softplus_without_the_absolute_value_is_caught(monkeypatch):
    def bad(t):
        t = np.asarray(t, dtype=np.float64)
        with np.errstate(over="ignore"):
            return np.maximum(t, 0.0) + np.log1p(np.exp(-t))
    monkeypatch.setattr(fo, "softplus", bad)
    _caught(pins.test_softplus_stable_branch_agrees_with_naive)


def test_wrong_sign_of_the_negative_rows_gradient_is_caught(monkeypatch):
    def bad(g, theta, B):
        g = np.asarray(g, dtype=np.float64)
        d = np.empty_like(g)
        d[:B] = -fo.sigmoid(theta - g[:B]) / B
        d[B:2 * B] = -fo.sigmoid(g[B:2 * B] - theta) / B
        return d
    monkeypatch.setattr(fo, "dloss_dg", bad)
    _caught(pins.test_gradient_matches_finite_differences_4_to_3)
    _caught(pins.test_loss_closed_forms)


def _step_with(dz_factor=2.0, transpose=False):
    """A copy of the oracle's fp64 layer step with one planted change: the
    factor of dL/dz = factor * c * h, or the weight-gradient product's
    operands swapped."""
    def step(state, x_in, B, theta, hp, emulate_bf16=False, rounding=None):
        x_in = np.asarray(x_in, dtype=np.float64)
        s = 1.0 / np.maximum(fo.row_norm(x_in), fo.NORM_EPS)
        x_hat = s[:, None] * x_in
        Z, H = fo.layer_forward(x_hat, state.W, state.b)
        g = fo.goodness(H)
        c = fo.dloss_dg(g, theta, B)
        dZ = dz_factor * c[:, None] * H * (Z > 0)
        dW = x_hat.T @ dZ if transpose else dZ.T @ x_hat
        return dict(H=H, g=g, s=s, loss=fo.ff_loss(g, theta, B), dW=dW, db=np.sum(dZ, axis=0))
    return step


def test_dropped_factor_two_of_the_local_gradient_is_caught(monkeypatch):
    monkeypatch.setattr(fo, "layer_train_step", _step_with(dz_factor=1.0))
    _caught(pins.test_gradient_matches_finite_differences_4_to_3)


def test_transposed_weight_gradient_is_caught(monkeypatch):
    monkeypatch.setattr(fo, "layer_train_step", _step_with(transpose=True))
    _caught(pins.test_gradient_matches_finite_differences_4_to_3, errors=(AssertionError, ValueError))


def test_the_planted_step_copy_itself_passes(monkeypatch):
    # the copy with no change passes the same pin, so the cases above fail for their plants
    monkeypatch.setattr(fo, "layer_train_step", _step_with())
    pins.test_gradient_matches_finite_differences_4_to_3()


# ------------------------------------------------------------------- Adam
def test_adam_without_bias_correction_is_caught(monkeypatch):
    def bad(w, grad, m, v, t, hp):
        grad = np.asarray(grad, dtype=np.float64)
        m = hp.beta1 * np.asarray(m, dtype=np.float64) + (1.0 - hp.beta1) * grad
        v = hp.beta2 * np.asarray(v, dtype=np.float64) + (1.0 - hp.beta2) * grad * grad
        return np.asarray(w, dtype=np.float64) - hp.lr * m / (np.sqrt(v) + hp.eps), m, v
    monkeypatch.setattr(fo, "adam_update", bad)
    _caught(pins.test_adam_first_step_closed_form_and_zero_gradient)


def test_adam_with_eps_inside_the_root_is_caught(monkeypatch):
    def bad(w, grad, m, v, t, hp):
        grad = np.asarray(grad, dtype=np.float64)
        m = hp.beta1 * np.asarray(m, dtype=np.float64) + (1.0 - hp.beta1) * grad
        v = hp.beta2 * np.asarray(v, dtype=np.float64) + (1.0 - hp.beta2) * grad * grad
        m_hat, v_hat = m / (1.0 - hp.beta1 ** t), v / (1.0 - hp.beta2 ** t)
        return np.asarray(w, dtype=np.float64) - hp.lr * m_hat / np.sqrt(v_hat + hp.eps), m, v
    monkeypatch.setattr(fo, "adam_update", bad)
    _caught(pins.test_adam_first_step_closed_form_and_zero_gradient)


def _adam_with_rates(b1, b2):
    """Adam whose moment decay rates are b1 (first) and b2 (second)
    regardless of the hyper-parameters passed in."""
    def bad(w, grad, m, v, t, hp):
        grad = np.asarray(grad, dtype=np.float64)
        m = b1 * np.asarray(m, dtype=np.float64) + (1.0 - b1) * grad
        v = b2 * np.asarray(v, dtype=np.float64) + (1.0 - b2) * grad * grad
        m_hat, v_hat = m / (1.0 - b1 ** t), v / (1.0 - b2 ** t)
        return np.asarray(w, dtype=np.float64) - hp.lr * m_hat / (np.sqrt(v_hat) + hp.eps), m, v
    return bad


def test_adam_with_the_decay_rates_swapped_is_caught(monkeypatch):
    # swapped consistently in the moments and their bias corrections: the
    # one-step and constant-gradient pins cannot see it
    monkeypatch.setattr(fo, "adam_update", _adam_with_rates(0.999, 0.9))
    pins.test_adam_first_step_closed_form_and_zero_gradient()
    _caught(pins.test_adam_two_steps_with_different_gradients_pin_both_decay_rates)


def test_adam_with_a_wrong_second_moment_rate_is_caught(monkeypatch):
    monkeypatch.setattr(fo, "adam_update", _adam_with_rates(0.9, 0.99))
    _caught(pins.test_adam_two_steps_with_different_gradients_pin_both_decay_rates)


def test_adam_with_a_wrong_first_moment_rate_is_caught(monkeypatch):
    monkeypatch.setattr(fo, "adam_update", _adam_with_rates(0.8, 0.999))
    _caught(pins.test_adam_two_steps_with_different_gradients_pin_both_decay_rates)


def test_the_planted_adam_copy_with_the_right_rates_passes(monkeypatch):
    monkeypatch.setattr(fo, "adam_update", _adam_with_rates(0.9, 0.999))
    pins.test_adam_two_steps_with_different_gradients_pin_both_decay_rates()


# ---------------------------------------------------------------- predict
def test_predict_counting_layer_one_is_caught(monkeypatch):
    def bad(states, x_raw, emulate_bf16=False, n_classes=fo.N_CLASSES):
        x_raw = np.asarray(x_raw, dtype=np.float64)
        G = np.zeros((x_raw.shape[0], n_classes))
        for c in range(n_classes):
            a = fo.overlay_label(x_raw, np.full(x_raw.shape[0], c))
            for st in states:
                f = fo.layer_forward_full(st, a)
                G[:, c] += f["g"]
                a = f["H"]
        return np.argmax(G, axis=1), G
    monkeypatch.setattr(fo, "predict", bad)
    _caught(pins.test_predict_matches_brute_force, (12, 5, 4, 3))


def test_predict_with_ties_to_the_highest_label_is_caught(monkeypatch):
    orig = fo.predict

    def bad(states, x_raw, emulate_bf16=False, n_classes=fo.N_CLASSES):
        _, G = orig(states, x_raw, emulate_bf16=emulate_bf16, n_classes=n_classes)
        return n_classes - 1 - np.argmax(G[:, ::-1], axis=1), G
    monkeypatch.setattr(fo, "predict", bad)
    _caught(pins.test_predict_ties_go_to_lowest_label)


# ----------------------------------------------------------- softmax head
def test_cross_entropy_summed_over_rows_is_caught(monkeypatch):
    def bad(z, labels):
        z = np.asarray(z, dtype=np.float64)
        m = np.max(z, axis=1)
        lse = m + np.log(np.sum(np.exp(z - m[:, None]), axis=1))
        return float(np.sum(lse - z[np.arange(z.shape[0]), np.asarray(labels)]))
    monkeypatch.setattr(fo, "cross_entropy", bad)
    _caught(pins.test_cross_entropy_closed_forms)


def test_head_gradient_without_the_row_mean_is_caught(monkeypatch):
    def bad(z, labels):
        p = fo.softmax(z)
        p[np.arange(p.shape[0]), np.asarray(labels)] -= 1.0
        return p
    monkeypatch.setattr(fo, "dce_dz", bad)
    _caught(pins.test_cross_entropy_closed_forms)
    _caught(pins.test_head_gradient_matches_finite_differences)


def test_po_predict_on_the_normalised_activity_is_caught(monkeypatch):
    def bad(states, heads, x_raw, emulate_bf16=False):
        a = fo.overlay_neutral(x_raw)
        for st in states:
            a = fo.layer_forward_full(st, a)["H"]
        return fo.head_predict(heads[-1], fo.normalise(a))
    monkeypatch.setattr(fo, "po_predict", bad)
    _caught(pins.test_po_predict_hand_built_block_selects_the_class)


def test_lr_cooldown_to_half_instead_of_zero_is_caught(monkeypatch):
    def bad(lr0, epoch, total_epochs, cooldown_start):
        if cooldown_start >= 1.0:
            return lr0
        e0 = cooldown_start * total_epochs
        if epoch < e0:
            return lr0
        return lr0 * (0.5 + 0.5 * (total_epochs - epoch) / (total_epochs - e0))
    monkeypatch.setattr(fo, "lr_at", bad)
    _caught(pins.test_lr_cooldown_closed_forms)


# ------------------------------------------------------------ bf16 rounding
def test_bf16_truncation_instead_of_nearest_even_is_caught(monkeypatch):
    def bad(a):
        m, e = np.frexp(np.asarray(a, dtype=np.float64))
        return np.ldexp(np.trunc(m * 256.0), e - 8)
    monkeypatch.setattr(fo, "bf16_round", bad)
    _caught(pins.test_bf16_round_matches_torch_conversion)


def test_bf16_ties_away_from_zero_is_caught(monkeypatch):
    def bad(a):
        m, e = np.frexp(np.asarray(a, dtype=np.float64))
        return np.ldexp(np.sign(m) * np.floor(np.abs(m) * 256.0 + 0.5), e - 8)
    monkeypatch.setattr(fo, "bf16_round", bad)
    _caught(pins.test_bf16_round_matches_torch_conversion)
