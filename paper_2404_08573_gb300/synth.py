"""Seeded synthetic inputs for the Forward-Forward (FF) train step and predict.

This module holds the input generators only: it does none of the method's
arithmetic (no overlay, normalisation, goodness, loss or update). The tests,
the benchmark and the CPU oracle's callers all draw their inputs here, so the
CUDA path and the oracle see the same numbers.

Random numbers come from a counter-based SplitMix64 generator (Steele, Lea and
Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014; the
64-bit finaliser constants of Vigna's public-domain splitmix64.c).  Output
``i`` (0-based) of stream ``(seed, stream)`` is ``mix(state0 + (i + 1) * GAMMA)``
with ``state0 = mix((seed << 8) | stream)``; a uniform double in [0, 1) is
``(out >> 11) * 2**-53``.  The device-side weight initialiser of the C library
implements the same definition, so ``he_uniform`` equals a freshly created
layer's weights bit for bit.

Shapes and distributions follow the paper's workloads: MNIST-shaped rows of
784 features (the 784-2000-2000-2000-2000 network of the implementation
details, §5.1) and CIFAR-shaped rows of 3072 features (§5.5).  The datasets
themselves are not used: each MNIST-shaped feature is 0 with probability 0.8,
else U(0, 1); CIFAR-shaped features are dense U(0, 1).  Labels are uniform over
the 10 classes; a negative label is uniform over the 9 wrong classes
(``(y + 1 + u9) mod 10``), the random-wrong-label negative data of §3 and §5
(RandomNEG), drawn fresh per sample.
"""

from __future__ import annotations

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)

# Stream identifiers (low 8 bits of the stream key).
STREAM_FEATURES = 1
STREAM_LABELS = 2
STREAM_NEG_OFFSETS = 3
STREAM_WEIGHTS = 4  # + 0 ; the device initialiser uses the same id
STREAM_PROTOTYPES = 5
STREAM_PROTO_PICK = 6

N_CLASSES = 10


def _mix(z: np.ndarray) -> np.ndarray:
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def stream_state(seed: int, stream: int) -> np.uint64:
    key = np.uint64(((int(seed) & ((1 << 56) - 1)) << 8) | (int(stream) & 0xFF))
    return _mix(np.array([key], dtype=np.uint64))[0]


def raw_u64(seed: int, stream: int, start: int, count: int) -> np.ndarray:
    """Outputs ``start .. start+count-1`` of the stream, as uint64."""
    s0 = stream_state(seed, stream)
    idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix(s0 + idx * GAMMA)


def uniform(seed: int, stream: int, count: int, start: int = 0) -> np.ndarray:
    """``count`` doubles in [0, 1) with 53 random bits each."""
    return (raw_u64(seed, stream, start, count) >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def mnist_like(n: int, seed: int = 0, features: int = 784, start_row: int = 0) -> np.ndarray:
    """[n, features] float32: each feature 0 w.p. 0.8, else U(0, 1).

    One uniform ``u`` per feature: ``u < 0.8`` gives 0, otherwise
    ``(u - 0.8) / 0.2`` (uniform on [0, 1) given ``u >= 0.8``).
    """
    u = uniform(seed, STREAM_FEATURES, n * features, start=start_row * features)
    v = np.where(u < 0.8, 0.0, (u - 0.8) / 0.2)
    return v.astype(np.float32).reshape(n, features)


def cifar_like(n: int, seed: int = 0, features: int = 3072, start_row: int = 0) -> np.ndarray:
    """[n, features] float32 dense U(0, 1) (32x32x3-shaped rows)."""
    u = uniform(seed, STREAM_FEATURES, n * features, start=start_row * features)
    return u.astype(np.float32).reshape(n, features)


def labels(n: int, seed: int = 0, start: int = 0) -> np.ndarray:
    """[n] int32 uniform over 0..9."""
    u = uniform(seed, STREAM_LABELS, n, start=start)
    return np.minimum((u * N_CLASSES).astype(np.int64), N_CLASSES - 1).astype(np.int32)


def negative_labels(y: np.ndarray, seed: int = 0, start: int = 0) -> np.ndarray:
    """[n] int32 wrong labels ``(y + 1 + u9) mod 10`` with u9 uniform on 0..8.

    ``start`` is the counter offset, so a fresh draw per step uses a new offset.
    """
    y = np.asarray(y, dtype=np.int64)
    u = uniform(seed, STREAM_NEG_OFFSETS, y.shape[0], start=start)
    u9 = np.minimum((u * (N_CLASSES - 1)).astype(np.int64), N_CLASSES - 2)
    return ((y + 1 + u9) % N_CLASSES).astype(np.int32)


def he_uniform(init_seed: int, out_features: int, in_features: int) -> np.ndarray:
    """[out, in] float32 W ~ U(-sqrt(6/in), +sqrt(6/in)) from stream ``STREAM_WEIGHTS``.

    Element (n, k) uses output ``n * in + k``; the value is computed in double
    as ``(2u - 1) * sqrt(6 / in)`` and rounded once to float32.
    """
    u = uniform(init_seed, STREAM_WEIGHTS, out_features * in_features)
    bound = np.sqrt(6.0 / in_features)
    return ((2.0 * u - 1.0) * bound).astype(np.float32).reshape(out_features, in_features)


def pair_batch(x: np.ndarray, y: np.ndarray, y_neg: np.ndarray):
    """The concatenated positive/negative batch of §4: rows 0..B-1 carry the
    true labels, rows B..2B-1 the same images with wrong labels.

    Returns (x2 [2B, in] float32, labels2 [2B] int32).
    """
    x2 = np.concatenate([x, x], axis=0).astype(np.float32, copy=False)
    l2 = np.concatenate([y, y_neg]).astype(np.int32)
    return np.ascontiguousarray(x2), l2


def learnable_task(n: int, seed: int = 0, features: int = 784, start_row: int = 0, on_support: float = 0.5):
    """A learnable MNIST-shaped task for end-to-end accuracy checks.

    Class c owns a fixed random support of 157 feature positions among
    features 10..783.  Each feature of a sample of class c is nonzero with
    probability 0.2; a nonzero feature lands on the class support with
    probability ``on_support`` (else anywhere), so about 20 % of features are
    nonzero and the class is recoverable from where the mass sits (less
    reliably for a smaller ``on_support``).  Values are U(0, 1).
    Returns (x [n, features] float32, y [n] int32).
    """
    rng_support = uniform(seed, STREAM_PROTOTYPES, N_CLASSES * (features - 10))
    order = np.argsort(rng_support.reshape(N_CLASSES, features - 10), axis=1, kind="stable")
    support = order[:, :157] + 10  # [10, 157]
    y = labels(n, seed, start=start_row)
    u = uniform(seed, STREAM_FEATURES, n * features * 2, start=start_row * features * 2).reshape(n, features, 2)
    x = np.zeros((n, features), dtype=np.float64)
    on = np.zeros((n, features), dtype=bool)
    on[np.arange(n)[:, None], support[y]] = True
    # nonzero probability: features on the class support carry the class mass.
    p_on = 0.2 * on_support * features / 157.0 + 0.2 * (1.0 - on_support)
    p_off = 0.2 * (1.0 - on_support)
    p = np.where(on, p_on, p_off)
    p[:, :10] = 0.0
    x = np.where(u[..., 0] < p, u[..., 1], 0.0)
    return x.astype(np.float32), y
