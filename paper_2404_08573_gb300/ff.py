"""Python binding of libff (ctypes).  Argument marshalling only.

Every computation runs in libff's CUDA kernels; PyTorch supplies device
memory (tensors whose data pointers are passed through) and streams.  There
is no fallback: if libff.so is missing or the GPU cannot run it, calls raise.

Names follow the C ABI in include/ff.h:
``Layer`` (ff_layer_*), ``overlay_label``, ``predict``, ``adaptive_negatives``,
``Net`` (ff_net_*), ``Head`` (ff_head_*), ``Pff`` (ff_pff_*), ``po_train_step_raw``/
``po_train_step_act``/``po_predict`` (ff_po_*), ``forward_noalloc``.
"""

from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_float, c_int, c_longlong, c_ulonglong, c_void_p

import numpy as np
import torch

FF_FP32, FF_BF16 = 0, 1
_STATUS = {
    0: "FF_OK", 1: "FF_ERR_INVALID_ARG", 2: "FF_ERR_CUDA", 3: "FF_ERR_OOM",
    4: "FF_ERR_TIMEOUT", 5: "FF_ERR_NONFINITE", 6: "FF_ERR_UNSUPPORTED", 7: "FF_ERR_DEVICE_CHECK",
}
# FF_LIB_VARIANT=checked loads the build with device-side checks (build.py).
LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)),
                        "libff_checked.so" if os.environ.get("FF_LIB_VARIANT") == "checked" else "libff.so")


class FFError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {_STATUS.get(status, status)}")


class LayerConfig(ctypes.Structure):
    _fields_ = [
        ("in_features", c_int), ("out_features", c_int), ("has_bias", c_int),
        ("theta", c_float), ("lr", c_float), ("beta1", c_float), ("beta2", c_float), ("eps", c_float),
        ("prec", c_int), ("init_seed", c_ulonglong), ("max_rows", c_int), ("keep_grad", c_int),
    ]


class HeadConfig(ctypes.Structure):
    _fields_ = [
        ("n_features", c_int), ("lr", c_float), ("beta1", c_float), ("beta2", c_float), ("eps", c_float),
        ("max_rows", c_int),
    ]


class PffConfig(ctypes.Structure):
    _fields_ = [
        ("n_pairs", c_int), ("batch_pairs", c_int), ("epochs_per_chapter", c_int), ("chapters", c_int),
        ("mode", c_int), ("nodes", c_int), ("cooldown_start", c_float),
    ]


_lib = None


def lib():
    """Loads libff.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                "libff.so is not built; run `python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        L.ff_status_string.restype = ctypes.c_char_p
        L.ff_status_string.argtypes = [c_int]
        L.ff_row_stride.restype = c_int
        L.ff_row_stride.argtypes = [c_int]
        L.ff_kernel_launches.restype = ctypes.c_ulonglong
        L.ff_kernel_launches.argtypes = []
        sig = {
            "ff_layer_create": [POINTER(LayerConfig), c_void_p, POINTER(c_void_p)],
            "ff_layer_destroy": [c_void_p],
            "ff_overlay_label": [c_void_p, c_void_p, c_int, c_int, c_void_p, c_void_p, c_int, c_void_p],
            "ff_layer_forward": [c_void_p, c_void_p, c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_void_p,
                                 c_void_p],
            "ff_layer_train_step": [c_void_p, c_void_p, c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_void_p,
                                    c_void_p, c_void_p],
            "ff_predict": [c_void_p, c_int, c_void_p, c_int, c_void_p, c_void_p, c_void_p],
            "ff_adaptive_negatives": [c_void_p, c_int, c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_void_p],
            "ff_layer_get_state": [c_void_p] + [c_void_p] * 6 + [POINTER(c_longlong)],
            "ff_layer_set_state": [c_void_p] + [c_void_p] * 6 + [c_longlong],
            "ff_layer_get_grad": [c_void_p, c_void_p, c_void_p],
            "ff_layer_get_grad_operand": [c_void_p, c_void_p, c_int],
            "ff_layer_check": [c_void_p],
            "ff_layer_set_fused_local_grad": [c_void_p, c_int],
            "ff_layer_get_stats": [c_void_p, c_void_p],
            "ff_layer_selftest_wait": [c_void_p, ctypes.c_uint, c_void_p],
            "ff_net_create": [c_void_p, c_int, c_int, c_int, POINTER(c_void_p)],
            "ff_net_destroy": [c_void_p],
            "ff_net_train_step": [c_void_p, c_void_p, c_void_p, c_int, c_void_p, c_void_p],
            "ff_net_train_step_images": [c_void_p, c_void_p, c_void_p, c_int, c_void_p, c_void_p],
            "ff_net_sync": [c_void_p, c_void_p],
            "ff_net_train_epoch": [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p],
            "ff_net_epoch_trace": [c_void_p, c_int, c_void_p, c_longlong],
            "ff_net_create_po": [c_void_p, c_void_p, c_int, c_int, c_int, POINTER(c_void_p)],
            "ff_net_po_train_step": [c_void_p, c_void_p, c_void_p, c_int, c_void_p, c_void_p],
            "ff_forward_noalloc": [c_void_p, c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p,
                                   c_void_p, c_void_p, c_void_p],
            "ff_head_create": [POINTER(HeadConfig), POINTER(c_void_p)],
            "ff_head_destroy": [c_void_p],
            "ff_head_train_step": [c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_int, c_void_p, c_void_p],
            "ff_head_train_epoch": [c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_int, c_int, c_void_p, c_void_p],
            "ff_head_predict": [c_void_p, c_void_p, c_int, c_void_p, c_int, c_void_p, c_void_p, c_void_p],
            "ff_head_get_state": [c_void_p] + [c_void_p] * 6 + [POINTER(c_longlong)],
            "ff_head_set_state": [c_void_p] + [c_void_p] * 6 + [c_longlong],
            "ff_head_get_grad": [c_void_p, c_void_p, c_void_p],
            "ff_head_check": [c_void_p],
            "ff_po_train_step": [c_void_p, c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_int, c_void_p, c_void_p,
                                 c_void_p, c_void_p],
            "ff_po_predict": [c_void_p, c_int, c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_void_p],
            "ff_pff_create": [c_void_p, c_int, POINTER(PffConfig), POINTER(c_void_p)],
            "ff_pff_destroy": [c_void_p],
            "ff_pff_wait": [c_void_p, ctypes.c_uint],
            "ff_net_wait": [c_void_p, ctypes.c_uint],
            "ff_pff_run": [c_void_p, c_void_p, c_void_p, c_int, c_int, c_void_p, c_void_p],
        }
        for name, args in sig.items():
            f = getattr(L, name)
            f.restype = c_int
            f.argtypes = args
        _lib = L
    return _lib


def _check(status: int, what: str):
    if status != 0:
        raise FFError(status, what)


def row_stride(features: int) -> int:
    return lib().ff_row_stride(int(features))


def kernel_launches() -> int:
    """ff_kernel_launches: libff's kernel launches in this process so far."""
    return int(lib().ff_kernel_launches())


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _ptr(t, dtype=None, what="tensor", need_cuda=True):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{what} must be a torch.Tensor")
    if need_cuda and not t.is_cuda:
        raise ValueError(f"{what} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{what} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{what} must be contiguous")
    return t.data_ptr()


def act_dtype(prec: str):
    return torch.bfloat16 if prec == "bf16" else torch.float32


class Layer:
    """One FF layer (``ff_layer``): parameters, Adam moments and workspace on the GPU."""

    def __init__(self, in_features: int, out_features: int, prec: str = "bf16", theta: float = 2.0,
                 lr: float = 0.03, beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8,
                 has_bias: bool = True, init_seed: int = 0, max_rows: int = 0, keep_grad: bool = False,
                 stream=None):
        if prec not in ("bf16", "fp32"):
            raise ValueError("prec must be 'bf16' or 'fp32'")
        self.in_features, self.out_features, self.prec = int(in_features), int(out_features), prec
        self.dtype = act_dtype(prec)
        self.cfg = LayerConfig(self.in_features, self.out_features, int(bool(has_bias)), theta, lr, beta1, beta2,
                               eps, FF_BF16 if prec == "bf16" else FF_FP32, int(init_seed), int(max_rows),
                               int(bool(keep_grad)))
        h = c_void_p()
        _check(lib().ff_layer_create(ctypes.byref(self.cfg), c_void_p(_stream(stream)), ctypes.byref(h)),
               "ff_layer_create")
        self._h = h

    @property
    def handle(self):
        return self._h

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            _check(lib().ff_layer_destroy(self._h), "ff_layer_destroy")
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # buffers in the layer's activation format
    def new_activation(self, rows: int, features: int | None = None, device="cuda"):
        f = self.out_features if features is None else features
        return torch.zeros(rows, row_stride(f), dtype=self.dtype, device=device)

    def _x_args(self, x, labels, row_scale):
        if labels is not None:
            xp = _ptr(x, torch.float32, "x (raw input)")
            if x.shape[-1] != self.in_features:
                raise ValueError("raw x must have in_features columns")
            return xp, _ptr(labels, torch.int32, "labels"), None
        xp = _ptr(x, self.dtype, "x (activation)")
        if x.shape[-1] != row_stride(self.in_features):
            raise ValueError("activation x must have ff_row_stride(in_features) columns")
        return xp, None, _ptr(row_scale, torch.float32, "row_scale")

    def train_step(self, x, labels=None, row_scale=None, B=None, h_out=None, next_scale=None, goodness=None,
                   loss=None, stream=None):
        """ff_layer_train_step: rows 0..B-1 positive, B..2B-1 negative."""
        if B is None:
            B = x.shape[0] // 2
        xp, lp, sp = self._x_args(x, labels, row_scale)
        _check(lib().ff_layer_train_step(
            self._h, xp, lp, sp, int(B), _ptr(h_out, self.dtype, "h_out"),
            _ptr(next_scale, torch.float32, "next_scale"), _ptr(goodness, torch.float32, "goodness"),
            _ptr(loss, torch.float32, "loss"), c_void_p(_stream(stream))), "ff_layer_train_step")

    def forward(self, x, labels=None, row_scale=None, rows=None, h_out=None, next_scale=None, goodness=None,
                stream=None):
        """ff_layer_forward (L_i(x)) without an update."""
        if rows is None:
            rows = x.shape[0]
        xp, lp, sp = self._x_args(x, labels, row_scale)
        _check(lib().ff_layer_forward(
            self._h, xp, lp, sp, int(rows), _ptr(h_out, self.dtype, "h_out"),
            _ptr(next_scale, torch.float32, "next_scale"), _ptr(goodness, torch.float32, "goodness"),
            c_void_p(_stream(stream))), "ff_layer_forward")

    def get_state(self):
        N, K = self.out_features, self.in_features
        W = np.empty((N, K), np.float32); mW = np.empty_like(W); vW = np.empty_like(W)
        b = np.empty(N, np.float32); mb = np.empty_like(b); vb = np.empty_like(b)
        step = c_longlong()
        _check(lib().ff_layer_get_state(self._h, W.ctypes.data, b.ctypes.data, mW.ctypes.data, vW.ctypes.data,
                                        mb.ctypes.data, vb.ctypes.data, ctypes.byref(step)), "ff_layer_get_state")
        return dict(W=W, b=b, mW=mW, vW=vW, mb=mb, vb=vb, t=step.value)

    def set_state(self, W=None, b=None, mW=None, vW=None, mb=None, vb=None, t=0):
        N, K = self.out_features, self.in_features

        def host(a, shape):
            if a is None:
                return None, None
            a = np.ascontiguousarray(np.asarray(a, dtype=np.float32))
            if a.shape != shape:
                raise ValueError(f"expected shape {shape}, got {a.shape}")
            return a, a.ctypes.data
        keep = [host(W, (N, K)), host(b, (N,)), host(mW, (N, K)), host(vW, (N, K)), host(mb, (N,)), host(vb, (N,))]
        _check(lib().ff_layer_set_state(self._h, *[k[1] for k in keep], int(t)), "ff_layer_set_state")

    def get_grad(self):
        N, K = self.out_features, self.in_features
        dW = np.empty((N, K), np.float32); db = np.empty(N, np.float32)
        _check(lib().ff_layer_get_grad(self._h, dW.ctypes.data, db.ctypes.data), "ff_layer_get_grad")
        return dW, db

    def get_grad_operand(self, rows: int):
        """ff_layer_get_grad_operand: the last step's weight-gradient operand
        G = diag(s) dZ [rows, ff_row_stride(out_features)] as float64 (from
        bf16 or fp32; exact)."""
        ld = row_stride(self.out_features)
        if self.prec == "bf16":
            raw = np.empty((rows, ld), np.uint16)
            _check(lib().ff_layer_get_grad_operand(self._h, raw.ctypes.data, int(rows)), "ff_layer_get_grad_operand")
            return (raw.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        out = np.empty((rows, ld), np.float32)
        _check(lib().ff_layer_get_grad_operand(self._h, out.ctypes.data, int(rows)), "ff_layer_get_grad_operand")
        return out.astype(np.float64)

    def stats(self):
        """ff_layer_get_stats: (mean positive goodness, mean negative goodness,
        active-ReLU fraction) of the last train step."""
        out = np.zeros(3, np.float32)
        _check(lib().ff_layer_get_stats(self._h, out.ctypes.data), "ff_layer_get_stats")
        return tuple(float(v) for v in out)

    def check(self):
        _check(lib().ff_layer_check(self._h), "ff_layer_check")

    def set_fused_local_grad(self, enable: bool):
        """ff_layer_set_fused_local_grad: bf16 train steps form the local step in
        the forward GEMM's epilogue (True) or in a separate kernel (False, the
        default); bitwise the same results."""
        _check(lib().ff_layer_set_fused_local_grad(self._h, 1 if enable else 0), "ff_layer_set_fused_local_grad")

    def selftest_wait(self, timeout_us: int, stream=None):
        """ff_layer_selftest_wait: a bounded wait that is made to run out."""
        _check(lib().ff_layer_selftest_wait(self._h, int(timeout_us), c_void_p(_stream(stream))),
               "ff_layer_selftest_wait")


def overlay_label(x, labels, prec="bf16", out=None, row_scale=None, stream=None):
    """ff_overlay_label: returns the overlaid activation buffer."""
    rows, F = x.shape
    if out is None:
        out = torch.empty(rows, row_stride(F), dtype=act_dtype(prec), device=x.device)
    _check(lib().ff_overlay_label(_ptr(x, torch.float32, "x"), _ptr(labels, torch.int32, "labels"), rows, F,
                                  _ptr(out, act_dtype(prec), "out"), _ptr(row_scale, torch.float32, "row_scale"),
                                  FF_BF16 if prec == "bf16" else FF_FP32, c_void_p(_stream(stream))),
           "ff_overlay_label")
    return out


def predict(layers, x, pred=None, goodness=None, stream=None):
    """ff_predict: goodness prediction over the 10 label overlays.  Returns (pred, goodness)."""
    n = x.shape[0]
    if pred is None:
        pred = torch.empty(n, dtype=torch.int32, device=x.device)
    arr = (c_void_p * len(layers))(*[l.handle.value for l in layers])
    _check(lib().ff_predict(arr, len(layers), _ptr(x, torch.float32, "x"), n, _ptr(pred, torch.int32, "pred"),
                            _ptr(goodness, torch.float32, "goodness"), c_void_p(_stream(stream))), "ff_predict")
    return pred, goodness


def adaptive_negatives(layers, x, labels, neg=None, goodness=None, stream=None):
    """ff_adaptive_negatives: AdaptiveNEG negative labels (§5), each sample's
    strongest wrong label under goodness prediction.  Returns (neg, goodness)."""
    n = x.shape[0]
    if labels.shape[0] != n:
        raise ValueError("labels must have one entry per row of x")
    if neg is None:
        neg = torch.empty(n, dtype=torch.int32, device=x.device)
    arr = (c_void_p * len(layers))(*[l.handle.value for l in layers])
    _check(lib().ff_adaptive_negatives(arr, len(layers), _ptr(x, torch.float32, "x"),
                                       _ptr(labels, torch.int32, "labels"), n, _ptr(neg, torch.int32, "neg"),
                                       _ptr(goodness, torch.float32, "goodness"), c_void_p(_stream(stream))),
           "ff_adaptive_negatives")
    return neg, goodness


class Net:
    """ff_net: the layers of a net trained concurrently, one CUDA stream per layer."""

    def __init__(self, layers, max_B: int, depth: int = 2):
        self.layers = list(layers)
        arr = (c_void_p * len(self.layers))(*[l.handle.value for l in self.layers])
        h = c_void_p()
        _check(lib().ff_net_create(arr, len(self.layers), int(max_B), int(depth), ctypes.byref(h)), "ff_net_create")
        self._h = h

    def train_step(self, x, labels, B=None, loss=None, stream=None):
        if B is None:
            B = x.shape[0] // 2
        _check(lib().ff_net_train_step(self._h, _ptr(x, torch.float32, "x"), _ptr(labels, torch.int32, "labels"),
                                       int(B), _ptr(loss, torch.float32, "loss"), c_void_p(_stream(stream))),
               "ff_net_train_step")

    def train_step_images(self, x, labels, loss=None, stream=None):
        """ff_net_train_step_images: x [B, in] holds one image per pair, labels
        [2B] the true labels then the wrong ones."""
        B = x.shape[0]
        if labels.shape[0] != 2 * B:
            raise ValueError("labels must hold 2 * x.shape[0] entries (true labels, then wrong labels)")
        _check(lib().ff_net_train_step_images(self._h, _ptr(x, torch.float32, "x"),
                                              _ptr(labels, torch.int32, "labels"), int(B),
                                              _ptr(loss, torch.float32, "loss"), c_void_p(_stream(stream))),
               "ff_net_train_step_images")

    def train_epoch(self, x, labels, n_pairs: int, B: int, images_per_pair_row: int = 2, loss=None, stream=None):
        """ff_net_train_epoch: n_pairs pairs in batches of B pairs through the
        net in one persistent kernel (the tail batch stepwise); x holds
        images_per_pair_row rows per pair (2: stacked pair batches, 1: one
        image per pair), labels [2 * n_pairs] (per batch the true labels, then
        the wrong ones)."""
        if x.shape[0] != images_per_pair_row * n_pairs or labels.shape[0] != 2 * n_pairs:
            raise ValueError("x must have images_per_pair_row * n_pairs rows and labels 2 * n_pairs entries")
        _check(lib().ff_net_train_epoch(self._h, _ptr(x, torch.float32, "x"), _ptr(labels, torch.int32, "labels"),
                                        int(n_pairs), int(B), int(images_per_pair_row),
                                        _ptr(loss, torch.float32, "loss"), c_void_p(_stream(stream))),
               "ff_net_train_epoch")

    def epoch_trace(self, enable=None):
        """ff_net_epoch_trace: with enable=True/False switches per-task tracing
        of later train_epoch calls; returns the last traced epoch as
        (gemm [G, 6], stream [S, 6]) uint64 arrays (see include/ff.h), or None."""
        L = lib()
        L.ff_net_epoch_trace.restype = c_longlong
        if enable is not None:
            L.ff_net_epoch_trace(self._h, 1 if enable else 0, None, 0)
            return None
        cap = 2 + 6 * (1 << 22)
        buf = np.zeros(cap, np.uint64)
        n = L.ff_net_epoch_trace(self._h, -1, buf.ctypes.data, cap)
        if n < 2:
            return None
        g, st = int(buf[0]), int(buf[1])
        rec = buf[2:n].reshape(-1, 6)
        return rec[:g], rec[g:g + st]

    def sync(self, stream=None):
        _check(lib().ff_net_sync(self._h, c_void_p(_stream(stream))), "ff_net_sync")

    def wait(self, timeout_ms: int):
        """ff_net_wait: host-side wait with a deadline (raises FFError FF_ERR_TIMEOUT)."""
        _check(lib().ff_net_wait(self._h, int(timeout_ms)), "ff_net_wait")

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            lib().ff_net_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def forward_noalloc(x, row_scale, W_bf16, in_features, out_features, h_out, bias=None, goodness=None,
                    next_scale=None, device_status=None, stream=None):
    """ff_forward_noalloc: the bf16 forward pass from caller buffers only (no
    device allocation inside the library); see include/ff.h."""
    rows = x.shape[0]
    _check(lib().ff_forward_noalloc(
        _ptr(x, torch.bfloat16, "x"), _ptr(row_scale, torch.float32, "row_scale"),
        _ptr(W_bf16, torch.bfloat16, "W_bf16"), _ptr(bias, torch.float32, "bias"), int(rows), int(in_features),
        int(out_features), _ptr(h_out, torch.bfloat16, "h_out"), _ptr(goodness, torch.float32, "goodness"),
        _ptr(next_scale, torch.float32, "next_scale"), _ptr(device_status, torch.int32, "device_status"),
        c_void_p(_stream(stream))), "ff_forward_noalloc")


def _layer_array(layers):
    return (c_void_p * len(layers))(*[l.handle.value for l in layers])


class Head:
    """The softmax prediction head (``ff_head``) over layers 2..L of a net."""

    N_CLASSES = 10

    def __init__(self, n_features: int, lr: float = 1e-4, beta1: float = 0.9, beta2: float = 0.999,
                 eps: float = 1e-8, max_rows: int = 0):
        self.n_features = int(n_features)
        self.cfg = HeadConfig(self.n_features, lr, beta1, beta2, eps, int(max_rows))
        h = c_void_p()
        _check(lib().ff_head_create(ctypes.byref(self.cfg), ctypes.byref(h)), "ff_head_create")
        self._h = h

    @staticmethod
    def features_of(layers) -> int:
        """n_features for a layer chain: out_features of layers 2..L (of layer 1 when L == 1)."""
        return sum(l.out_features for l in (layers[1:] if len(layers) > 1 else layers))

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            _check(lib().ff_head_destroy(self._h), "ff_head_destroy")
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def train_step(self, layers, x, labels, loss=None, stream=None):
        n = x.shape[0]
        if labels.shape[0] != n:
            raise ValueError("labels must have one entry per row of x")
        _check(lib().ff_head_train_step(self._h, _layer_array(layers), len(layers), _ptr(x, torch.float32, "x"),
                                        _ptr(labels, torch.int32, "labels"), n, _ptr(loss, torch.float32, "loss"),
                                        c_void_p(_stream(stream))), "ff_head_train_step")

    def train_epoch(self, layers, x, labels, B, loss=None, stream=None):
        """ff_head_train_epoch: ceil(n / B) train steps on consecutive rows, the
        features of many steps formed by one forward pass."""
        n = x.shape[0]
        if labels.shape[0] != n:
            raise ValueError("labels must have one entry per row of x")
        _check(lib().ff_head_train_epoch(self._h, _layer_array(layers), len(layers), _ptr(x, torch.float32, "x"),
                                         _ptr(labels, torch.int32, "labels"), n, int(B),
                                         _ptr(loss, torch.float32, "loss"), c_void_p(_stream(stream))),
               "ff_head_train_epoch")

    def predict(self, layers, x, pred=None, logits=None, stream=None):
        """Returns (pred, logits)."""
        n = x.shape[0]
        if pred is None:
            pred = torch.empty(n, dtype=torch.int32, device=x.device)
        _check(lib().ff_head_predict(self._h, _layer_array(layers), len(layers), _ptr(x, torch.float32, "x"), n,
                                     _ptr(pred, torch.int32, "pred"), _ptr(logits, torch.float32, "logits"),
                                     c_void_p(_stream(stream))), "ff_head_predict")
        return pred, logits

    def get_state(self):
        C, F = self.N_CLASSES, self.n_features
        V = np.empty((C, F), np.float32); mV = np.empty_like(V); vV = np.empty_like(V)
        c = np.empty(C, np.float32); mc = np.empty_like(c); vc = np.empty_like(c)
        step = c_longlong()
        _check(lib().ff_head_get_state(self._h, V.ctypes.data, c.ctypes.data, mV.ctypes.data, vV.ctypes.data,
                                       mc.ctypes.data, vc.ctypes.data, ctypes.byref(step)), "ff_head_get_state")
        return dict(V=V, c=c, mV=mV, vV=vV, mc=mc, vc=vc, t=step.value)

    def set_state(self, V=None, c=None, mV=None, vV=None, mc=None, vc=None, t=0):
        C, F = self.N_CLASSES, self.n_features

        def host(a, shape):
            if a is None:
                return None, None
            a = np.ascontiguousarray(np.asarray(a, dtype=np.float32))
            if a.shape != shape:
                raise ValueError(f"expected shape {shape}, got {a.shape}")
            return a, a.ctypes.data
        keep = [host(V, (C, F)), host(c, (C,)), host(mV, (C, F)), host(vV, (C, F)), host(mc, (C,)), host(vc, (C,))]
        _check(lib().ff_head_set_state(self._h, *[k[1] for k in keep], int(t)), "ff_head_set_state")

    def get_grad(self):
        dV = np.empty((self.N_CLASSES, self.n_features), np.float32); dc = np.empty(self.N_CLASSES, np.float32)
        _check(lib().ff_head_get_grad(self._h, dV.ctypes.data, dc.ctypes.data), "ff_head_get_grad")
        return dV, dc

    def check(self):
        _check(lib().ff_head_check(self._h), "ff_head_check")


class Pff:
    """The chapter schedule (``ff_pff``) of a layer chain: Single-Layer PFF
    (one stream per layer) or All-Layers PFF (``nodes`` streams taking the
    chapters in turn)."""

    def __init__(self, layers, n_pairs: int, batch_pairs: int, epochs_per_chapter: int, chapters: int,
                 mode: str = "single_layer", nodes: int = 1, cooldown_start: float = 1.0):
        if mode not in ("single_layer", "all_layers"):
            raise ValueError("mode must be 'single_layer' or 'all_layers'")
        self.layers = list(layers)
        self.cfg = PffConfig(int(n_pairs), int(batch_pairs), int(epochs_per_chapter), int(chapters),
                             0 if mode == "single_layer" else 1, int(nodes), float(cooldown_start))
        h = c_void_p()
        _check(lib().ff_pff_create(_layer_array(self.layers), len(self.layers), ctypes.byref(self.cfg),
                                   ctypes.byref(h)), "ff_pff_create")
        self._h = h

    @property
    def batches(self) -> int:
        return (self.cfg.n_pairs + self.cfg.batch_pairs - 1) // self.cfg.batch_pairs

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            _check(lib().ff_pff_destroy(self._h), "ff_pff_destroy")
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def wait(self, timeout_ms: int):
        """ff_pff_wait: host-side wait with a deadline (raises FFError FF_ERR_TIMEOUT)."""
        _check(lib().ff_pff_wait(self._h, int(timeout_ms)), "ff_pff_wait")

    def run(self, x, labels, first: int, count: int, loss=None, stream=None):
        """Enqueues chapters first .. first+count-1; labels [count, 2P] int32."""
        _check(lib().ff_pff_run(self._h, _ptr(x, torch.float32, "x"), _ptr(labels, torch.int32, "labels"),
                                int(first), int(count), _ptr(loss, torch.float32, "loss"),
                                c_void_p(_stream(stream))), "ff_pff_run")


def _po_step(layer, block, x, labels, raw, row_scale, h_out, next_scale, loss, stream):
    n = x.shape[0]
    if labels.shape[0] != n:
        raise ValueError("labels must have one entry per row of x")
    xp = _ptr(x, torch.float32 if raw else layer.dtype, "x")
    _check(lib().ff_po_train_step(layer.handle, block._h, xp, int(bool(raw)),
                                  _ptr(row_scale, torch.float32, "row_scale"), _ptr(labels, torch.int32, "labels"), n,
                                  _ptr(h_out, layer.dtype, "h_out"), _ptr(next_scale, torch.float32, "next_scale"),
                                  _ptr(loss, torch.float32, "loss"), c_void_p(_stream(stream))), "ff_po_train_step")


def po_train_step_raw(layer, block, x, labels, h_out=None, next_scale=None, loss=None, stream=None):
    """ff_po_train_step on raw float32 input rows (the first layer, with the
    neutral label): one Performance-Optimized step of ``layer`` and its
    softmax ``block`` (a Head with n_features == layer.out_features)."""
    _po_step(layer, block, x, labels, True, None, h_out, next_scale, loss, stream)


def po_train_step_act(layer, block, x, labels, row_scale=None, h_out=None, next_scale=None, loss=None, stream=None):
    """ff_po_train_step on an activation buffer of the layer (a hidden layer)."""
    _po_step(layer, block, x, labels, False, row_scale, h_out, next_scale, loss, stream)


def po_predict(layers, block, x, pred=None, logits=None, stream=None):
    """ff_po_predict: the last layer's block's prediction.  Returns (pred, logits)."""
    n = x.shape[0]
    if pred is None:
        pred = torch.empty(n, dtype=torch.int32, device=x.device)
    _check(lib().ff_po_predict(_layer_array(layers), len(layers), block._h, _ptr(x, torch.float32, "x"), n,
                               _ptr(pred, torch.int32, "pred"), _ptr(logits, torch.float32, "logits"),
                               c_void_p(_stream(stream))), "ff_po_predict")
    return pred, logits



def save_checkpoint(path, layers, heads=()):
    """Writes every layer's and head's full state (parameters, Adam moments
    and step) to one .npz file, with the shapes needed to check a restore."""
    arrays = {}
    for k, l in enumerate(layers):
        st = l.get_state()
        for name, v in st.items():
            arrays[f"layer{k}.{name}"] = np.asarray(v)
        arrays[f"layer{k}.shape"] = np.array([l.in_features, l.out_features])
    for k, h in enumerate(heads):
        st = h.get_state()
        for name, v in st.items():
            arrays[f"head{k}.{name}"] = np.asarray(v)
    np.savez(path, n_layers=np.array(len(layers)), n_heads=np.array(len(heads)), **arrays)


def load_checkpoint(path, layers, heads=()):
    """Restores states written by save_checkpoint into layers (and heads) of
    the same shapes; raises ValueError on a mismatch."""
    with np.load(path) as z:
        if int(z["n_layers"]) != len(layers) or int(z["n_heads"]) != len(heads):
            raise ValueError("checkpoint holds a different number of layers or heads")
        for k, l in enumerate(layers):
            if tuple(z[f"layer{k}.shape"]) != (l.in_features, l.out_features):
                raise ValueError(f"layer {k}: checkpoint shape {tuple(z[f'layer{k}.shape'])}")
            l.set_state(**{n: z[f"layer{k}.{n}"] for n in ("W", "b", "mW", "vW", "mb", "vb")},
                        t=int(z[f"layer{k}.t"]))
        for k, h in enumerate(heads):
            h.set_state(**{n: z[f"head{k}.{n}"] for n in ("V", "c", "mV", "vV", "mc", "vc")},
                        t=int(z[f"head{k}.t"]))


class PoNet(Net):
    """A Performance-Optimized net on one CUDA stream per layer
    (ff_net_create_po): layer k with its softmax block blocks[k]."""

    def __init__(self, layers, blocks, max_rows: int, depth: int = 2):
        self.layers, self.blocks = list(layers), list(blocks)
        h = c_void_p()
        _check(lib().ff_net_create_po(_layer_array(self.layers),
                                      (c_void_p * len(self.blocks))(*[b._h.value for b in self.blocks]),
                                      len(self.layers), int(max_rows), int(depth), ctypes.byref(h)),
               "ff_net_create_po")
        self._h = h

    def train_step(self, x, labels, loss=None, stream=None):
        n = x.shape[0]
        if labels.shape[0] != n:
            raise ValueError("labels must have one entry per row of x")
        _check(lib().ff_net_po_train_step(self._h, _ptr(x, torch.float32, "x"), _ptr(labels, torch.int32, "labels"),
                                          n, _ptr(loss, torch.float32, "loss"), c_void_p(_stream(stream))),
               "ff_net_po_train_step")

