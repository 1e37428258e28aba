"""Host-side checks of the C ABI that need no GPU: the library builds for
sm_103a, loads, exports every function include/ff.h declares, and rejects bad
arguments before touching the device."""

import ctypes
import os
import re
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ff.h")


def _declared():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^FF_API\s+[\w\s\*]*?\b(ff_\w+)\s*\(", text, flags=re.M)))


@pytest.fixture(scope="module")
def libff():
    if not shutil.which("nvcc") and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no CUDA toolkit")
    from paper_2404_08573_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_boundary():
    names = _declared()
    for required in ("ff_layer_create", "ff_layer_train_step", "ff_overlay_label", "ff_predict",
                     "ff_layer_destroy", "ff_layer_forward", "ff_layer_get_state", "ff_layer_set_state",
                     "ff_net_create", "ff_net_train_step"):
        assert required in names


def test_every_declared_symbol_is_exported(libff):
    for name in _declared():
        assert hasattr(libff, name), f"{name} declared in ff.h but not exported"


def test_status_strings_and_row_stride(libff):
    libff.ff_status_string.restype = ctypes.c_char_p
    names = [libff.ff_status_string(i).decode() for i in range(7)]
    assert names == ["FF_OK", "FF_ERR_INVALID_ARG", "FF_ERR_CUDA", "FF_ERR_OOM", "FF_ERR_TIMEOUT",
                     "FF_ERR_NONFINITE", "FF_ERR_UNSUPPORTED"]
    assert [libff.ff_row_stride(f) for f in (1, 8, 9, 784, 2000, 777, 0)] == [8, 8, 16, 784, 2000, 784, 0]


def test_invalid_arguments_are_rejected_on_the_host(libff):
    from paper_2404_08573_gb300.ff import LayerConfig
    out = ctypes.c_void_p(1234)
    # null config: rejected before any CUDA call, *out cleared
    assert libff.ff_layer_create(None, None, ctypes.byref(out)) == 1 and out.value is None
    bad = LayerConfig(0, 10, 1, 2.0, 0.03, 0.9, 0.999, 1e-8, 1, 0, 0, 0)
    assert libff.ff_layer_create(ctypes.byref(bad), None, ctypes.byref(out)) == 1
    bad = LayerConfig(10, 10, 1, 2.0, 0.03, 1.5, 0.999, 1e-8, 1, 0, 0, 0)
    assert libff.ff_layer_create(ctypes.byref(bad), None, ctypes.byref(out)) == 1
    bad = LayerConfig(10, 10, 1, 2.0, 0.03, 0.9, 0.999, 1e-8, 7, 0, 0, 0)
    assert libff.ff_layer_create(ctypes.byref(bad), None, ctypes.byref(out)) == 1
    assert libff.ff_layer_destroy(None) == 0
    assert libff.ff_layer_train_step(None, None, None, None, 1, None, None, None, None, None) == 1
    assert libff.ff_layer_forward(None, None, None, None, 1, None, None, None, None) == 1
    assert libff.ff_overlay_label(None, None, 4, 5, None, None, 1, None) == 1   # features < 10
    assert libff.ff_overlay_label(None, None, 0, 784, None, None, 1, None) == 0  # empty: no-op
    assert libff.ff_predict(None, 1, None, 4, None, None, None) == 1
    assert libff.ff_adaptive_negatives(None, 1, None, None, 4, None, None, None) == 1
    assert libff.ff_head_destroy(None) == 0
    assert libff.ff_head_create(None, ctypes.byref(out)) == 1
    assert libff.ff_head_train_step(None, None, 1, None, None, 4, None, None) == 1
    assert libff.ff_head_predict(None, None, 1, None, 4, None, None, None) == 1
    assert libff.ff_head_check(None) == 1
    assert libff.ff_pff_destroy(None) == 0
    assert libff.ff_pff_wait(None, 10) == 1
    assert libff.ff_net_wait(None, 10) == 1
    assert libff.ff_layer_get_stats(None, None) == 1
    assert libff.ff_net_create_po(None, None, 2, 8, 2, ctypes.byref(out)) == 1
    assert libff.ff_net_po_train_step(None, None, None, 4, None, None) == 1
    assert libff.ff_po_train_step(None, None, None, 1, None, None, 4, None, None, None, None) == 1
    assert libff.ff_po_predict(None, 1, None, None, 4, None, None, None) == 1
    assert libff.ff_pff_create(None, 2, None, ctypes.byref(out)) == 1
    assert libff.ff_pff_run(None, None, None, 0, 1, None, None) == 1
    assert libff.ff_net_create(None, 2, 8, 2, ctypes.byref(out)) == 1
    assert libff.ff_net_train_step(None, None, None, 1, None, None) == 1
    assert libff.ff_net_train_step_images(None, None, None, 1, None, None) == 1
    assert libff.ff_layer_get_state(None, None, None, None, None, None, None, None) == 1
    assert libff.ff_layer_check(None) == 1
    assert libff.ff_layer_set_fused_local_grad(None, 1) == 1
    assert libff.ff_layer_get_grad_operand(None, None, 4) == 1
    assert libff.ff_net_train_epoch(None, None, None, 4, 2, 2, None, None) == 1
    libff.ff_net_epoch_trace.restype = ctypes.c_longlong
    assert libff.ff_net_epoch_trace(None, 1, None, ctypes.c_longlong(0)) == -1
    assert libff.ff_head_train_epoch(None, None, 1, None, None, 4, 2, None, None) == 1
    # the allocation-free forward: sizes and pointers checked, and the scratch limit
    # (rows * 2 * ceil(out / 256) partials) applied, before any CUDA call
    fake = ctypes.c_void_p(256)
    assert libff.ff_forward_noalloc(None, None, None, None, -1, 16, 8, None, None, None, None, None) == 1
    assert libff.ff_forward_noalloc(None, None, None, None, 0, 16, 8, None, None, None, None, None) == 0
    assert libff.ff_forward_noalloc(None, None, None, None, 4, 16, 8, None, None, None, None, None) == 1
    assert libff.ff_forward_noalloc(fake, fake, fake, None, 4, 0, 8, fake, None, None, None, None) == 1
    assert libff.ff_forward_noalloc(fake, fake, fake, None, 1 << 21, 16, 8, fake, None, None, None, None) == 1


def test_every_function_the_binding_calls_has_a_declared_signature(libff):
    """ctypes passes an undeclared argument list as C ints: a device pointer
    would lose its upper 32 bits.  Every ff_* function the binding calls must
    therefore have its argument types set, and exist in include/ff.h."""
    from paper_2404_08573_gb300 import ff
    src = open(os.path.join(ROOT, "paper_2404_08573_gb300", "ff.py")).read()
    called = sorted(set(re.findall(r"lib\(\)\.(ff_\w+)\(", src)))
    assert called, "no calls found"
    L = ff.lib()
    declared = set(_declared())
    for name in called:
        assert name in declared, f"{name} is called by the binding but not declared in ff.h"
        assert getattr(L, name).argtypes is not None, f"{name} has no argtypes in the binding"
