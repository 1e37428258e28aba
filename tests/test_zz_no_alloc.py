"""The allocation-free forward entry point, for callers that cannot call
cudaMalloc (their device memory is owned by a host application's pool, or
their footprint must stay fixed after start-up), against the regular forward
pass of an ff_layer on the same inputs, on two calls in a row.

This file is collected last on purpose: the entry point's scratch array is
shared process-wide, and the test must pass both alone and after every other
GPU test."""

import numpy as np
import pytest

from tests.gpu_common import lib_ready, torch_cuda

pytestmark = pytest.mark.gpu


def test_noalloc_forward_matches_layer_forward_on_two_calls():
    """The same GEMM with the same tile shape and the same goodness kernel as
    ff_layer_forward, so the two agree bit for bit on every output.  The
    second call passes no status pointer (the error word then lives in the
    shared array); a third call with no rows still clears the status word."""
    torch = torch_cuda()
    ff = lib_ready()
    K, N, M = 784, 2000, 300           # several column tiles and a ragged row tile
    layer = ff.Layer(K, N, prec="bf16", init_seed=11)
    rng = np.random.default_rng(5)
    st = layer.get_state()
    layer.set_state(W=st["W"], b=(rng.standard_normal(N) * 0.05).astype(np.float32))
    st = layer.get_state()
    ldK = ff.row_stride(K)
    Wb = torch.zeros(N, ldK, dtype=torch.bfloat16, device="cuda")
    Wb[:, :K] = torch.from_numpy(st["W"]).cuda().to(torch.bfloat16)
    bias = torch.from_numpy(st["b"]).cuda()
    status = torch.full((1,), 7, dtype=torch.int32, device="cuda")
    for call in range(2):
        x = layer.new_activation(M, K)
        x[:, :K] = torch.rand(M, K, device="cuda", generator=torch.Generator("cuda").manual_seed(call)).to(
            torch.bfloat16)
        s = 1.0 / torch.linalg.vector_norm(x.float(), dim=1).clamp_min(1e-12)
        h_ref, h = layer.new_activation(M), layer.new_activation(M)
        g_ref, g = torch.empty(M, device="cuda"), torch.empty(M, device="cuda")
        n_ref, n = torch.empty(M, device="cuda"), torch.empty(M, device="cuda")
        layer.forward(x, row_scale=s, h_out=h_ref, goodness=g_ref, next_scale=n_ref)
        ff.forward_noalloc(x, s, Wb, K, N, h, bias=bias, goodness=g, next_scale=n,
                           device_status=status if call == 0 else None)
        torch.cuda.synchronize()
        if call == 0:
            assert status.item() == 0
        assert torch.equal(g, g_ref), f"call {call}: goodness differs"
        assert torch.equal(n, n_ref), f"call {call}: next-layer scale differs"
        assert torch.equal(h, h_ref), f"call {call}: activity differs"
        assert np.isfinite(g.cpu().numpy()).all()
    status.fill_(7)
    empty = layer.new_activation(0, K)
    ff.forward_noalloc(empty, torch.empty(0, device="cuda"), Wb, K, N, layer.new_activation(0), device_status=status)
    torch.cuda.synchronize()
    assert status.item() == 0


def test_noalloc_forward_rejects_requests_beyond_its_scratch():
    torch = torch_cuda()
    ff = lib_ready()
    x = torch.zeros(8, 16, dtype=torch.bfloat16, device="cuda")
    s = torch.ones(8, device="cuda")
    W = torch.zeros(8, 16, dtype=torch.bfloat16, device="cuda")
    h = torch.zeros(8, 8, dtype=torch.bfloat16, device="cuda")
    # rows * ceil(out / 256) beyond the 4 MiB scratch: rejected on the host, nothing enqueued
    st = ff.lib().ff_forward_noalloc(x.data_ptr(), s.data_ptr(), W.data_ptr(), None, 1 << 21, 16, 8,
                                     h.data_ptr(), None, None, None, None)
    assert st == 1
