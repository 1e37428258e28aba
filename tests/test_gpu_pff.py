"""Chapter schedule of §4 (Single-Layer and All-Layers PFF) on the GPU:
against the oracle's schedule, between its two stream assignments, and
against the same steps issued one call at a time through the layer API."""

import numpy as np
import pytest

from oracle import ff_oracle as fo
from paper_2404_08573_gb300 import synth

from .gpu_common import lib_ready, rel_norm, torch_cuda

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    torch = torch_cuda()
    ff = lib_ready()
    return torch, ff


def _data(P, B, S, seed, features=784):
    """Batch-major pairs and per-chapter labels (fresh negatives per chapter)."""
    x = synth.mnist_like(P, seed=seed, features=features)
    y = synth.labels(P, seed=seed)
    xs, labs = [], []
    for r0, b in fo.pair_batches(P, B):
        s0 = r0 // 2
        x2, _ = synth.pair_batch(x[s0:s0 + b], y[s0:s0 + b], y[s0:s0 + b])
        xs.append(x2)
    for c in range(S):
        lc = []
        for r0, b in fo.pair_batches(P, B):
            s0 = r0 // 2
            yn = synth.negative_labels(y[s0:s0 + b], seed=seed, start=c * P + s0)
            lc.append(np.concatenate([y[s0:s0 + b], yn]).astype(np.int32))
        labs.append(np.concatenate(lc))
    return np.concatenate(xs), np.stack(labs)


def _layers(ff, dims, prec, seed, lr=0.03, theta=2.0, max_rows=0):
    return [ff.Layer(dims[i], dims[i + 1], prec=prec, init_seed=seed + i, lr=lr, theta=theta, max_rows=max_rows)
            for i in range(len(dims) - 1)]


def _states(layers):
    return [l.get_state() for l in layers]


def test_pff_modes_and_host_loop_are_bitwise_equal(env):
    torch, ff = env
    dims, P, B, C, S = (784, 96, 64, 48), 200, 64, 2, 3
    x, labs = _data(P, B, S, seed=11)
    xg, lg = torch.from_numpy(x).cuda(), torch.from_numpy(labs).cuda()
    nb = len(fo.pair_batches(P, B))
    results = {}
    for mode, nodes in (("single_layer", 1), ("all_layers", 2), ("all_layers", 3)):
        layers = _layers(ff, dims, "bf16", seed=20, max_rows=2 * B)
        pff = ff.Pff(layers, P, B, C, S, mode=mode, nodes=nodes)
        loss = torch.zeros(S, len(layers), C * nb, device="cuda")
        pff.run(xg, lg, 0, S, loss=loss)
        torch.cuda.synchronize()
        for l in layers:
            l.check()
        results[(mode, nodes)] = (_states(layers), loss.cpu().numpy())
        pff.close()
    # the same steps, one API call at a time on one stream, chapter by chapter
    layers = _layers(ff, dims, "bf16", seed=20, max_rows=2 * B)
    loss = torch.zeros(S, len(layers), C * nb, device="cuda")
    for c in range(S):
        inp, scale = None, None
        for i, l in enumerate(layers):
            for m in range(C):
                for j, (r0, b) in enumerate(fo.pair_batches(P, B)):
                    if i == 0:
                        l.train_step(xg[r0:r0 + 2 * b], labels=lg[c, r0:r0 + 2 * b], B=b, loss=loss[c, i, m * nb + j])
                    else:
                        l.train_step(inp[r0:r0 + 2 * b], row_scale=scale[r0:r0 + 2 * b], B=b,
                                     loss=loss[c, i, m * nb + j])
            if i + 1 < len(layers):
                out = l.new_activation(2 * P)
                sn = torch.empty(2 * P, device="cuda")
                for r0, b in fo.pair_batches(P, B):
                    if i == 0:
                        l.forward(xg[r0:r0 + 2 * b], labels=lg[c, r0:r0 + 2 * b], h_out=out[r0:r0 + 2 * b],
                                  next_scale=sn[r0:r0 + 2 * b])
                    else:
                        l.forward(inp[r0:r0 + 2 * b], row_scale=scale[r0:r0 + 2 * b], h_out=out[r0:r0 + 2 * b],
                                  next_scale=sn[r0:r0 + 2 * b])
                inp, scale = out, sn
    torch.cuda.synchronize()
    ref_states, ref_loss = _states(layers), loss.cpu().numpy()
    for key, (st, ls) in results.items():
        assert np.array_equal(ls, ref_loss), key
        for a, b in zip(st, ref_states):
            for name in ("W", "b", "mW", "vW"):
                assert np.array_equal(a[name], b[name]), (key, name)
            assert a["t"] == b["t"] == S * C * nb


def test_pff_chapters_in_several_calls_equal_one_call(env):
    torch, ff = env
    dims, P, B, C, S = (784, 64, 32), 96, 32, 1, 4
    x, labs = _data(P, B, S, seed=12)
    xg, lg = torch.from_numpy(x).cuda(), torch.from_numpy(labs).cuda()
    a = _layers(ff, dims, "bf16", seed=30, max_rows=2 * B)
    pa = ff.Pff(a, P, B, C, S, cooldown_start=0.5)
    pa.run(xg, lg, 0, S)
    b = _layers(ff, dims, "bf16", seed=30, max_rows=2 * B)
    pb = ff.Pff(b, P, B, C, S, cooldown_start=0.5)
    pb.run(xg, lg[0:1], 0, 1)
    pb.run(xg, lg[1:3], 1, 2)
    pb.run(xg, lg[3:4], 3, 1)
    torch.cuda.synchronize()
    for la, lb in zip(a, b):
        sa, sb = la.get_state(), lb.get_state()
        assert np.array_equal(sa["W"], sb["W"]) and np.array_equal(sa["vW"], sb["vW"])


def test_pff_matches_oracle_schedule_fp32(env):
    """fp32, 2 chapters x 2 epochs x 3 batches, lr cooldown from half way:
    every step's loss and the final weights against the oracle's schedule."""
    torch, ff = env
    dims, P, B, C, S, theta, lr = (784, 48, 32), 48, 16, 2, 2, 2.0, 1e-3
    x, labs = _data(P, B, S, seed=13)
    layers = _layers(ff, dims, "fp32", seed=40, lr=lr, theta=theta, max_rows=2 * B)
    states = [fo.LayerState(l.get_state()["W"], l.get_state()["b"]) for l in layers]
    pff = ff.Pff(layers, P, B, C, S, cooldown_start=0.5)
    nb = len(fo.pair_batches(P, B))
    loss = torch.zeros(S, len(layers), C * nb, device="cuda")
    pff.run(torch.from_numpy(x).cuda(), torch.from_numpy(labs).cuda(), 0, S, loss=loss)
    torch.cuda.synchronize()
    ref_loss = fo.chapter_schedule(states, x, labs, B, C, theta, fo.AdamHyper(lr=lr), cooldown_start=0.5)
    got = loss.cpu().numpy()
    assert np.all(np.abs(got - ref_loss) <= 1e-4 * np.abs(ref_loss) + 1e-6), float(np.max(np.abs(got - ref_loss)))
    for l, st in zip(layers, states):
        g = l.get_state()
        assert g["t"] == st.t == S * C * nb
        assert rel_norm(g["W"], st.W) < 1e-4, rel_norm(g["W"], st.W)
        assert rel_norm(g["b"], st.b) < 1e-3, rel_norm(g["b"], st.b)


def test_pff_argument_errors(env):
    torch, ff = env
    layers = _layers(ff, (784, 32, 16), "bf16", seed=50)
    with pytest.raises(ff.FFError):
        ff.Pff(layers, 0, 16, 1, 1)
    with pytest.raises(ff.FFError):
        ff.Pff([layers[1], layers[0]], 16, 16, 1, 1)     # not a chain
    with pytest.raises(ff.FFError):
        ff.Pff(layers, 16, 16, 1, 2, mode="all_layers", nodes=0)
    p = ff.Pff(layers, 16, 16, 1, 2)
    x = torch.zeros(32, 784, device="cuda")
    lab = torch.zeros(2, 32, dtype=torch.int32, device="cuda")
    with pytest.raises(ff.FFError):
        p.run(x, lab, 1, 2)                               # past the last chapter
    p.run(x, lab, 0, 0)                                   # nothing to do
