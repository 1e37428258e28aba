"""End to end: FF training in bf16-operand mode (fp32 accumulate and master
weights) on the learnable synthetic task reaches, after the whole schedule,
the oracle's fp64 accuracy within 0.5 points.

The run is the chapter schedule of §4 (Single-Layer PFF: 4 chapters of 2
epochs per layer) with the learning rate cooled linearly to 0 over each
layer's second half of epochs (§5.1), on 784-500-500 with 4096 training pairs
of 128 per batch; accuracy is goodness prediction (§3, layer 2's goodness)
on 10 000 held-out samples of the same task.  The task's class signal is
weakened (a nonzero feature lands on its class support with probability
0.15) so that the accuracy settles near 0.89 rather than at 1."""

import numpy as np
import pytest

from oracle import ff_oracle as fo
from paper_2404_08573_gb300 import synth

from .gpu_common import lib_ready, torch_cuda

pytestmark = pytest.mark.gpu

DIMS, P, B, C, S = (784, 500, 500), 4096, 128, 2, 4
LR, THETA, COOL, ON_SUPPORT, SEED, N_EVAL = 0.003, 2.0, 0.5, 0.15, 5, 10000


def _data():
    """Batch-major training pairs, per-chapter labels (fresh negatives per
    chapter) and the held-out set."""
    x, y = synth.learnable_task(P, seed=SEED, on_support=ON_SUPPORT)
    xs, labs = [], []
    for r0, b in fo.pair_batches(P, B):
        s0 = r0 // 2
        x2, _ = synth.pair_batch(x[s0:s0 + b], y[s0:s0 + b], y[s0:s0 + b])
        xs.append(x2)
    for c in range(S):
        lc = []
        for r0, b in fo.pair_batches(P, B):
            s0 = r0 // 2
            yn = synth.negative_labels(y[s0:s0 + b], seed=SEED, start=c * P + s0)
            lc.append(np.concatenate([y[s0:s0 + b], yn]).astype(np.int32))
        labs.append(np.concatenate(lc))
    xe, ye = synth.learnable_task(N_EVAL, seed=SEED, start_row=200000, on_support=ON_SUPPORT)
    return np.concatenate(xs), np.stack(labs), xe, ye


def test_bf16_training_reaches_the_oracle_accuracy():
    torch = torch_cuda()
    ff = lib_ready()
    x, labs, xe, ye = _data()
    W0 = [synth.he_uniform(100 + k, DIMS[k + 1], DIMS[k]) for k in range(len(DIMS) - 1)]
    # oracle, fp64
    states = [fo.LayerState(W0[k], np.zeros(DIMS[k + 1], np.float32)) for k in range(len(DIMS) - 1)]
    fo.chapter_schedule(states, x, labs, B, C, THETA, fo.AdamHyper(lr=LR), cooldown_start=COOL)
    pred_ref, _ = fo.predict(states, xe)
    acc_ref = float(np.mean(pred_ref == ye))
    # GPU, bf16 operands
    layers = [ff.Layer(DIMS[k], DIMS[k + 1], prec="bf16", lr=LR, theta=THETA, max_rows=2 * B)
              for k in range(len(DIMS) - 1)]
    for k, l in enumerate(layers):
        l.set_state(W=W0[k], b=np.zeros(DIMS[k + 1], np.float32))
    pff = ff.Pff(layers, P, B, C, S, mode="single_layer", nodes=1, cooldown_start=COOL)
    pff.run(torch.from_numpy(x).cuda(), torch.from_numpy(labs).cuda(), 0, S)
    torch.cuda.synchronize()
    pff.close()
    for l in layers:
        l.check()
    pred, _ = ff.predict(layers, torch.from_numpy(xe).cuda())
    torch.cuda.synchronize()
    acc = float(np.mean(pred.cpu().numpy() == ye))
    print(f"final accuracy: GPU bf16 {acc:.4f}, oracle fp64 {acc_ref:.4f}")
    assert acc_ref > 0.8, acc_ref                  # the task is learned
    assert abs(acc - acc_ref) <= 0.005, (acc, acc_ref)
