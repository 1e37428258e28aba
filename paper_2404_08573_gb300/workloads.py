"""Named workloads of the FF method (shapes, batch, hyper-parameters).

Each is a plain description used by the benchmark and available to users;
the shapes follow the paper's MNIST net (§5: 784 inputs, four hidden layers
of 2000 ReLUs) and its larger variants.  Nothing here computes anything.
"""

from __future__ import annotations

from dataclasses import dataclass
from typing import Tuple


@dataclass(frozen=True)
class Workload:
    name: str
    net: Tuple[int, ...]   # layer widths, input first
    prec: str              # "bf16" (bf16 operands, fp32 accumulate) or "fp32"
    batch_pairs: int       # positive/negative pairs per train step
    pairs: int             # pairs per epoch (train) or samples (predict)
    theta: float           # goodness threshold of Eq. 1
    lr: float              # Adam learning rate of the FF layers
    streams: int = 1       # layer streams (the one-GPU pipeline of §4)


WORKLOADS = {
    w.name: w
    for w in (
        Workload("ff_train_784-500-500_fp32_B64", (784, 500, 500), "fp32", 64, 64 * 16, 2.0, 0.03),
        Workload("ff_train_784-2000x4_bf16_epoch60000_B1024", (784, 2000, 2000, 2000, 2000), "bf16", 1024, 60000,
                 2.0, 0.03, streams=4),
        Workload("ff_predict_784-2000x4_n10000", (784, 2000, 2000, 2000, 2000), "bf16", 0, 10000, 2.0, 0.03),
        Workload("ff_train_784-2000x5_bf16_5streams_60x1000", (784, 2000, 2000, 2000, 2000, 2000), "bf16", 1000,
                 60000, 2.0, 0.03, streams=5),
        Workload("ff_train_3072-8192x4_bf16_B4096_theta8", (3072, 8192, 8192, 8192, 8192), "bf16", 4096, 4096, 8.0,
                 0.03),
    )
}
