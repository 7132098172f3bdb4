"""The five workload configurations of the compression step.

Each gives the gradient length d, the number of simulated workers P, the sketch shape
r x c, the number k of selected coordinates, the number of steps, and the recipe of the
synthetic gradient entries.
"""

from __future__ import annotations

import dataclasses

from . import blocks as _blocks


@dataclasses.dataclass(frozen=True)
class Workload:
    cid: int                 # configuration number, used in the seeds
    name: str
    d: int
    P: int
    r: int
    c: int
    k: int
    steps: int
    dist: str                # "normal" or "laplace"
    scale_lo: float          # per-block scale drawn log-uniform in [scale_lo, scale_hi]
    scale_hi: float
    spike_frac: float        # fraction of coordinates carrying a spike (0 = none)
    spike_mag: float
    block_sizes: tuple = ()  # empty = a single block of length d
    worker_batch: int = 0    # workers resident at a time (0 = all P)
    rho: float = 0.9

    @property
    def blocks(self) -> list[int]:
        return list(self.block_sizes) if self.block_sizes else [self.d]


def _mk():
    r18 = tuple(_blocks.resnet18_cifar_blocks())
    r50 = tuple(_blocks.resnet50_imagenet_blocks())
    vgg = tuple(_blocks.vgg16_imagenet_blocks())
    bert = tuple(_blocks.bert_large_blocks())
    return {
        # d = 2^20, P = 4, N(0, 1e-4^2) plus 0.5 % spikes of magnitude 1e-2, random sign
        "tiny-2^20": Workload(0, "tiny-2^20", 1 << 20, 4, 5, 1 << 14, 1000, 3, "normal",
                              1e-4, 1e-4, 0.005, 1e-2),
        # ResNet-18 sized, 62 blocks with N(0, s_l^2), s_l log-uniform in [1e-5, 1e-2]
        "resnet18": Workload(1, "resnet18", sum(r18), 8, 5, 1 << 17, 11200, 10, "normal",
                             1e-5, 1e-2, 0.0, 0.0, r18),
        # ResNet-50 sized, 161 blocks with Laplace(0, b_l), b_l log-uniform in [1e-5, 1e-2]
        "resnet50": Workload(2, "resnet50", sum(r50), 8, 5, 1 << 18, 25600, 10, "laplace",
                             1e-5, 1e-2, 0.0, 0.0, r50),
        # VGG-16 sized, 32 blocks with N(0, s_l^2), s_l in [1e-6, 1e-3], plus 0.1 % spikes
        "vgg16": Workload(3, "vgg16", sum(vgg), 16, 7, 1 << 20, 138000, 5, "normal",
                          1e-6, 1e-3, 0.001, 1e-2, vgg),
        # BERT-large sized, 145 blocks with N(0, s_l^2), s_l in [1e-6, 1e-3], P = 32 in
        # batches of 8 resident workers
        "bert-large": Workload(4, "bert-large", sum(bert), 32, 5, 1 << 21, 340000, 3,
                               "normal", 1e-6, 1e-3, 0.0, 0.0, bert, worker_batch=8),
    }


CONFIGS = _mk()


def get_config(name: str) -> Workload:
    return CONFIGS[name]
