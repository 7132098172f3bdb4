"""Seeded synthetic gradient workloads for the gs-SGD compression step.

This module only makes inputs: the five workload configurations, the parameter-block
sizes of the networks whose gradients they imitate, and seeded per-(step, worker)
gradient vectors.  It holds none of the compression method's arithmetic, and both the CPU
oracle and the GPU library are fed from it.

The paper trains ResNet-20 and VGG-16 on CIFAR-10 (Sec. IV); neither the dataset nor
trained weights are needed here.  Synthetic gradients with the block structure of real
networks stand in for them: every parameter block draws its own scale once per
configuration, and entries are i.i.d. within a block.
"""

from .blocks import (  # noqa: F401
    resnet18_cifar_blocks,
    resnet50_imagenet_blocks,
    vgg16_imagenet_blocks,
    bert_large_blocks,
)
from .configs import CONFIGS, Workload, get_config  # noqa: F401
from .gradients import (  # noqa: F401
    BASE_SEED,
    block_scales,
    spike_positions,
    make_gradient,
    make_gradients,
    make_gradient_torch,
    torch_seed,
)
