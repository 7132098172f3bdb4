"""Parameter-block sizes of four networks, derived from their architecture rules.

Each function returns the list of parameter-tensor sizes in registration order (weights
and biases are separate blocks, batch-norm scale and shift are separate blocks).
"""

from __future__ import annotations


def resnet18_cifar_blocks() -> list[int]:
    """ResNet-18, CIFAR variant: 3x3 stem (64, no bias) + BN, four stages of two basic
    blocks (widths 64/128/256/512, stride 2 at stages 2-4), 1x1 projection shortcut + BN
    where the shape changes, and a 512x10 linear head with bias.  62 blocks, 11,173,962
    parameters."""
    blocks = [3 * 64 * 9, 64, 64]
    cin = 64
    for width, stride in ((64, 1), (128, 2), (256, 2), (512, 2)):
        for b in range(2):
            s = stride if b == 0 else 1
            blocks += [cin * width * 9, width, width, width * width * 9, width, width]
            if s != 1 or cin != width:
                blocks += [cin * width, width, width]
            cin = width
    blocks += [512 * 10, 10]
    return blocks


def resnet50_imagenet_blocks() -> list[int]:
    """ResNet-50 (ImageNet): 7x7 stem (64, no bias) + BN, bottleneck stages [3, 4, 6, 3]
    with widths 64/128/256/512 and expansion 4 (1x1, 3x3, 1x1 convs, each with BN), a 1x1
    projection + BN on each stage's first block, and a 2048x1000 linear head with bias.
    161 blocks, 25,557,032 parameters."""
    blocks = [3 * 64 * 49, 64, 64]
    cin = 64
    for width, n in ((64, 3), (128, 4), (256, 6), (512, 3)):
        out = 4 * width
        for b in range(n):
            blocks += [cin * width, width, width,
                       width * width * 9, width, width,
                       width * out, out, out]
            if b == 0:
                blocks += [cin * out, out, out]
            cin = out
    blocks += [2048 * 1000, 1000]
    return blocks


def vgg16_imagenet_blocks() -> list[int]:
    """VGG-16 (ImageNet): 13 3x3 convs with bias (64,64 | 128,128 | 256x3 | 512x3 | 512x3)
    and three linear layers 25088->4096->4096->1000 with bias.  32 blocks, 138,357,544
    parameters."""
    widths = [64, 64, 128, 128, 256, 256, 256, 512, 512, 512, 512, 512, 512]
    blocks = []
    cin = 3
    for w in widths:
        blocks += [cin * w * 9, w]
        cin = w
    for fin, fout in ((512 * 7 * 7, 4096), (4096, 4096), (4096, 1000)):
        blocks += [fin * fout, fout]
    return blocks


def bert_large_blocks() -> list[int]:
    """BERT-large as the workload states it: a 30522x1024 token-embedding block, then 24
    layers of four 1024x1024 attention projections and a 1024x4096 / 4096x1024 FFN pair.
    145 blocks, 333,244,416 parameters."""
    hidden, ffn, vocab, layers = 1024, 4096, 30522, 24
    blocks = [vocab * hidden]
    for _ in range(layers):
        blocks += [hidden * hidden] * 4
        blocks += [hidden * ffn, ffn * hidden]
    return blocks
