"""The synthetic workloads: block structure derived from the architectures, seeding."""

import numpy as np

import workloads as W


def test_block_totals_from_architecture_rules():
    assert (len(W.resnet18_cifar_blocks()), sum(W.resnet18_cifar_blocks())) == (62, 11_173_962)
    assert (len(W.resnet50_imagenet_blocks()), sum(W.resnet50_imagenet_blocks())) == (161, 25_557_032)
    assert (len(W.vgg16_imagenet_blocks()), sum(W.vgg16_imagenet_blocks())) == (32, 138_357_544)
    assert (len(W.bert_large_blocks()), sum(W.bert_large_blocks())) == (145, 333_244_416)
    fc = sorted(W.vgg16_imagenet_blocks())[-3:]
    assert fc == [4_096_000, 16_777_216, 102_760_448]


def test_config_shapes():
    c = W.CONFIGS
    assert [(w.d, w.P, w.r, w.c, w.k, w.steps) for w in c.values()] == [
        (1 << 20, 4, 5, 1 << 14, 1000, 3),
        (11_173_962, 8, 5, 1 << 17, 11200, 10),
        (25_557_032, 8, 5, 1 << 18, 25600, 10),
        (138_357_544, 16, 7, 1 << 20, 138000, 5),
        (333_244_416, 32, 5, 1 << 21, 340000, 3),
    ]


def test_gradients_seeded_and_prefix_consistent():
    w = W.get_config("resnet18")
    a = W.make_gradient(w, 2, 3, d=300_000)
    b = W.make_gradient(w, 2, 3, d=300_000)
    assert np.array_equal(a, b) and a.dtype == np.float32
    assert not np.array_equal(a, W.make_gradient(w, 2, 4, d=300_000))
    assert np.array_equal(W.make_gradient(w, 2, 3, d=1000), a[:1000])
    lap = W.get_config("resnet50")
    x = W.make_gradient(lap, 0, 0, d=200_000)
    assert np.array_equal(W.make_gradient(lap, 0, 0, d=5000), x[:5000])
    scales = W.block_scales(lap)
    assert scales.min() >= 1e-5 and scales.max() <= 1e-2


def test_spikes_shared_across_workers():
    w = W.get_config("tiny-2^20")
    pos, sgn = W.spike_positions(w)
    assert pos.size == round(0.005 * w.d) and np.all(np.diff(pos) > 0)
    g0 = W.make_gradient(w, 0, 0)
    g1 = W.make_gradient(w, 1, 3)
    assert np.all(np.sign(g0[pos]) == sgn) and np.all(np.sign(g1[pos]) == sgn)


def test_device_draw_follows_the_block_recipe():
    """The device-side draw (here on the CPU generator): seeded per (step, worker), and each
    block's entries have the block's scale."""
    import torch
    w = W.get_config("resnet18")
    a = W.make_gradient_torch(w, 1, 2, torch.empty(w.d))
    b = W.make_gradient_torch(w, 1, 2, torch.empty(w.d))
    c = W.make_gradient_torch(w, 1, 3, torch.empty(w.d))
    assert torch.equal(a, b) and not torch.equal(a, c)
    x = a.numpy().astype(np.float64)
    off = 0
    for n, s in zip(w.blocks, W.block_scales(w)):
        if n >= 20_000:
            sd = x[off:off + n].std()
            assert abs(sd / s - 1) < 0.05, (n, s, sd)
            assert abs(x[off:off + n].mean()) < 5 * s / np.sqrt(n)
        off += n
    assert off == w.d
