"""Synthetic scheduling workloads and seeded random instance recipes.

This module only describes INPUTS: the five scheduling batches (layer shape
tables of standard CNNs and the distributions of device rate, link bandwidth
and per-segment latency) and numpy recipes for random test instances. It holds
none of the scheduling arithmetic and is shared by the tests, the benchmark and
the oracle-side checks.

The paper profiles VGG-19, GoogLeNet, Inception-v4 and ResNet-152 on ILSVRC12
(Sec. V-A2). Those measured profiles are not available here; the batches below
stand in for them with cost vectors derived from standard layer shapes, and
every instance draws its own device speed, bandwidth and latency.

Layer decomposition follows Sec. III-A: every layer with parameters is one
schedulable layer; parameter-free operations (pooling, flatten, ReLU) are part
of the compute of the layer before them. Per-layer FLOPs = 2 * MACs * batch.
"""
from __future__ import annotations

import numpy as np

# Enum values of the profile-generator config (same numbers in include/dynacomm.h).
LAYERS_FIXED, LAYERS_UNIFORM, LAYERS_LOGUNIFORM = 0, 1, 2
DIST_UNIFORM, DIST_LOGUNIFORM = 0, 1


def _conv(cin: int, cout: int, k: int, hw_out: int, bias: bool = True, bn: bool = False):
    params = cout * cin * k * k + (cout if bias else 0) + (2 * cout if bn else 0)
    macs = hw_out * hw_out * cout * cin * k * k
    return params, macs


def _fc(cin: int, cout: int):
    return cin * cout + cout, cin * cout


def alexnet_layers():
    """AlexNet, single-tower (torchvision) layout at 224x224: 5 conv + 3 fc."""
    return [
        _conv(3, 64, 11, 55), _conv(64, 192, 5, 27), _conv(192, 384, 3, 13),
        _conv(384, 256, 3, 13), _conv(256, 256, 3, 13),
        _fc(256 * 6 * 6, 4096), _fc(4096, 4096), _fc(4096, 1000),
    ]


def vgg16_layers():
    """VGG-16 (configuration D) at 224x224: 13 conv + 3 fc."""
    spec = [(3, 64, 224), (64, 64, 224), (64, 128, 112), (128, 128, 112),
            (128, 256, 56), (256, 256, 56), (256, 256, 56),
            (256, 512, 28), (512, 512, 28), (512, 512, 28),
            (512, 512, 14), (512, 512, 14), (512, 512, 14)]
    layers = [_conv(ci, co, 3, hw) for ci, co, hw in spec]
    return layers + [_fc(512 * 7 * 7, 4096), _fc(4096, 4096), _fc(4096, 1000)]


def resnet50_layers():
    """ResNet-50 v1.5 at 224x224: 53 conv (BN folded into each conv's
    parameters) + 1 fc. Each bottleneck is 1x1 -> 3x3 (carrying the stride) ->
    1x1; the downsample 1x1 of a stage's first block is its own layer, placed
    after that block's last 1x1."""
    layers = [_conv(3, 64, 7, 112, bias=False, bn=True)]
    cin, hw = 64, 56
    for width, blocks, stride in ((64, 3, 1), (128, 4, 2), (256, 6, 2), (512, 3, 2)):
        for b in range(blocks):
            s = stride if b == 0 else 1
            hw_out = hw // s
            layers.append(_conv(cin, width, 1, hw, bias=False, bn=True))
            layers.append(_conv(width, width, 3, hw_out, bias=False, bn=True))
            layers.append(_conv(width, 4 * width, 1, hw_out, bias=False, bn=True))
            if b == 0:
                layers.append(_conv(cin, 4 * width, 1, hw_out, bias=False, bn=True))
            cin, hw = 4 * width, hw_out
    layers.append(_fc(2048, 1000))
    return layers


def _fixed(layers, batch_size: int):
    params = np.array([p for p, _ in layers], dtype=np.int64)
    flops = np.array([2 * m * batch_size for _, m in layers], dtype=np.int64)
    return params, flops


def _cfg(name, L, batch, seed, **kw):
    base = dict(name=name, L=L, batch=batch, seed=seed, inst0=0, bwd_flops_mult=2,
                bits_per_param=32, params_lo=0, params_hi=0, flops_lo=0, flops_hi=0)
    base.update(kw)
    return base


def config(name: str) -> dict:
    """The five batches. Units: rate FLOP/us (1 GFLOP/s = 1000), bandwidth kbit/s
    (1 Mbps = 1000), latency us. Backward compute = 2x forward FLOPs; the gradient
    of a layer has its parameter tensor's size, so gt = pt."""
    if name == "tiny":
        return _cfg("tiny", 8, 4096, 0, layer_mode=LAYERS_UNIFORM,
                    params_lo=1_000, params_hi=1_000_000,
                    flops_lo=1_000_000, flops_hi=1_000_000_000,
                    rate_dist=DIST_UNIFORM, rate_lo=10_000, rate_hi=100_000,
                    bw_dist=DIST_LOGUNIFORM, bw_lo=1_000, bw_hi=100_000,
                    dt_lo=1_000, dt_hi=50_000)
    shared = dict(rate_dist=DIST_LOGUNIFORM, rate_lo=5_000, rate_hi=200_000,
                  bw_dist=DIST_LOGUNIFORM, bw_lo=1_000, bw_hi=1_000_000,
                  dt_lo=1_000, dt_hi=100_000)
    if name in ("alexnet", "vgg16", "resnet50"):
        layers, bs, batch, seed = {
            "alexnet": (alexnet_layers(), 32, 1_000_000, 1),
            "vgg16": (vgg16_layers(), 16, 1_000_000, 2),
            "resnet50": (resnet50_layers(), 32, 262_144, 3),
        }[name]
        params, flops = _fixed(layers, bs)
        return _cfg(name, len(layers), batch, seed, layer_mode=LAYERS_FIXED,
                    fixed_params=params, fixed_flops=flops, model_batch=bs, **shared)
    if name == "deepchain":
        return _cfg("deepchain", 1024, 16_384, 4, layer_mode=LAYERS_LOGUNIFORM,
                    params_lo=1_000, params_hi=10_000_000,
                    flops_lo=1_000_000, flops_hi=10_000_000_000, **shared)
    raise KeyError(name)


CONFIG_NAMES = ("tiny", "alexnet", "vgg16", "resnet50", "deepchain")

# Depths of the scheduling-time-versus-L sweep (the paper's Fig. 12 times its
# schedulers on randomly generated profiles of growing depth).
LSWEEP_LS = (8, 16, 32, 64, 128, 256, 512, 1024, 2048)


def lsweep_config(L: int, batch: int, seed: int = 5) -> dict:
    """The deep-chain draws (per-instance log-uniform params and FLOPs per layer,
    per-instance rate, bandwidth and latency) at depth L."""
    c = config("deepchain")
    c.update(name=f"lsweep{L}", L=int(L), batch=int(batch), seed=int(seed))
    return c


def with_batch(cfg: dict, batch: int, inst0: int = 0) -> dict:
    c = dict(cfg)
    c["batch"] = int(batch)
    c["inst0"] = int(inst0)
    return c


def shard_range(batch: int, rank: int, world: int):
    """Contiguous instance range [lo, hi) of `rank` among `world` equal shares."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("bad rank/world")
    return batch * rank // world, batch * (rank + 1) // world


def random_instances(seed: int, batch: int, L: int, lo: int = 0, hi: int = 1000,
                     dt_lo: int = 0, dt_hi: int = 1000):
    """Uniform integer costs: (comp [batch, L], xfer [batch, L], dt [batch])."""
    rng = np.random.default_rng(seed)
    comp = rng.integers(lo, hi + 1, size=(batch, L), dtype=np.int64)
    xfer = rng.integers(lo, hi + 1, size=(batch, L), dtype=np.int64)
    dt = rng.integers(dt_lo, dt_hi + 1, size=batch, dtype=np.int64)
    return comp, xfer, dt


def tie_heavy_instances(seed: int, batch: int, L: int):
    """Tiny value ranges so that equal candidates (ties in k and in n) are common."""
    return random_instances(seed, batch, L, 0, 3, 0, 3)


def skewed_instances(seed: int, batch: int, L: int):
    """Per-instance log-scale costs spanning several decades, with some zeros."""
    rng = np.random.default_rng(seed)
    scale_c = 10.0 ** rng.uniform(0, 6, size=(batch, 1))
    scale_x = 10.0 ** rng.uniform(0, 6, size=(batch, 1))
    comp = np.floor(scale_c * rng.random((batch, L)) ** 3).astype(np.int64)
    xfer = np.floor(scale_x * rng.random((batch, L)) ** 3).astype(np.int64)
    dt = np.floor(10.0 ** rng.uniform(0, 5, size=batch)).astype(np.int64)
    return comp, xfer, dt


def random_decisions(seed: int, batch: int, L: int, density: float = 0.5) -> np.ndarray:
    """Random packed decision words [batch, ceil((L-1)/32)] with bits 0..L-2 only."""
    W = (L - 1 + 31) // 32
    rng = np.random.default_rng(seed)
    dense = (rng.random((batch, max(L - 1, 0))) < density).astype(np.uint64)
    out = np.zeros((batch, W), dtype=np.uint32)
    for l in range(L - 1):
        out[:, l // 32] |= (dense[:, l] << np.uint64(l % 32)).astype(np.uint32)
    return out
