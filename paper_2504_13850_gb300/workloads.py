"""Workload definitions and seeded synthetic inputs.

This module holds only the *inputs* of the server-side hot path: the
server-part architectures (as op lists), their batch shapes, queue sizes and
step counts, and seeded generators for initial weights, uploaded activation
batches, labels, sequence lengths, device-side models and device arrival
orders.  It contains none of the method's arithmetic, so both the CUDA path
and the CPU oracle may consume it.

The architectures stand in for the paper's workloads (Sec. 5.2, Table 4:
VGG-style CNNs on CIFAR-10-shaped data, ResNet-18 stages, transformer
encoders on SST-2/IMDB-shaped sequences, the MobileNetV3-Large server part
on Tiny-ImageNet-shaped activations).  No dataset item is used: every
activation is drawn from a PCG64 generator.

Op list format (one dict per op, executed in order).  Tensor 0 is the
uploaded activation batch; op ``i`` (0-based) produces tensor ``i + 1``.

  conv      in0, cin, cout, k (1 or 3), stride (1 or 2), bias (0/1); pad = k // 2
            params: W[cout][k][k][cin], then b[cout] if bias
  affine    in0, c                       params: scale[c], shift[c]
  relu      in0
  maxpool2  in0                          2x2 window, stride 2
  add       in0, in1
  avgpool   in0                          global mean over H, W
  flatten   in0                          [B,H,W,C] -> [B, H*W*C] (h, w, c order)
  linear    in0, cin, cout, bias         params: W[cout][cin], then b[cout]
  layernorm in0, c                       params: gamma[c], beta[c]; eps 1e-5
  gelu      in0                          exact (erf) GELU
  attention in0, c, heads                in0 is [B, L, 3c] = q | k | v
  meanpool  in0                          mean over the valid tokens of each row
  dwconv    in0, c, k (odd), stride, bias  depthwise k x k, pad k // 2
            params: W[c][k][k], then b[c] if bias
  hswish    in0                          hard swish x * relu6(x + 3) / 6
  hsigmoid  in0                          hard sigmoid relu6(x + 3) / 6
  chmul     in0, in1                     y[b,h,w,c] = in0[b,h,w,c] * in1[b,c] (squeeze-and-excite)

Activations are NHWC.  A sequence batch [B, L, d] is carried as H = L,
W = 1, C = d.  The last op's output is the logits [B, classes]; the loss is
softmax cross-entropy averaged over the batch.
"""
from __future__ import annotations

import numpy as np

F32 = "f32"
BF16 = "bf16"


# --------------------------------------------------------------------------
# architectures
# --------------------------------------------------------------------------

class _Builder:
    def __init__(self):
        self.ops = []

    def add(self, kind, in0, **kw):
        op = {"kind": kind, "in0": int(in0)}
        op.update(kw)
        self.ops.append(op)
        return len(self.ops)          # id of the tensor this op produces


def tiny_cnn_ops():
    """conv3x3 32->64 pad 1 + ReLU + maxpool 2 + FC 64*8*8 -> 10."""
    b = _Builder()
    t = b.add("conv", 0, cin=32, cout=64, k=3, stride=1, bias=1)
    t = b.add("relu", t)
    t = b.add("maxpool2", t)
    t = b.add("flatten", t)
    b.add("linear", t, cin=64 * 8 * 8, cout=10, bias=1)
    return b.ops


def vgg_ops():
    """2x(conv3x3 ->256, ReLU), pool, 2x(conv3x3 ->512, ReLU), pool,
    FC 512*4*4 -> 512, ReLU, FC 512 -> 10, on a [16,16,128] input."""
    b = _Builder()
    t = 0
    for cin, cout in ((128, 256), (256, 256)):
        t = b.add("conv", t, cin=cin, cout=cout, k=3, stride=1, bias=1)
        t = b.add("relu", t)
    t = b.add("maxpool2", t)
    for cin, cout in ((256, 512), (512, 512)):
        t = b.add("conv", t, cin=cin, cout=cout, k=3, stride=1, bias=1)
        t = b.add("relu", t)
    t = b.add("maxpool2", t)
    t = b.add("flatten", t)
    t = b.add("linear", t, cin=512 * 4 * 4, cout=512, bias=1)
    t = b.add("relu", t)
    b.add("linear", t, cin=512, cout=10, bias=1)
    return b.ops


def vgg_device_ops():
    """A device's network for the VGG-style split (Alg. 1): M_dk = conv3x3
    3->128 + ReLU + maxpool 2 on a [32,32,3] image, whose [16,16,128] output
    (tensor 3) is the activation uploaded to the server; then the default
    auxiliary network (one layer of the same type as M_dk's last layer and a
    dense classifier): conv3x3 128->128 + ReLU, global average pool,
    FC 128 -> 10."""
    b = _Builder()
    t = b.add("conv", 0, cin=3, cout=128, k=3, stride=1, bias=1)
    t = b.add("relu", t)
    t = b.add("maxpool2", t)
    t = b.add("conv", t, cin=128, cout=128, k=3, stride=1, bias=1)
    t = b.add("relu", t)
    t = b.add("avgpool", t)
    b.add("linear", t, cin=128, cout=10, bias=1)
    return b.ops


VGG_DEVICE_SPLIT = 3      # tensor id of M_dk's output in vgg_device_ops()


def _bneck(b, x, cin, exp, cout, k, stride, se=True, act="hswish"):
    """MobileNetV3 bottleneck: 1x1 expansion, k x k depthwise (stride),
    squeeze-and-excite, 1x1 projection; batch norms folded to affines;
    residual when the shape is kept."""
    t = b.add("conv", x, cin=cin, cout=exp, k=1, stride=1, bias=0)
    t = b.add("affine", t, c=exp)
    t = b.add(act, t)
    t = b.add("dwconv", t, c=exp, k=k, stride=stride, bias=0)
    t = b.add("affine", t, c=exp)
    t = b.add(act, t)
    if se:
        sq = b.add("avgpool", t)
        sq = b.add("linear", sq, cin=exp, cout=exp // 4, bias=1)
        sq = b.add("relu", sq)
        sq = b.add("linear", sq, cin=exp // 4, cout=exp, bias=1)
        sq = b.add("hsigmoid", sq)
        t = b.add("chmul", t, in1=sq)
    t = b.add("conv", t, cin=exp, cout=cout, k=1, stride=1, bias=0)
    t = b.add("affine", t, c=cout)
    if stride == 1 and cin == cout:
        t = b.add("add", t, in1=x)
    return t


def mobilenet_ops(classes=200):
    """Server part of MobileNetV3-Large (the paper's Table 4) after its
    BNECK-3-112 stage: BNECK-5-160 x 3 (the first with stride 2),
    CONV-1-960, global average pool, CONV-1-1280 (on the pooled 1 x 1 map,
    a dense layer) and FC -> classes (200, Tiny ImageNet's), with hard swish
    activations, on a [4,4,112] input."""
    b = _Builder()
    t = _bneck(b, 0, 112, 672, 160, 5, 2)
    t = _bneck(b, t, 160, 960, 160, 5, 1)
    t = _bneck(b, t, 160, 960, 160, 5, 1)
    t = b.add("conv", t, cin=160, cout=960, k=1, stride=1, bias=0)
    t = b.add("affine", t, c=960)
    t = b.add("hswish", t)
    t = b.add("avgpool", t)
    t = b.add("linear", t, cin=960, cout=1280, bias=1)
    t = b.add("hswish", t)
    b.add("linear", t, cin=1280, cout=classes, bias=1)
    return b.ops


def _basic_block(b, x, cin, cout, stride):
    """ResNet basic block with BN folded to a trainable per-channel affine."""
    t = b.add("conv", x, cin=cin, cout=cout, k=3, stride=stride, bias=0)
    t = b.add("affine", t, c=cout)
    t = b.add("relu", t)
    t = b.add("conv", t, cin=cout, cout=cout, k=3, stride=1, bias=0)
    t = b.add("affine", t, c=cout)
    if stride != 1 or cin != cout:
        s = b.add("conv", x, cin=cin, cout=cout, k=1, stride=stride, bias=0)
        s = b.add("affine", s, c=cout)
    else:
        s = x
    t = b.add("add", t, in1=s)
    return b.add("relu", t)


def resnet_ops(classes=100):
    """ResNet-18 stages 3-4 (256 and 512 channels, stride-2 entry blocks,
    two basic blocks per stage) + global avgpool + FC 512 -> classes, on a
    [16,16,128] input."""
    b = _Builder()
    t = 0
    t = _basic_block(b, t, 128, 256, 2)
    t = _basic_block(b, t, 256, 256, 1)
    t = _basic_block(b, t, 256, 512, 2)
    t = _basic_block(b, t, 512, 512, 1)
    t = b.add("avgpool", t)
    b.add("linear", t, cin=512, cout=classes, bias=1)
    return b.ops


def transformer_ops(d=512, heads=8, ffn=2048, blocks=4, classes=2):
    """Pre-LN encoder blocks: x += proj(attn(LN1(x))); x += W2 GELU(W1 LN2(x));
    then a final LN, masked mean-pool and a linear classifier."""
    b = _Builder()
    x = 0
    for _ in range(blocks):
        t = b.add("layernorm", x, c=d)
        t = b.add("linear", t, cin=d, cout=3 * d, bias=1)
        t = b.add("attention", t, c=d, heads=heads)
        t = b.add("linear", t, cin=d, cout=d, bias=1)
        x = b.add("add", x, in1=t)
        t = b.add("layernorm", x, c=d)
        t = b.add("linear", t, cin=d, cout=ffn, bias=1)
        t = b.add("gelu", t)
        t = b.add("linear", t, cin=ffn, cout=d, bias=1)
        x = b.add("add", x, in1=t)
    t = b.add("layernorm", x, c=d)
    t = b.add("meanpool", t)
    b.add("linear", t, cin=d, cout=classes, bias=1)
    return b.ops


# --------------------------------------------------------------------------
# configurations
# --------------------------------------------------------------------------

def _cfg(name, ops, K, depth, omega, batch, in_hwc, dtype, classes, seed,
         steps, agg_params, rates, seq=False, lr=0.01, momentum=0.9):
    return {
        "name": name, "ops": ops, "K": K, "depth": depth, "omega": omega,
        "batch": batch, "in_hwc": tuple(in_hwc), "dtype": dtype,
        "classes": classes, "seed": seed, "steps": steps,
        "agg_params": agg_params, "rates": rates, "seq": seq,
        "lr": lr, "momentum": momentum,
    }


# Device compute rates of the paper's testbed B groups (GPU clocks in MHz,
# Table 3): four equal groups of devices.
GROUP_RATES = (240.0, 320.0, 640.0, 921.0)


def group_rates(K):
    return [GROUP_RATES[min(3, (4 * k) // K)] for k in range(K)]


def zipf_rates(K, s=1.2):
    return [float((k + 1) ** -s) for k in range(K)]


CONFIGS = {
    "tiny": _cfg("tiny", tiny_cnn_ops(), K=4, depth=2, omega=8, batch=16,
                 in_hwc=(16, 16, 32), dtype=F32, classes=10, seed=0, steps=8,
                 agg_params=20_000, rates=[1.0] * 4),
    "vgg": _cfg("vgg", vgg_ops(), K=10, depth=4, omega=40, batch=64,
                in_hwc=(16, 16, 128), dtype=BF16, classes=10, seed=1,
                steps=200, agg_params=1_000_000, rates=group_rates(10)),
    "resnet": _cfg("resnet", resnet_ops(), K=20, depth=4, omega=80, batch=128,
                   in_hwc=(16, 16, 128), dtype=BF16, classes=100, seed=2,
                   steps=500, agg_params=700_000, rates=group_rates(20)),
    "transformer": _cfg("transformer", transformer_ops(), K=16, depth=4,
                        omega=64, batch=32, in_hwc=(128, 1, 512), dtype=BF16,
                        classes=2, seed=3, steps=300,
                        agg_params=30522 * 512 + 2 * 3_152_384,
                        rates=group_rates(16), seq=True),
    "scale": _cfg("scale", resnet_ops(), K=100, depth=4, omega=400, batch=64,
                  in_hwc=(16, 16, 128), dtype=BF16, classes=100, seed=4,
                  steps=1000, agg_params=700_000, rates=zipf_rates(100)),
    "mobilenet": _cfg("mobilenet", mobilenet_ops(), K=10, depth=4, omega=40, batch=64,
                      in_hwc=(4, 4, 112), dtype=BF16, classes=200, seed=6, steps=200,
                      agg_params=1_000_000, rates=group_rates(10)),
    # one device's own trainer for the live VGG pipeline: its local data
    # queue (K = 1) feeds M_dk + the auxiliary network
    "vgg_device": _cfg("vgg_device", vgg_device_ops(), K=1, depth=2, omega=2, batch=64,
                       in_hwc=(32, 32, 3), dtype=BF16, classes=10, seed=5, steps=0,
                       agg_params=0, rates=[1.0]),
}


def shrink(cfg, **over):
    """A copy of a configuration with some fields replaced (small test cases)."""
    c = dict(cfg)
    c.update(over)
    return c


# --------------------------------------------------------------------------
# parameter shapes (the flat parameter vector's layout)
# --------------------------------------------------------------------------

def param_shapes(ops):
    """Shapes of every parameter tensor, in flat-vector order."""
    shapes = []
    for op in ops:
        kind = op["kind"]
        if kind == "conv":
            shapes.append(("W", (op["cout"], op["k"], op["k"], op["cin"])))
            if op["bias"]:
                shapes.append(("b", (op["cout"],)))
        elif kind == "linear":
            shapes.append(("W", (op["cout"], op["cin"])))
            if op["bias"]:
                shapes.append(("b", (op["cout"],)))
        elif kind == "affine":
            shapes.append(("scale", (op["c"],)))
            shapes.append(("shift", (op["c"],)))
        elif kind == "layernorm":
            shapes.append(("gamma", (op["c"],)))
            shapes.append(("beta", (op["c"],)))
        elif kind == "dwconv":
            shapes.append(("W", (op["c"], op["k"], op["k"])))
            if op["bias"]:
                shapes.append(("b", (op["c"],)))
    return shapes


def num_params(ops):
    return int(sum(int(np.prod(s)) for _, s in param_shapes(ops)))


# --------------------------------------------------------------------------
# seeded generators
# --------------------------------------------------------------------------

def _rng(*key):
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(list(key))))


def round_to_bf16(x):
    """Round fp32 values to the nearest bf16 (ties to even); returns
    (fp32 values, uint16 bit patterns).  Inputs are finite."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    bits = u.astype(np.uint16)
    vals = (bits.astype(np.uint32) << 16).view(np.float32)
    return vals, bits


def init_params(cfg):
    """Initial server weights: conv/linear W ~ N(0, 2/fan_in), biases 0,
    affine scale 1 / shift 0, layernorm gamma 1 / beta 0.  fp32, flat."""
    rng = _rng(cfg["seed"], 0)
    out = []
    for name, shape in param_shapes(cfg["ops"]):
        n = int(np.prod(shape))
        if name == "W":
            fan_in = int(np.prod(shape[1:]))
            out.append(rng.standard_normal(n, dtype=np.float32)
                       * np.float32(np.sqrt(2.0 / fan_in)))
        elif name in ("scale", "gamma"):
            out.append(np.ones(n, np.float32))
        else:
            out.append(np.zeros(n, np.float32))
    return np.concatenate(out).astype(np.float32)


def device_batch(cfg, k, j, batch=None):
    """Batch j uploaded by device k: (acts fp32 [B,H,W,C], acts_bits or None,
    labels int32 [B], lengths int32 [B] or None).  For bf16 configurations
    the activations are bf16-rounded fp32 values and acts_bits holds the
    bf16 bit patterns that are actually uploaded."""
    B = cfg["batch"] if batch is None else batch
    H, W, C = cfg["in_hwc"]
    rng = _rng(cfg["seed"], 1, k, j)
    x = rng.standard_normal((B, H, W, C), dtype=np.float32)
    if not cfg["seq"]:
        x = np.maximum(x, 0.0, dtype=np.float32)
    if cfg.get("kink_values"):
        # edge cases: about a quarter of the elements set exactly to the given
        # values (e.g. the hard-swish kinks -3 and 3)
        kv = np.asarray(cfg["kink_values"], np.float32)
        pick = rng.random(x.shape) < 0.25
        x = np.where(pick, kv[rng.integers(0, len(kv), size=x.shape)], x).astype(np.float32)
    if cfg["seq"]:
        labels = rng.integers(0, 2, size=B).astype(np.int32)
        lengths = rng.integers(32, 129, size=B).astype(np.int32)
        lengths = np.minimum(lengths, H).astype(np.int32)
        if cfg.get("fixed_len") is not None:   # edge cases: every sequence of one length
            lengths = np.full(B, cfg["fixed_len"], np.int32)
    else:
        labels = rng.integers(0, cfg["classes"], size=B).astype(np.int32)
        lengths = None
    bits = None
    if cfg["dtype"] == BF16:
        x, bits = round_to_bf16(x)
    return x, bits, labels, lengths


def device_model(n, seed, k, j):
    """Local device-side model (theta_dk and aux params, flattened), N(0, 0.05)."""
    return (_rng(seed, 2, k, j).standard_normal(n, dtype=np.float32)
            * np.float32(0.05)).astype(np.float32)


def global_model(n, seed):
    """Initial global device-side model, N(0, 0.05)."""
    return (_rng(seed, 3).standard_normal(n, dtype=np.float32)
            * np.float32(0.05)).astype(np.float32)


def arrival_order(rates, n_events, seed):
    """Device ids of the next n_events activation uploads when device k
    uploads as a Poisson process of rate rates[k]."""
    rng = _rng(seed, 4)
    rates = np.asarray(rates, np.float64)
    nxt = rng.exponential(1.0 / rates)
    out = []
    for _ in range(n_events):
        k = int(np.argmin(nxt))
        out.append(k)
        nxt[k] += rng.exponential(1.0 / rates[k])
    return out


def trace(cfg, n_steps, uploads_per_step=1, prefill=True, agg_every=0,
          seed_offset=0):
    """A deterministic event list: optional prefill (every device uploads
    `depth` batches), then per server step `uploads_per_step` uploads in
    Poisson arrival order and one step; every `agg_every` steps a device model
    arrives (device ids in arrival order).  Events: ("enq", k), ("step",),
    ("agg", k)."""
    K = cfg["K"]
    ev = []
    if prefill:
        for r in range(cfg["depth"]):
            for k in range(K):
                ev.append(("enq", k))
    order = arrival_order(cfg["rates"], n_steps * uploads_per_step + n_steps,
                          cfg["seed"] + seed_offset)
    it = iter(order)
    for s in range(n_steps):
        for _ in range(uploads_per_step):
            ev.append(("enq", next(it)))
        ev.append(("step",))
        if agg_every and (s + 1) % agg_every == 0:
            ev.append(("agg", next(it)))
    return ev
