"""Seeded synthetic workloads shared by the tests, the smoke check and the benchmark.

This module only *draws* inputs and describes layer shapes; it holds none of
the method's arithmetic (no statistics, no FLOP counting, no dispatch, no
operator math).  Values are drawn in fp32 on the CPU with a seeded
``torch.Generator`` and stored as bf16 bit patterns (uint16 numpy arrays),
which both the CUDA path and the oracle read byte for byte.

Workloads (stand-ins for the paper's ImageNet / COCO inputs and pretrained
weights, which are not available; same shapes, 224x224 RGB, batch 1/8/32):
  fc_layer        single FC operator, x [64, 512] ReLU(N(0,1)) with whole
                  K-columns zeroed at p = 0.4, W [512, 512] N(0, 1/512)
  conv_layer      single 3x3 conv, stride 1, pad 1, NHWC [8, 56, 56, 64],
                  x = ReLU(N(0,1)), W He-normal, BN(1, 0, 0, 1) + ReLU epilogue
  resnet18        ResNet-18 topology, He-normal weights, BN (gamma 1, beta 0,
                  mean 0, var 1) after every conv, input N(0,1) [B, 224, 224, 3]
  mobilenet_v2    MobileNetV2 (width 1.0) topology, ReLU6, He-normal weights
  mlp_hidden      the hidden activation of a 768 -> 3072 -> 768 ReLU MLP drawn
                  directly at a target zero fraction, unstructured or in
                  32-channel blocks per 128-token tile
  vit             ViT-B/16 shaped transformer (patch conv, class token, pre-norm
                  encoder layers with GELU MLPs, head), random weights
  structured_activation  a [M, K] or NHWC activation at a target zero
                  fraction, unstructured or in blocks (threshold calibration;
                  drawn on the device the caller names)
"""
from __future__ import annotations

import math

import numpy as np
import torch

ACT_NONE, ACT_RELU, ACT_RELU6, ACT_GELU = 0, 1, 2, 3


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator()
    g.manual_seed(int(seed))
    return g


def to_bf16_bits(t: torch.Tensor) -> np.ndarray:
    """fp32 tensor -> bf16 (round to nearest even) -> uint16 bit patterns."""
    return t.to(torch.bfloat16).contiguous().view(torch.int16).numpy().view(np.uint16).copy()


def bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> float32 values (exact)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def he_normal(shape, fan_in: int, g: torch.Generator) -> torch.Tensor:
    return torch.randn(shape, generator=g, dtype=torch.float32) * math.sqrt(2.0 / fan_in)


def identity_bn(c: int) -> np.ndarray:
    """Batch-norm parameters gamma=1, beta=0, mean=0, var=1 as a [4, c] fp32 array."""
    bn = np.zeros((4, c), dtype=np.float32)
    bn[0] = 1.0
    bn[3] = 1.0
    return bn


def random_bn(c: int, g: torch.Generator) -> np.ndarray:
    """Non-trivial batch-norm parameters, used by the epilogue tests."""
    gamma = 0.5 + torch.rand(c, generator=g)
    beta = 0.2 * torch.randn(c, generator=g)
    mean = 0.2 * torch.randn(c, generator=g)
    var = 0.5 + torch.rand(c, generator=g)
    return torch.stack([gamma, beta, mean, var]).numpy().astype(np.float32)


# --------------------------------------------------------------------------
# single operators
# --------------------------------------------------------------------------
def fc_layer(seed: int = 0, M: int = 64, K: int = 512, N: int = 512, col_zero_p: float = 0.4):
    """FC operator: x = ReLU(N(0,1))[M, K] with whole K-columns zeroed with
    probability ``col_zero_p`` (one mask shared by all rows); W ~ N(0, 1/K) [N, K];
    bias fp32 zeros."""
    g = _gen(seed)
    x = torch.relu(torch.randn(M, K, generator=g))
    keep = (torch.rand(K, generator=g) >= col_zero_p).to(torch.float32)
    x = x * keep[None, :]
    w = torch.randn(N, K, generator=g) * math.sqrt(1.0 / K)
    return {
        "x": to_bf16_bits(x), "M": M, "K": K, "N": N,
        "w": to_bf16_bits(w),
        "w_kn": to_bf16_bits(w.t().contiguous()),
        "bias": np.zeros(N, dtype=np.float32),
    }


def conv_layer(seed: int = 0, N: int = 8, H: int = 56, W: int = 56, Cin: int = 64,
               Cout: int = 64, k: int = 3, stride: int = 1, pad: int = 1, bn: str = "identity",
               act: int = ACT_RELU, zero_p: float | None = None):
    """Conv operator: x = ReLU(N(0,1)) NHWC (about half zeros), or, with
    ``zero_p``, |N(0,1)| on a Bernoulli(1 - zero_p) support; W He-normal stored
    [Cout, k, k, Cin]; batch norm after the conv, then ``act``."""
    g = _gen(seed)
    if zero_p is None:
        x = torch.relu(torch.randn(N, H, W, Cin, generator=g))
    else:
        x = torch.randn(N, H, W, Cin, generator=g).abs()
        x = x * (torch.rand(N, H, W, Cin, generator=g) >= zero_p).to(torch.float32)
    w = he_normal((Cout, Cin, k, k), Cin * k * k, g).permute(0, 2, 3, 1).contiguous()
    bnp = identity_bn(Cout) if bn == "identity" else random_bn(Cout, g)
    return {
        "x": to_bf16_bits(x), "N": N, "H": H, "W": W, "Cin": Cin, "Cout": Cout,
        "k": k, "stride": stride, "pad": pad, "w": to_bf16_bits(w),
        "bias": None, "bn": bnp, "eps": 1e-5, "act": act,
    }


# --------------------------------------------------------------------------
# graphs
# --------------------------------------------------------------------------
def _conv_op(g, inp, cin, cout, k, stride, pad, act, groups=1, residual=-1, thr=None):
    fan_in = (cin // groups) * k * k
    w = he_normal((cout, cin // groups, k, k), fan_in, g).permute(0, 2, 3, 1).contiguous()
    return {
        "kind": "conv", "input": inp, "residual": residual, "cin": cin, "cout": cout, "k": k,
        "stride": stride, "pad": pad, "groups": groups, "act": act,
        "w": to_bf16_bits(w), "bias": None, "bn": identity_bn(cout), "eps": 1e-5,
        "thr": dict(thr or {}),
    }


def _fc_op(g, inp, cin, cout, thr=None):
    w = he_normal((cout, cin), cin, g)
    return {
        "kind": "fc", "input": inp, "residual": -1, "cin": cin, "cout": cout, "act": ACT_NONE,
        "w": to_bf16_bits(w), "w_kn": to_bf16_bits(w.t().contiguous()),
        "bias": np.zeros(cout, dtype=np.float32), "bn": None, "eps": 1e-5,
        "thr": dict(thr or {}),
    }


def resnet18(batch: int = 1, seed: int = 0, thr=None):
    """ResNet-18 on [batch, 224, 224, 3] NHWC: 20 convs (3 of them 1x1
    downsample), max pool, global average pool, FC 512 -> 1000 (23 operators).
    Residual additions are fused into the second conv of each block.
    Returns (ops, x_bits, x_shape); op i reads value ``op["input"]`` (0 = graph
    input, j + 1 = output of op j)."""
    g = _gen(seed)
    x = torch.randn(batch, 224, 224, 3, generator=g)
    ops = []

    def add(op):
        ops.append(op)
        return len(ops)  # value index of its output

    v = add(_conv_op(g, 0, 3, 64, 7, 2, 3, ACT_RELU, thr=thr))
    v = add({"kind": "maxpool", "input": v, "residual": -1, "k": 3, "stride": 2, "pad": 1})
    cin = 64
    for stage, cout in enumerate([64, 128, 256, 512]):
        for blk in range(2):
            stride = 2 if (stage > 0 and blk == 0) else 1
            a = add(_conv_op(g, v, cin, cout, 3, stride, 1, ACT_RELU, thr=thr))
            if stride != 1 or cin != cout:
                sc = add(_conv_op(g, v, cin, cout, 1, stride, 0, ACT_NONE, thr=thr))
            else:
                sc = v
            v = add(_conv_op(g, a, cout, cout, 3, 1, 1, ACT_RELU, residual=sc, thr=thr))
            cin = cout
    v = add({"kind": "avgpool", "input": v, "residual": -1})
    add(_fc_op(g, v, 512, 1000, thr=thr))
    return ops, to_bf16_bits(x), (batch, 224, 224, 3)


MBV2_SETTINGS = [(1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2),
                 (6, 96, 3, 1), (6, 160, 3, 2), (6, 320, 1, 1)]


def mobilenet_v2(batch: int = 1, seed: int = 0, thr=None):
    """MobileNetV2, width 1.0, on [batch, 224, 224, 3]: stem 3x3/2 conv,
    17 inverted-residual blocks (1x1 expand + ReLU6, 3x3 depthwise + ReLU6,
    1x1 linear projection, residual when stride 1 and channels match),
    1x1 conv to 1280 + ReLU6, global average pool, FC 1280 -> 1000."""
    g = _gen(seed)
    x = torch.randn(batch, 224, 224, 3, generator=g)
    ops = []

    def add(op):
        ops.append(op)
        return len(ops)

    v = add(_conv_op(g, 0, 3, 32, 3, 2, 1, ACT_RELU6, thr=thr))
    cin = 32
    for t, c, n, s in MBV2_SETTINGS:
        for i in range(n):
            stride = s if i == 0 else 1
            hidden = cin * t
            inp = v
            h = v
            if t != 1:
                h = add(_conv_op(g, h, cin, hidden, 1, 1, 0, ACT_RELU6, thr=thr))
            h = add(_conv_op(g, h, hidden, hidden, 3, stride, 1, ACT_RELU6, groups=hidden, thr=thr))
            res = inp if (stride == 1 and cin == c) else -1
            v = add(_conv_op(g, h, hidden, c, 1, 1, 0, ACT_NONE, residual=res, thr=thr))
            cin = c
    v = add(_conv_op(g, v, 320, 1280, 1, 1, 0, ACT_RELU6, thr=thr))
    v = add({"kind": "avgpool", "input": v, "residual": -1})
    add(_fc_op(g, v, 1280, 1000, thr=thr))
    return ops, to_bf16_bits(x), (batch, 224, 224, 3)


# --------------------------------------------------------------------------
# MLP sparsity sweep
# --------------------------------------------------------------------------
def mlp_weights(seed: int = 0, d: int = 768, hidden: int = 3072):
    g = _gen(seed)
    w1 = he_normal((hidden, d), d, g)
    w2 = he_normal((d, hidden), hidden, g)
    return {"w1": to_bf16_bits(w1), "w2": to_bf16_bits(w2),
            "w2_kn": to_bf16_bits(w2.t().contiguous()), "d": d, "hidden": hidden}


def mlp_hidden(M: int, rho: float, structure: str = "unstructured", seed: int = 0,
               hidden: int = 3072):
    """Hidden activation h [M, hidden] with |N(0,1)| values and a target zero
    fraction ``rho``:
      unstructured  iid Bernoulli(rho) zeros
      block32       32-channel blocks zeroed as units, one draw per
                    (128-token tile, 32-channel group)
      token         whole tokens (rows) zeroed"""
    g = _gen(seed)
    h = torch.randn(M, hidden, generator=g).abs() + 1e-3
    if structure == "unstructured":
        keep = torch.rand(M, hidden, generator=g) >= rho
    elif structure == "block32":
        tiles = (M + 127) // 128
        kb = torch.rand(tiles, hidden // 32, generator=g) >= rho
        keep = kb.repeat_interleave(128, dim=0)[:M].repeat_interleave(32, dim=1)
    elif structure == "token":
        keep = (torch.rand(M, 1, generator=g) >= rho).expand(M, hidden)
    else:
        raise ValueError(structure)
    return to_bf16_bits(h * keep.to(torch.float32))


# --------------------------------------------------------------------------
# threshold calibration inputs
# --------------------------------------------------------------------------
STRUCTURES = ("unstructured", "block")


def structured_activation(shape, rho: float, structure: str, gen: torch.Generator,
                          device="cpu") -> torch.Tensor:
    """A bf16 activation of ``shape`` with |N(0,1)| + 1e-3 values and a target
    zero fraction ``rho``, drawn with ``gen`` on ``device``:
      unstructured  iid Bernoulli(rho) zeros (a ReLU output)
      block         units zeroed together: 128 rows x 32 channels of a 2-D
                    [M, K] input; 8 image rows x 64 channels of one image of
                    an NHWC [B, H, W, C] input (spatially clustered zeros)"""
    v = torch.randn(*shape, device=device, generator=gen).abs_() + 1e-3
    if structure == "unstructured":
        keep = torch.rand(*shape, device=device, generator=gen) >= rho
    elif structure == "block" and len(shape) == 2:
        M, K = shape
        kb = torch.rand((M + 127) // 128, (K + 31) // 32, device=device, generator=gen) >= rho
        keep = kb.repeat_interleave(128, dim=0)[:M].repeat_interleave(32, dim=1)[:, :K]
    elif structure == "block" and len(shape) == 4:
        B, H, W, C = shape
        kb = torch.rand(B, (H + 7) // 8, 1, (C + 63) // 64, device=device, generator=gen) >= rho
        keep = kb.repeat_interleave(8, dim=1)[:, :H].repeat_interleave(64, dim=3)[..., :C]
        keep = keep.expand(B, H, W, C)
    else:
        raise ValueError(f"structure {structure!r} for shape {tuple(shape)}")
    return (v * keep.to(v.dtype)).to(torch.bfloat16)


# --------------------------------------------------------------------------
# vision transformer
# --------------------------------------------------------------------------
def _lin_op(g, inp, cin, cout, act, residual=-1, thr=None):
    """Token-wise linear layer as a 1x1 conv with bias (no batch norm)."""
    w = torch.randn(cout, cin, generator=g) / math.sqrt(cin)
    return {
        "kind": "conv", "input": inp, "residual": residual, "cin": cin, "cout": cout, "k": 1,
        "stride": 1, "pad": 0, "groups": 1, "act": act,
        "w": to_bf16_bits(w.reshape(cout, 1, 1, cin)),
        "bias": (0.02 * torch.randn(cout, generator=g)).numpy().astype(np.float32), "bn": None,
        "eps": 1e-5, "thr": dict(thr or {}),
    }


def _ln_op(g, inp, c):
    gb = np.stack([1.0 + 0.1 * torch.randn(c, generator=g).numpy(),
                   0.02 * torch.randn(c, generator=g).numpy()]).astype(np.float32)
    return {"kind": "layernorm", "input": inp, "residual": -1, "gamma_beta": gb, "eps": 1e-6}


def vit(batch: int = 1, seed: int = 0, img: int = 224, patch: int = 16, dim: int = 768, depth: int = 12,
        heads: int = 12, mlp: int = 3072, classes: int = 1000, act: int = 3, thr=None):
    """ViT-B/16 shaped (Table 2: 86M parameters, 17.6 G): 16x16/16 patch
    embedding (conv) on [batch, 224, 224, 3], class token + position
    embedding, `depth` pre-norm encoder layers (LN, QKV, MHSA, projection +
    residual, LN, MLP dim -> mlp (GELU, act = 3) -> dim + residual), final LN,
    the class token, FC -> classes.  Random N(0, 1/fan_in) weights; tokens
    live as [batch, 1, T, dim]."""
    g = _gen(seed)
    x = torch.randn(batch, img, img, 3, generator=g)
    ops = []

    def add(op):
        ops.append(op)
        return len(ops)

    P = (img // patch) ** 2
    w = torch.randn(dim, 3 * patch * patch, generator=g) / math.sqrt(3 * patch * patch)
    v = add({"kind": "conv", "input": 0, "residual": -1, "cin": 3, "cout": dim, "k": patch,
             "stride": patch, "pad": 0, "groups": 1, "act": ACT_NONE,
             "w": to_bf16_bits(w.reshape(dim, patch, patch, 3)),
             "bias": (0.02 * torch.randn(dim, generator=g)).numpy().astype(np.float32), "bn": None,
             "eps": 1e-5, "thr": dict(thr or {})})
    v = add({"kind": "tokens", "input": v, "residual": -1,
             "cls": to_bf16_bits(0.02 * torch.randn(dim, generator=g)),
             "pos": (0.02 * torch.randn(P + 1, dim, generator=g)).numpy().astype(np.float32)})
    for _ in range(depth):
        a = add(_ln_op(g, v, dim))
        q = add(_lin_op(g, a, dim, 3 * dim, ACT_NONE, thr=thr))
        o = add({"kind": "attention", "input": q, "residual": -1, "heads": heads})
        v = add(_lin_op(g, o, dim, dim, ACT_NONE, residual=v, thr=thr))
        b = add(_ln_op(g, v, dim))
        h = add(_lin_op(g, b, dim, mlp, act, thr=thr))
        v = add(_lin_op(g, h, mlp, dim, ACT_NONE, residual=v, thr=thr))
    v = add(_ln_op(g, v, dim))
    v = add({"kind": "select", "input": v, "residual": -1, "index": 0})
    add(_fc_op(g, v, dim, classes, thr=thr))
    return ops, to_bf16_bits(x), (batch, img, img, 3)
