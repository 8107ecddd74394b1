"""Seeded synthetic workloads for the carry-through checksum hot path.

This module is shared by the CPU oracle (``oracle/``) and the CUDA path
(``paper_2609_16742_gb300``).  It holds NO arithmetic of the method itself:
no carry-through filter, no zero slice, no BN folding, no checksum, no
verification.  It only describes the five network shapes, draws their
parameters and input images from a counter-based generator, and draws fault
sites uniformly from buffer sizes that the caller supplies.

Random numbers: SplitMix64 (Steele, Lea, Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014) evaluated in counter mode, so
value ``i`` of stream ``(seed, stream)`` does not depend on how many values
were drawn before it.  Uniforms take the top 53 bits; normals use the
Box-Muller transform (Box & Muller, 1958) on consecutive uniform pairs.

Network shapes follow the five workloads of the evaluation:
  * LeNet-5, 1x28x28 inputs uniform in [0, 1], FP32, batch 64;
  * ResNet-18 with a 3x3 CIFAR stem, 3x32x32 N(0,1) inputs, FP32, batch 128;
  * ResNet-18 with the 7x7/2 ImageNet stem + 3x3/2 max-pool, 3x224x224
    N(0,1) inputs, FP16 storage, batch 256;
  * VGG-16, 3x224x224 N(0,1) inputs, FP16 storage, batch 64;
  * the CIFAR ResNet-18 again for the fault-injection campaign.
Weights are Kaiming-normal (fan-in mode, gain sqrt(2)), biases zero.  The
ResNets carry BatchNorm parameters (gamma, beta, running mean, running var)
drawn from fixed ranges that keep activations near unit scale; folding them
into the convolutions is the job of each consumer, not of this module.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np

__all__ = [
    "Layer", "Workload", "WORKLOADS", "workload", "make_params", "make_input",
    "splitmix64_stream", "uniform", "normal", "draw_faults", "lenet5",
    "resnet18", "vgg16",
]

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def _mix(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function on an array of uint64 states (in place)."""
    t = np.empty_like(z)
    np.right_shift(z, np.uint64(30), out=t)
    np.bitwise_xor(z, t, out=z)
    np.multiply(z, _M1, out=z)
    np.right_shift(z, np.uint64(27), out=t)
    np.bitwise_xor(z, t, out=z)
    np.multiply(z, _M2, out=z)
    np.right_shift(z, np.uint64(31), out=t)
    np.bitwise_xor(z, t, out=z)
    return z


def _key(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        s = _mix(np.array([np.uint64(seed & 0xFFFFFFFFFFFFFFFF)], dtype=np.uint64))[0]
        s = _mix(np.array([s ^ np.uint64((stream * 0x632BE59BD9B4E019) & 0xFFFFFFFFFFFFFFFF)],
                          dtype=np.uint64))[0]
    return s


_CHUNK = 1 << 18


def _stream_into(key: np.uint64, offset: int, out: np.ndarray) -> None:
    """out[i] = mix(key + (offset + i + 1) * golden), computed chunk by chunk."""
    n = out.shape[0]
    with np.errstate(over="ignore"):
        for a in range(0, n, _CHUNK):
            b = min(n, a + _CHUNK)
            z = np.arange(offset + a + 1, offset + b + 1, dtype=np.uint64)
            np.multiply(z, _GOLDEN, out=z)
            np.add(z, key, out=z)
            out[a:b] = _mix(z)


def splitmix64_stream(seed: int, stream: int, n: int, offset: int = 0) -> np.ndarray:
    """Values ``offset .. offset+n-1`` of the counter-mode SplitMix64 stream."""
    out = np.empty(n, dtype=np.uint64)
    _stream_into(_key(seed, stream), offset, out)
    return out


def _to_unit(z: np.ndarray) -> np.ndarray:
    """Top 53 bits of each uint64 as a float64 in [0, 1)."""
    u = (z >> np.uint64(11)).view(np.int64)         # < 2**53, exact in int64
    return u.astype(np.float64) * (1.0 / 9007199254740992.0)


def uniform(seed: int, stream: int, n: int) -> np.ndarray:
    """n float64 values uniform in [0, 1), 53-bit resolution."""
    return _to_unit(splitmix64_stream(seed, stream, n))


def normal(seed: int, stream: int, n: int) -> np.ndarray:
    """n float64 standard normals by Box-Muller on consecutive uniform pairs.

    Pair j uses uniforms 2j (radius) and 2j+1 (angle) of the stream and gives
    normals 2j (cosine branch) and 2j+1 (sine branch).
    """
    m = (n + 1) // 2
    key = _key(seed, stream)
    z = np.empty(2 * m, dtype=np.float64)
    buf = np.empty(2 * _CHUNK, dtype=np.uint64)
    for a in range(0, m, _CHUNK):
        b = min(m, a + _CHUNK)
        raw = buf[:2 * (b - a)]
        _stream_into(key, 2 * a, raw)
        u = _to_unit(raw)
        u1, u2 = 1.0 - u[0::2], u[1::2]          # u1 in (0, 1]
        rad = np.sqrt(-2.0 * np.log(u1))
        ang = (2.0 * math.pi) * u2
        z[2 * a:2 * b:2] = rad * np.cos(ang)
        z[2 * a + 1:2 * b:2] = rad * np.sin(ang)
    return z[:n]


# --------------------------------------------------------------------------
# Network description
# --------------------------------------------------------------------------

@dataclass
class Layer:
    """One operation of a feed-forward CNN over numbered tensor slots.

    Slot 0 is the network input.  ``op`` is one of
      conv    : KxK convolution (+ optional BatchNorm, residual add, ReLU)
      maxpool : k x k max-pool, stride s, padding p
      gap     : global average pool to a vector
      fc      : fully connected layer (input flattened in (C, H, W) order)
    ``ct`` names the role the layer plays in the protection scheme:
      "ct"   : the layer gets a carry-through filter
      "none" : the layer gets none (first conv of a residual block)
      "pass" : a 1x1 shortcut convolution
    How each role is realised is decided by the consumer.
    ``groups`` > 1 is a depthwise convolution (groups == cin == cout):
    output channel c reads input channel c only.
    """
    op: str
    src: int
    dst: int
    cin: int = 0
    cout: int = 0
    k: int = 1
    stride: int = 1
    pad: int = 0
    ct: str = "ct"
    bn: bool = False
    relu: bool = False
    res: int = -1
    final: bool = False
    ct_shift: int = 0      # carry-through coefficient is 2**-ct_shift
    groups: int = 1


@dataclass
class Workload:
    name: str
    layers: List[Layer]
    in_shape: tuple           # (C, H, W)
    n_classes: int
    batch: int
    precision: str            # "fp32" | "fp16"
    seed: int
    input_kind: str           # "uniform01" | "normal"
    bn_eps: float = 1e-5
    notes: str = ""
    calib_seed: int = 0


def lenet5() -> List[Layer]:
    return [
        Layer("conv", 0, 1, cin=1, cout=6, k=5, stride=1, pad=0, ct="ct", relu=True),
        Layer("maxpool", 1, 2, k=2, stride=2, pad=0),
        Layer("conv", 2, 3, cin=6, cout=16, k=5, stride=1, pad=0, ct="ct", relu=True),
        Layer("maxpool", 3, 4, k=2, stride=2, pad=0),
        Layer("fc", 4, 5, cin=256, cout=120, relu=True),
        Layer("fc", 5, 6, cin=120, cout=84, relu=True),
        Layer("fc", 6, 7, cin=84, cout=10, final=True),
    ]


def resnet18(imagenet_stem: bool, n_classes: int, downsample_ct: str = "pass") -> List[Layer]:
    L: List[Layer] = []
    slot = 0

    def new() -> int:
        nonlocal slot
        slot += 1
        return slot

    if imagenet_stem:
        s1 = new()
        L.append(Layer("conv", 0, s1, cin=3, cout=64, k=7, stride=2, pad=3, ct="ct", bn=True, relu=True))
        s2 = new()
        L.append(Layer("maxpool", s1, s2, k=3, stride=2, pad=1))
        x = s2
    else:
        s1 = new()
        L.append(Layer("conv", 0, s1, cin=3, cout=64, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True))
        x = s1
    cin = 64
    for stage, cout in enumerate((64, 128, 256, 512)):
        for blk in range(2):
            stride = 2 if (stage > 0 and blk == 0) else 1
            h = new()
            L.append(Layer("conv", x, h, cin=cin, cout=cout, k=3, stride=stride, pad=1,
                           ct="none", bn=True, relu=True))
            if stride != 1 or cin != cout:
                d = new()
                L.append(Layer("conv", x, d, cin=cin, cout=cout, k=1, stride=stride, pad=0,
                               ct=downsample_ct, bn=True, relu=False))
                res = d
            else:
                res = x
            y = new()
            L.append(Layer("conv", h, y, cin=cout, cout=cout, k=3, stride=1, pad=1,
                           ct="ct", bn=True, relu=True, res=res))
            x, cin = y, cout
    g = new()
    L.append(Layer("gap", x, g))
    o = new()
    L.append(Layer("fc", g, o, cin=512, cout=n_classes, final=True))
    return L


def vgg16(n_classes: int = 1000, fc1_shift: int = 0) -> List[Layer]:
    plan = [64, 64, "M", 128, 128, "M", 256, 256, 256, "M", 512, 512, 512, "M", 512, 512, 512, "M"]
    L: List[Layer] = []
    slot, cin = 0, 3
    for v in plan:
        if v == "M":
            L.append(Layer("maxpool", slot, slot + 1, k=2, stride=2, pad=0))
        else:
            L.append(Layer("conv", slot, slot + 1, cin=cin, cout=v, k=3, stride=1, pad=1,
                           ct="ct", relu=True))
            cin = v
        slot += 1
    L.append(Layer("fc", slot, slot + 1, cin=512 * 7 * 7, cout=4096, relu=True, ct_shift=fc1_shift))
    L.append(Layer("fc", slot + 1, slot + 2, cin=4096, cout=4096, relu=True))
    L.append(Layer("fc", slot + 2, slot + 3, cin=4096, cout=n_classes, final=True))
    return L


def mobilenet_v2(n_classes: int = 10) -> List[Layer]:
    """MobileNet-V2 for 32 x 32 inputs (first convolution and first
    bottleneck stage at stride 1): stem 3x3 -> 32, inverted-residual
    bottlenecks (t, c, n, s) = (1,16,1,1) (6,24,2,1) (6,32,3,2) (6,64,4,2)
    (6,96,3,1) (6,160,3,2) (6,320,1,1), 1x1 -> 1280, global average pool,
    FC.  A bottleneck is 1x1 expand (t * cin, BN, ReLU; absent for t = 1),
    3x3 depthwise (BN, ReLU), 1x1 project (BN, no activation), plus the
    block input when the stride is 1 and cin == cout.  ReLU stands for the
    ReLU6 of the original network (Sec. II-A: ReLU6 would saturate the
    checksum).  Roles: a block with a residual input gets no carry-through
    filter on its first convolution (Sec. II-A); depthwise layers have the
    role "pass" (their checksum group sees only the incoming checksum)."""
    L: List[Layer] = []
    slot = 0

    def new() -> int:
        nonlocal slot
        slot += 1
        return slot

    s1 = new()
    L.append(Layer("conv", 0, s1, cin=3, cout=32, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True))
    x, cin = s1, 32
    for t, c, n, s in ((1, 16, 1, 1), (6, 24, 2, 1), (6, 32, 3, 2), (6, 64, 4, 2), (6, 96, 3, 1),
                       (6, 160, 3, 2), (6, 320, 1, 1)):
        for i in range(n):
            stride = s if i == 0 else 1
            residual = stride == 1 and cin == c
            h, hid = x, cin
            first = True
            if t != 1:
                hid = t * cin
                e = new()
                L.append(Layer("conv", x, e, cin=cin, cout=hid, k=1, stride=1, pad=0,
                               ct="none" if residual else "ct", bn=True, relu=True))
                h, first = e, False
            d = new()
            L.append(Layer("conv", h, d, cin=hid, cout=hid, k=3, stride=stride, pad=1,
                           ct="pass", bn=True, relu=True, groups=hid))
            y = new()
            L.append(Layer("conv", d, y, cin=hid, cout=c, k=1, stride=1, pad=0, ct="ct", bn=True,
                           relu=False, res=x if residual else -1))
            assert not (first and residual)
            x, cin = y, c
    f = new()
    L.append(Layer("conv", x, f, cin=cin, cout=1280, k=1, stride=1, pad=0, ct="ct", bn=True, relu=True))
    g = new()
    L.append(Layer("gap", f, g))
    o = new()
    L.append(Layer("fc", g, o, cin=1280, cout=n_classes, final=True))
    return L


WORKLOADS: Dict[str, Workload] = {
    "lenet5": Workload("lenet5", lenet5(), (1, 28, 28), 10, 64, "fp32", 0, "uniform01",
                       calib_seed=100),
    "resnet18_cifar": Workload("resnet18_cifar", resnet18(False, 10), (3, 32, 32), 10, 128,
                               "fp32", 1, "normal", calib_seed=101),
    "resnet18_imagenet": Workload("resnet18_imagenet", resnet18(True, 1000), (3, 224, 224), 1000,
                                  256, "fp16", 2, "normal", calib_seed=102),
    # The FC1 carry-through neuron sums 25,088 + 49 inputs and reaches ~3e5 on
    # these weights, beyond the fp16 range; its coefficient is 2**-4.
    "vgg16": Workload("vgg16", vgg16(1000, fc1_shift=4), (3, 224, 224), 1000, 64, "fp16", 3,
                      "normal", calib_seed=103),
    "campaign_resnet18_cifar": Workload("campaign_resnet18_cifar", resnet18(False, 10),
                                        (3, 32, 32), 10, 128, "fp32", 5, "normal",
                                        calib_seed=105),
    "mobilenetv2_cifar": Workload("mobilenetv2_cifar", mobilenet_v2(10), (3, 32, 32), 10, 128,
                                  "fp32", 6, "normal", calib_seed=106),
}


def workload(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    if not overrides:
        return w
    d = dict(w.__dict__)
    d.update(overrides)
    return Workload(**d)


def shapes(layers: List[Layer], in_shape: tuple) -> Dict[int, tuple]:
    """Data-channel shape (C, H, W) of every slot; fc/gap outputs are (C, 1, 1)."""
    sh = {0: tuple(in_shape)}
    for L in layers:
        C, H, W = sh[L.src]
        if L.op == "conv":
            P = (H + 2 * L.pad - L.k) // L.stride + 1
            Q = (W + 2 * L.pad - L.k) // L.stride + 1
            sh[L.dst] = (L.cout, P, Q)
        elif L.op == "maxpool":
            sh[L.dst] = (C, (H + 2 * L.pad - L.k) // L.stride + 1, (W + 2 * L.pad - L.k) // L.stride + 1)
        elif L.op == "gap":
            sh[L.dst] = (C, 1, 1)
        elif L.op == "fc":
            sh[L.dst] = (L.cout, 1, 1)
        else:
            raise ValueError(L.op)
    return sh


# --------------------------------------------------------------------------
# Parameters and inputs
# --------------------------------------------------------------------------

def make_params(layers: List[Layer], seed: int) -> List[Dict[str, np.ndarray]]:
    """Seeded float32 parameters, one dict per layer (empty for pools).

    conv: "w" [cout, cin / groups, k, k] Kaiming-normal (std sqrt(2/fan_in)),
          "b" zeros [cout]; with bn also "gamma" U[0.9,1.1], "beta" N(0,0.1^2),
          "mean" N(0,0.1^2), "var" U[1,2] (all [cout]).
    fc:   "w" [cout, cin] Kaiming-normal (std sqrt(2/cin)), "b" zeros [cout].
    """
    out: List[Dict[str, np.ndarray]] = []
    for li, L in enumerate(layers):
        st = 16 * (li + 1)
        p: Dict[str, np.ndarray] = {}
        if L.op == "conv":
            cg = L.cin // L.groups                 # input channels each filter reads
            fan = cg * L.k * L.k
            n = L.cout * fan
            p["w"] = (normal(seed, st, n) * math.sqrt(2.0 / fan)).astype(np.float32).reshape(
                L.cout, cg, L.k, L.k)
            p["b"] = np.zeros(L.cout, np.float32)
            if L.bn:
                p["gamma"] = (0.9 + 0.2 * uniform(seed, st + 1, L.cout)).astype(np.float32)
                p["beta"] = (0.1 * normal(seed, st + 2, L.cout)).astype(np.float32)
                p["mean"] = (0.1 * normal(seed, st + 3, L.cout)).astype(np.float32)
                p["var"] = (1.0 + uniform(seed, st + 4, L.cout)).astype(np.float32)
        elif L.op == "fc":
            n = L.cout * L.cin
            p["w"] = (normal(seed, st, n) * math.sqrt(2.0 / L.cin)).astype(np.float32).reshape(
                L.cout, L.cin)
            p["b"] = np.zeros(L.cout, np.float32)
        out.append(p)
    return out


def make_input(w: Workload, batch: Optional[int] = None, seed: Optional[int] = None,
               first: int = 0) -> np.ndarray:
    """float32 NCHW batch of images ``first .. first+batch-1`` of the seeded set.

    Image i of a set depends only on (seed, i), so a slice of a large batch
    equals the same images generated on their own.
    """
    B = w.batch if batch is None else batch
    s = w.seed if seed is None else seed
    C, H, W = w.in_shape
    n = C * H * W
    imgs = np.empty((B, C, H, W), np.float32)
    for j in range(B):
        i = first + j
        if w.input_kind == "uniform01":
            v = uniform(s, 1_000_000 + i, n)
        else:
            v = normal(s, 1_000_000 + i, n)
        imgs[j] = v.astype(np.float32).reshape(C, H, W)
    return imgs


# --------------------------------------------------------------------------
# Fault sites
# --------------------------------------------------------------------------

def draw_faults(buffers: List[tuple], n: int, seed: int) -> np.ndarray:
    """Draw n fault sites uniformly over the union of (element, bit) pairs.

    ``buffers`` is a list of (kind, layer, n_elements, bits_per_element) with
    kind 0 = weight, 1 = activation.  Returns an int64 array [n, 4] of
    (kind, layer, element, bit).  Draws use 64-bit integers reduced modulo
    the total, whose bias (< total / 2**64) is negligible.
    """
    sizes = np.array([b[2] * b[3] for b in buffers], dtype=np.int64)
    cum = np.cumsum(sizes)
    total = int(cum[-1])
    raw = splitmix64_stream(seed, 777, n)
    pos = (raw % np.uint64(total)).astype(np.int64)
    which = np.searchsorted(cum, pos, side="right")
    start = np.concatenate([[0], cum[:-1]])
    off = pos - start[which]
    bits = np.array([b[3] for b in buffers], dtype=np.int64)[which]
    out = np.empty((n, 4), np.int64)
    out[:, 0] = np.array([b[0] for b in buffers], dtype=np.int64)[which]
    out[:, 1] = np.array([b[1] for b in buffers], dtype=np.int64)[which]
    out[:, 2] = off // bits
    out[:, 3] = off % bits
    return out
