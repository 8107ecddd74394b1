"""CPU oracle for the carry-through checksum method -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It shares no code with the CUDA path;
the only common module is ``synth`` (seeded shapes, parameters and inputs,
which holds none of the method's arithmetic).

What it computes, in the paper's own layout (the checksum is the LAST
channel of every feature map that carries one):

* Carry-through filter (Sec. II-A, Fig. 1): an extra output filter that is 0
  everywhere except a 1 at the kernel centre, repeated over every input
  channel, so the new output channel is the channel-wise sum of the
  co-located input values.  This build APPENDS it as output channel C_out
  (the widened variant); data filters are unchanged.
* Input-channel level (Sec. II-A): in every data filter the 2-D slice that
  multiplies the incoming checksum channel is zero.
* Residual networks (Sec. II-A, last paragraph): the first convolution of a
  residual block gets no carry-through filter, so its input is not summed
  twice; a 1x1 downsample shortcut passes the incoming checksum through
  (weight 1 on the checksum input only), or drops it when built with
  ``ds_mode="zero"``.
* BatchNorm (Eq. 1): folded into the convolution; on the checksum channel it
  is the identity (scale exactly 1, bias 0).
* FC layers (Sec. II-A, end of "input-channel level"): a hidden FC layer gets
  one extra neuron whose weights are all 1; the final FC layer gets the
  accumulated-checksum neuron S, weight 1 on every input (Sec. II-B).
* Detection (Sec. II-B): flag an image when |S - r| > tau (NaN or inf S is
  flagged); r and tau come from the distribution-based rule of Sec. II-C:
  r = mean of fault-free S, tau = the nearest-rank (1 - alpha) quantile of
  |S - r| over a fault-free calibration set.
* Faults (Sec. III-A): single bit flips in the stored word of a convolution
  weight or of a convolution's input activation, transient, one per run.

Arithmetic: every convolution and FC sum accumulates in IEEE double
(``conv_ref.c``); values are rounded to the storage precision (fp32 or fp16,
round-to-nearest-even) where the tensor is stored: after each convolution
epilogue (bias, residual add, ReLU), after each hidden FC layer; max-pool is
exact on stored values; the global average pool and the final FC layer
produce fp32.  Biases are stored in fp32 in every precision.  Precision
"fp64" rounds nowhere (used by the exact pins).

Readings of points the paper leaves open are stated next to the code that
takes them.  The paper's own replace-mode construction (prune the least
important channel and put the carry-through filter in its place) is in
``oracle/replace.py``.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence

import numpy as np

import synth

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "_conv_ref.so")
_lib = None


def build_lib(force: bool = False) -> str:
    """Compile conv_ref.c into _conv_ref.so next to it (gcc, OpenMP)."""
    src = os.path.join(_HERE, "conv_ref.c")
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(src):
        tmp = _SO + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-O3", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
                               "-o", tmp, src])
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    if _lib is None:
        build_lib()
        lib = ctypes.CDLL(_SO)
        dp = ctypes.POINTER(ctypes.c_double)
        up = ctypes.POINTER(ctypes.c_ubyte)
        lib.or_conv2d.argtypes = [dp, ctypes.c_int, ctypes.c_int, ctypes.c_int, dp, up,
                                  ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                  ctypes.c_int, ctypes.c_int, ctypes.c_int, dp]
        lib.or_conv2d.restype = None
        lib.or_set_threads.argtypes = [ctypes.c_int]
        lib.or_get_threads.restype = ctypes.c_int
        _lib = lib
    return _lib


def set_threads(n: int) -> None:
    _load().or_set_threads(int(n))


def get_threads() -> int:
    return int(_load().or_get_threads())


# ---------------------------------------------------------------------------
# Primitives
# ---------------------------------------------------------------------------

def round_to(x, prec: str) -> np.ndarray:
    """Round float64 values to the storage precision (nearest-even).  Values
    beyond the format's range become +-inf, as in the stored tensors (bit
    flips in exponents produce them on purpose), without a warning."""
    x = np.asarray(x, dtype=np.float64)
    if prec == "fp64":
        return x.copy()
    with np.errstate(over="ignore"):
        if prec == "fp32":
            return x.astype(np.float32).astype(np.float64)
        if prec == "fp16":
            return x.astype(np.float16).astype(np.float64)
    raise ValueError(prec)


def bits_of(prec: str) -> int:
    return {"fp16": 16, "fp32": 32, "fp64": 64}[prec]


def flip_bit(value: float, bit: int, prec: str) -> float:
    """The value whose storage word is ``value``'s word with ``bit`` inverted."""
    if prec == "fp16":
        u = np.array([value], dtype=np.float16).view(np.uint16)
        u ^= np.uint16(1 << bit)
        return float(u.view(np.float16)[0])
    if prec == "fp32":
        u = np.array([value], dtype=np.float32).view(np.uint32)
        u ^= np.uint32(1 << bit)
        return float(u.view(np.float32)[0])
    u = np.array([value], dtype=np.float64).view(np.uint64)
    u ^= np.uint64(1 << bit)
    return float(u.view(np.float64)[0])


def conv2d(x: np.ndarray, w: np.ndarray, skip: Optional[np.ndarray], stride: int, pad: int) -> np.ndarray:
    """Direct convolution of one image x [C, H, W] with w [K, C, R, S] (double)."""
    lib = _load()
    x = np.ascontiguousarray(x, dtype=np.float64)
    w = np.ascontiguousarray(w, dtype=np.float64)
    C, H, W = x.shape
    K, C2, R, S = w.shape
    assert C2 == C, (C2, C)
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    y = np.empty((K, P, Q), np.float64)
    dp = ctypes.POINTER(ctypes.c_double)
    if skip is not None:
        skip = np.ascontiguousarray(skip, dtype=np.uint8)
        sp = skip.ctypes.data_as(ctypes.POINTER(ctypes.c_ubyte))
    else:
        sp = ctypes.POINTER(ctypes.c_ubyte)()
    lib.or_conv2d(x.ctypes.data_as(dp), C, H, W, w.ctypes.data_as(dp), sp, K, R, S, stride, pad,
                  P, Q, y.ctypes.data_as(dp))
    return y


def depthwise2d(x: np.ndarray, w: np.ndarray, skip: Optional[np.ndarray], stride: int, pad: int) -> np.ndarray:
    """Depthwise convolution of one image x [C, H, W] with w [C, 1, R, S]
    (double): output channel c is the correlation of input channel c with
    its filter, taps added in (r, s) order; skipped taps are not multiplied."""
    C, H, W = x.shape
    K, one, R, S = w.shape
    assert K == C and one == 1, (w.shape, x.shape)
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    xp = np.zeros((C, H + 2 * pad, W + 2 * pad))
    xp[:, pad:pad + H, pad:pad + W] = x
    y = np.zeros((C, P, Q))
    for r in range(R):
        for s_ in range(S):
            win = xp[:, r:r + stride * (P - 1) + 1:stride, s_:s_ + stride * (Q - 1) + 1:stride]
            tap = w[:, 0, r, s_].astype(np.float64)
            if skip is not None:
                tap = np.where(skip[:, 0, r, s_] != 0, 0.0, tap)
                live = skip[:, 0, r, s_] == 0
                y[live] += tap[live, None, None] * win[live]
            else:
                y += tap[:, None, None] * win
    return y


def relu(y: np.ndarray) -> np.ndarray:
    """max(y, 0) that keeps NaN (and -0.0) as they are: y < 0 -> +0."""
    return np.where(y < 0, 0.0, y)


def maxpool(x: np.ndarray, k: int, s: int, p: int) -> np.ndarray:
    """k x k max-pool of [C, H, W]; padding never wins; any NaN in a window gives NaN."""
    C, H, W = x.shape
    P = (H + 2 * p - k) // s + 1
    Q = (W + 2 * p - k) // s + 1
    xp = np.full((C, H + 2 * p, W + 2 * p), -np.inf)
    xp[:, p:p + H, p:p + W] = x
    y = np.full((C, P, Q), -np.inf)
    for i in range(k):
        for j in range(k):
            win = xp[:, i:i + s * (P - 1) + 1:s, j:j + s * (Q - 1) + 1:s]
            y = np.maximum(y, win)          # np.maximum propagates NaN
    return y


def fold_bn(w: np.ndarray, b: np.ndarray, p: Dict[str, np.ndarray], eps: float):
    """Eq. 1 folded into the preceding convolution, in double."""
    scale = p["gamma"].astype(np.float64) / np.sqrt(p["var"].astype(np.float64) + eps)
    wf = w.astype(np.float64) * scale[:, None, None, None]
    bf = (b.astype(np.float64) - p["mean"].astype(np.float64)) * scale + p["beta"].astype(np.float64)
    return wf, bf


# ---------------------------------------------------------------------------
# The augmented network in the paper's literal layout
# ---------------------------------------------------------------------------

@dataclass
class OLayer:
    op: str
    src: int
    dst: int
    res: int = -1
    relu: bool = False
    final: bool = False
    stride: int = 1
    pad: int = 0
    k: int = 1
    ct: str = "none"
    groups: int = 1                     # > 1: depthwise (W is [K_tot, 1, k, k])
    W: Optional[np.ndarray] = None      # literal weights (float64 holding storage values)
    skip: Optional[np.ndarray] = None   # structural zeros of the construction
    b: Optional[np.ndarray] = None      # fp32 biases as float64
    n_data_out: int = 0                 # data output channels / neurons
    has_ct_out: bool = False            # an extra output channel / neuron exists


@dataclass
class ONet:
    layers: List[OLayer]
    prec: str
    protected: bool
    in_shape: tuple
    n_classes: int
    has_cs: Dict[int, bool]
    n_data: Dict[int, int]              # data channels per slot


def build(layers: Sequence[synth.Layer], params, prec: str, protected: bool = True,
          ds_mode: str = "pass", bn_eps: float = 1e-5, in_shape=None, n_classes=None) -> ONet:
    """Construct the (un)protected network; weights rounded to ``prec``."""
    has_cs = {0: False}
    n_data = {0: in_shape[0] if in_shape else None}
    out: List[OLayer] = []
    for L, P in zip(layers, params):
        if L.op == "conv" and L.groups > 1:
            # Depthwise (reading: the paper builds the carry-through filter for
            # dense convolutions only).  The checksum is one more group: its
            # filter sees only the incoming checksum channel, so it passes the
            # checksum through at the centre tap (weight 1); off-centre taps
            # of that filter are structural zeros.  Without an incoming
            # checksum there is nothing to pass.
            assert L.groups == L.cin == L.cout
            cs_in = has_cs[L.src]
            w = P["w"].astype(np.float64)
            b = P["b"].astype(np.float64)
            if L.bn:
                w, b = fold_bn(w, b, P, bn_eps)
            w = round_to(w, prec)
            b = round_to(b, "fp32") if prec != "fp64" else b
            passes = protected and cs_in and L.ct != "none"
            K = L.cout + (1 if passes else 0)
            W = np.zeros((K, 1, L.k, L.k))
            skip = np.zeros((K, 1, L.k, L.k), dtype=np.uint8)
            W[:L.cout] = w
            ctr = (L.k - 1) // 2
            if passes:
                skip[L.cout] = 1
                skip[L.cout, 0, ctr, ctr] = 0
                W[L.cout, 0, ctr, ctr] = 1.0
            bb = np.zeros(K)
            bb[:L.cout] = b
            has_cs[L.dst] = passes
            n_data[L.dst] = L.cout
            out.append(OLayer("conv", L.src, L.dst, res=L.res, relu=L.relu, stride=L.stride,
                              pad=L.pad, k=L.k, ct="pass" if passes else "none", groups=L.groups, W=W,
                              skip=skip, b=bb, n_data_out=L.cout, has_ct_out=passes))
        elif L.op == "conv":
            ct = L.ct if protected else "none"
            if ct == "pass" and ds_mode == "zero":
                ct = "none"
            cs_in = has_cs[L.src]
            w = P["w"].astype(np.float64)
            b = P["b"].astype(np.float64)
            if L.bn:
                w, b = fold_bn(w, b, P, bn_eps)
            w = round_to(w, prec)
            b = round_to(b, "fp32") if prec != "fp64" else b
            K = L.cout + (1 if ct in ("ct", "pass") else 0)
            C = L.cin + (1 if cs_in else 0)
            W = np.zeros((K, C, L.k, L.k))
            skip = np.zeros((K, C, L.k, L.k), dtype=np.uint8)
            W[:L.cout, :L.cin] = w
            if cs_in:
                # input-channel level: the data filters do not see the checksum
                skip[:L.cout, L.cin] = 1
            ctr = (L.k - 1) // 2           # centre tap (reading for k != 3)
            coef = 2.0 ** (-L.ct_shift)
            if ct == "ct":
                skip[L.cout] = 1
                skip[L.cout, :, ctr, ctr] = 0
                W[L.cout, :, ctr, ctr] = coef   # every input channel, checksum included
            elif ct == "pass":
                skip[L.cout] = 1
                if cs_in:
                    skip[L.cout, L.cin, ctr, ctr] = 0
                    W[L.cout, L.cin, ctr, ctr] = 1.0
            bb = np.zeros(K)
            bb[:L.cout] = b                     # checksum bias 0 (BN identity)
            res_cs = has_cs[L.res] if L.res >= 0 else False
            has_cs[L.dst] = (ct in ("ct", "pass")) or res_cs
            n_data[L.dst] = L.cout
            out.append(OLayer("conv", L.src, L.dst, res=L.res, relu=L.relu, stride=L.stride,
                              pad=L.pad, k=L.k, ct=ct, W=W, skip=skip, b=bb, n_data_out=L.cout,
                              has_ct_out=ct in ("ct", "pass")))
        elif L.op in ("maxpool", "gap"):
            has_cs[L.dst] = has_cs[L.src]
            n_data[L.dst] = n_data[L.src]
            out.append(OLayer(L.op, L.src, L.dst, k=L.k, stride=L.stride, pad=L.pad))
        elif L.op == "fc":
            cs_in = has_cs[L.src]
            n_in_data = L.cin
            # checksum inputs = the checksum plane of the source, flattened
            n_cs = 0
            if cs_in:
                n_cs = L.cin // n_data[L.src]   # H*W of the source map
            w = round_to(P["w"].astype(np.float64), prec)
            b = P["b"].astype(np.float64)
            b = round_to(b, "fp32") if prec != "fp64" else b
            ct_row = protected
            K = L.cout + (1 if ct_row else 0)
            C = n_in_data + n_cs
            W = np.zeros((K, C))
            skip = np.zeros((K, C), dtype=np.uint8)
            W[:L.cout, :n_in_data] = w
            skip[:L.cout, n_in_data:] = 1
            if ct_row:
                W[L.cout, :] = 2.0 ** (-L.ct_shift)
            bb = np.zeros(K)
            bb[:L.cout] = b
            has_cs[L.dst] = ct_row and not L.final
            n_data[L.dst] = L.cout
            out.append(OLayer("fc", L.src, L.dst, relu=L.relu, final=L.final, W=W, skip=skip,
                              b=bb, n_data_out=L.cout, has_ct_out=ct_row))
        else:
            raise ValueError(L.op)
    return ONet(out, prec, protected, tuple(in_shape) if in_shape else None,
                n_classes, has_cs, n_data)


def build_workload(wl: synth.Workload, prec: Optional[str] = None, protected: bool = True,
                   ds_mode: str = "pass", params=None) -> ONet:
    if params is None:
        params = synth.make_params(wl.layers, wl.seed)
    return build(wl.layers, params, prec or wl.precision, protected, ds_mode, wl.bn_eps,
                 wl.in_shape, wl.n_classes)


# ---------------------------------------------------------------------------
# Forward pass, faults, verification
# ---------------------------------------------------------------------------

@dataclass
class Fault:
    kind: int          # 0 = weight of conv layer `layer`, 1 = input activation of conv `layer`
    layer: int
    element: int       # flat index into the literal layout
    bit: int


def weight_shape(net: ONet, layer: int) -> tuple:
    return net.layers[layer].W.shape


def _in_channels(net: ONet, L: OLayer) -> int:
    """Channels of a convolution's input tensor, checksum included."""
    if L.groups > 1:
        return net.n_data[L.src] + (1 if net.has_cs[L.src] else 0)
    return L.W.shape[1]


def act_shape(net: ONet, layer: int, batch: int) -> tuple:
    """Literal layout [B, C_tot, H, W] of the input tensor of conv ``layer``."""
    L = net.layers[layer]
    assert L.op == "conv"
    H, W = slot_hw(net)[L.src]
    return (batch, _in_channels(net, L), H, W)


def slot_hw(net: ONet) -> Dict[int, tuple]:
    hw = {0: net.in_shape[1:]}
    for L in net.layers:
        H, W = hw[L.src]
        if L.op == "conv":
            hw[L.dst] = ((H + 2 * L.pad - L.k) // L.stride + 1, (W + 2 * L.pad - L.k) // L.stride + 1)
        elif L.op == "maxpool":
            hw[L.dst] = ((H + 2 * L.pad - L.k) // L.stride + 1, (W + 2 * L.pad - L.k) // L.stride + 1)
        else:
            hw[L.dst] = (1, 1)
    return hw


def fault_buffers(net: ONet, batch: int, include_input: bool = False) -> List[tuple]:
    """(kind, layer, n_elements, bits) of every fault-able buffer (literal layout).

    Weight buffers: every convolution's literal weight tensor.  Activation
    buffers: every distinct tensor that a convolution reads, addressed by the
    first convolution that reads it; the network input is left out unless
    ``include_input``.
    """
    bits = bits_of(net.prec)
    hw = slot_hw(net)
    bufs = []
    for i, L in enumerate(net.layers):
        if L.op == "conv":
            bufs.append((0, i, int(L.W.size), bits))
    seen = set()
    for i, L in enumerate(net.layers):
        if L.op == "conv" and L.src not in seen:
            seen.add(L.src)
            if L.src == 0 and not include_input:
                continue
            C = _in_channels(net, L)
            H, W = hw[L.src]
            bufs.append((1, i, int(batch * C * H * W), bits))
    return bufs


def forward(net: ONet, x: np.ndarray, fault: Optional[Fault] = None, keep: bool = False):
    """Run a batch x [B, C, H, W]; returns dict(logits [B, n], S [B], acts?)."""
    B = x.shape[0]
    logits, S, acts_all = [], [], []
    prec = net.prec
    layers = net.layers
    wfault_layer = None
    if fault is not None and fault.kind == 0:
        L = layers[fault.layer]
        W = L.W.copy()
        sk = L.skip.copy()
        flat = W.reshape(-1)
        old = flat[fault.element]
        flat[fault.element] = flip_bit(old, fault.bit, prec)
        sk.reshape(-1)[fault.element] = 0            # a faulted zero is applied
        wfault_layer = (fault.layer, W, sk)
    a_slot = layers[fault.layer].src if (fault is not None and fault.kind == 1) else None
    for n in range(B):
        acts = {0: round_to(x[n], prec)}
        if a_slot == 0:
            acts[0] = _maybe_flip_act(acts[0], 0, a_slot, fault, n, prec)
        for li, L in enumerate(layers):
            if L.op == "conv":
                W, sk = L.W, L.skip
                if wfault_layer is not None and wfault_layer[0] == li:
                    W, sk = wfault_layer[1], wfault_layer[2]
                xin = acts[L.src]
                if L.groups > 1:
                    # the filters read the first K_tot input channels (the
                    # checksum filter the checksum channel, when it exists)
                    y = depthwise2d(xin[:W.shape[0]], W, sk, L.stride, L.pad) + L.b[:, None, None]
                else:
                    y = conv2d(xin, W, sk, L.stride, L.pad) + L.b[:, None, None]
                if L.res >= 0:
                    r = acts[L.res]
                    nd = L.n_data_out
                    y[:nd] += r[:nd]
                    if net.has_cs[L.res]:
                        if L.has_ct_out:
                            y[nd] += r[nd]
                        else:
                            y = np.concatenate([y, r[nd:nd + 1]], axis=0)
                if L.relu:
                    y = relu(y)
                y = round_to(y, prec)
            elif L.op == "maxpool":
                y = maxpool(acts[L.src], L.k, L.stride, L.pad)
            elif L.op == "gap":
                a = acts[L.src]
                y = a.reshape(a.shape[0], -1).mean(axis=1)[:, None, None]
                y = round_to(y, "fp32") if prec != "fp64" else y
            elif L.op == "fc":
                v = _fc_input(net, L.src, acts[L.src])
                y = conv2d(v[:, None, None], L.W[:, :, None, None], L.skip[:, :, None, None], 1, 0)
                y = y[:, 0, 0] + L.b
                if L.relu:
                    y = relu(y)
                if L.final:
                    y = round_to(y, "fp32") if prec != "fp64" else y
                else:
                    y = round_to(y, prec)
                y = y[:, None, None]
            if a_slot is not None and L.dst == a_slot:
                y = _maybe_flip_act(y, L.dst, a_slot, fault, n, prec)
            acts[L.dst] = y
        out = acts[layers[-1].dst][:, 0, 0]
        logits.append(out[:net.n_classes])
        S.append(out[net.n_classes] if net.protected else np.nan)
        if keep:
            acts_all.append(acts)
    res = {"logits": np.array(logits), "S": np.array(S)}
    if keep:
        res["acts"] = acts_all
    return res


def _fc_input(net: ONet, slot: int, a: np.ndarray) -> np.ndarray:
    """Flatten [C_tot, H, W] in (C, H, W) order: data channels, then the checksum plane."""
    return a.reshape(-1)


def _maybe_flip_act(y: np.ndarray, slot: int, target_slot: int, fault: Fault, n: int, prec: str):
    per_img = y.size
    img, off = divmod(fault.element, per_img)
    if img != n:
        return y
    y = y.copy()
    flat = y.reshape(-1)
    flat[off] = flip_bit(flat[off], fault.bit, prec)
    return y


def residual_roles(layers: Sequence[synth.Layer]) -> List[Optional[str]]:
    """Sec. II-A, residual networks: the role of each convolution that the
    network graph fixes (None for other layers).

    A tensor read by two layers reaches a later residual add along two paths
    (the block's main path and its shortcut), and its checksum arrives along
    the shortcut already.  So a convolution reading such a tensor gets no
    carry-through filter ("none"), or the checksum would be accumulated
    twice -- unless it is the shortcut itself: a convolution whose output
    goes to nothing but a residual add passes the checksum through ("pass").
    A depthwise convolution passes its incoming checksum through as well
    (its checksum group sees only the checksum channel); every other
    convolution carries a carry-through filter ("ct").
    """
    uses: Dict[int, int] = {}
    added: set = set()
    for L in layers:
        uses[L.src] = uses.get(L.src, 0) + 1
        if L.res >= 0:
            uses[L.res] = uses.get(L.res, 0) + 1
            added.add(L.res)
    out: List[Optional[str]] = []
    for L in layers:
        if L.op != "conv":
            out.append(None)
        elif uses[L.src] > 1:
            out.append("pass" if L.dst in added and uses[L.dst] == 1 else "none")
        elif L.groups > 1:
            out.append("pass")
        else:
            out.append("ct")
    return out


def top1(logits: np.ndarray) -> np.ndarray:
    """Top-1 class per row; ties go to the lowest index; any NaN gives -1."""
    logits = np.asarray(logits, dtype=np.float64)
    out = np.empty(logits.shape[0], dtype=np.int64)
    for i, row in enumerate(logits):
        if np.isnan(row).any():
            out[i] = -1
            continue
        best, bi = row[0], 0
        for j in range(1, row.shape[0]):
            if row[j] > best:
                best, bi = row[j], j
        out[i] = bi
    return out


def verdict(S: np.ndarray, r: float, tau: float) -> np.ndarray:
    """Sec. II-B: flag when the deviation of S from r exceeds tau (NaN flags)."""
    S = np.asarray(S, dtype=np.float64)
    return ~(np.abs(S - r) <= tau)


def calibrate(S: np.ndarray, alpha: float):
    """Sec. II-C distribution-based threshold: (r, tau).

    r is the mean of the fault-free S values; tau is the nearest-rank
    ceil((1 - alpha) * N)-th smallest |S - r|, so at most alpha of the
    calibration images are flagged by the strict comparison.
    """
    S = np.asarray(S, dtype=np.float64)
    assert np.isfinite(S).all()
    r = float(np.mean(S))
    dev = np.sort(np.abs(S - r))
    rank = int(math.ceil((1.0 - alpha) * len(dev)))
    rank = min(max(rank, 1), len(dev))
    return r, float(dev[rank - 1])


def fi_threshold(S: np.ndarray, critical: np.ndarray, r: float, alpha: float) -> float:
    """Sec. II-C FI-based threshold: tau such that at most alpha of the
    non-critical fault trials of a calibration campaign are flagged.

    Deviations |S - r| of the non-critical trials (a non-finite S is an
    infinite deviation); tau is their nearest-rank ceil((1 - alpha) * m)-th
    smallest value, as in calibrate().
    """
    S = np.asarray(S, dtype=np.float64)
    crit = np.asarray(critical).astype(bool)
    dev = np.abs(S[~crit] - r)
    dev = np.where(np.isfinite(dev), dev, np.inf)
    assert dev.size > 0
    dev = np.sort(dev)
    rank = int(math.ceil((1.0 - alpha) * len(dev)))
    rank = min(max(rank, 1), len(dev))
    return float(dev[rank - 1])


def detection_rates(S: np.ndarray, critical: np.ndarray, r: float, tau: float):
    """Sec. III-A metrics: (TPR, FPR, Youden's J = TPR - FPR).

    TPR = flagged fraction of critical trials, FPR = flagged fraction of
    non-critical trials, with the verdict of Sec. II-B (NOT |S - r| <= tau).
    """
    crit = np.asarray(critical).astype(bool)
    flag = verdict(np.asarray(S, dtype=np.float64), r, tau).astype(bool)
    tpr = float(flag[crit].mean()) if crit.any() else float("nan")
    fpr = float(flag[~crit].mean()) if (~crit).any() else float("nan")
    return tpr, fpr, tpr - fpr


# ---------------------------------------------------------------------------
# Second code path: the checksum recursion on the unprotected network
# ---------------------------------------------------------------------------

def closed_form_S(net_u: ONet, layers: Sequence[synth.Layer], acts_u: Dict[int, np.ndarray],
                  ds_mode: str = "pass") -> float:
    """S recomputed from the unprotected network's stored activations.

    Per carry-through layer, the checksum at output position (p, q) is the
    sum over input channels of the input at the filter centre plus the
    incoming checksum there (Sec. II-A), then the same bias (0), residual add,
    ReLU and pooling as the data; S is the sum of every input of the final
    FC layer, checksum features included (Sec. II-B).  No rounding (fp64).
    """
    cs: Dict[int, Optional[np.ndarray]] = {0: None}
    S = None
    for L in layers:
        if L.op == "conv":
            x = acts_u[L.src]
            C, H, W = x.shape
            P = (H + 2 * L.pad - L.k) // L.stride + 1
            Q = (W + 2 * L.pad - L.k) // L.stride + 1
            ctr = (L.k - 1) // 2
            coef = 2.0 ** (-L.ct_shift)
            ct = L.ct
            if ct == "pass" and ds_mode == "zero":
                ct = "none"

            def centre(plane):
                # out[p, q] = plane[p*stride + ctr - pad, q*stride + ctr - pad], 0 outside
                hs = np.arange(P) * L.stride + ctr - L.pad
                ws = np.arange(Q) * L.stride + ctr - L.pad
                okh, okw = (hs >= 0) & (hs < H), (ws >= 0) & (ws < W)
                out = np.zeros((P, Q))
                out[np.ix_(okh, okw)] = plane[np.ix_(hs[okh], ws[okw])]
                return out
            pre = None
            if ct == "ct":
                tot = x.sum(axis=0)
                if cs[L.src] is not None:
                    tot = tot + cs[L.src]
                pre = coef * centre(tot)
            elif ct == "pass":
                pre = centre(cs[L.src]) if cs[L.src] is not None else np.zeros((P, Q))
            if L.res >= 0 and cs.get(L.res) is not None:
                pre = (pre if pre is not None else 0.0) + cs[L.res]
            if pre is not None and L.relu:
                pre = relu(pre)
            cs[L.dst] = pre
        elif L.op == "maxpool":
            c = cs[L.src]
            cs[L.dst] = None if c is None else maxpool(c[None], L.k, L.stride, L.pad)[0]
        elif L.op == "gap":
            c = cs[L.src]
            cs[L.dst] = None if c is None else np.array([[c.mean()]])
        elif L.op == "fc":
            tot = acts_u[L.src].sum()
            if cs[L.src] is not None:
                tot += cs[L.src].sum()
            v = 2.0 ** (-L.ct_shift) * tot
            if L.final:
                S = v
            else:
                cs[L.dst] = np.array([[relu(np.array(v))[()]]])
    return float(S)
