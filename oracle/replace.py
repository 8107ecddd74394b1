"""Replace mode, the paper's own construction (Sec. II-A) -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may
use it.  It shares no code with the CUDA path.

Sec. II-A builds the carry-through scheme without widening the network:

* Output-channel level: in every convolution the least important output
  channel is pruned and the carry-through filter takes the freed place as
  the LAST output channel.  Importance = the combined L1 norm of the
  channel's filter in this layer and of the 2-D slices that read it in the
  next layer; the smallest is pruned.  Those next-layer slices go with it.
* Input-channel level: the incoming checksum arrives as the last input
  channel; every normal filter's slice for it is zero.  Tensor widths and
  filter depths are those of the original network.
* The first convolution of a residual block prunes a channel too but gets
  no carry-through filter: its last output channel is all zero.
* FC layers: the least important neuron is pruned and a neuron with all
  weights 1 takes its place (last); the final FC layer keeps its classes
  and gets the accumulated-checksum neuron S (weights 1) as an extra output
  (Sec. II-B).

Readings (the paper is silent on these):

* Importance uses the stored filters before BatchNorm folding, summed over
  every writer and reader of the tensor.  Tensors tied by a residual add or
  by pooling (a "stream") share one pruned index, chosen from the sum of
  the scores of all their writers and readers; ties go to the lowest index.
* A reader FC layer's slice of channel c is its H*W columns of that channel
  in the (C, H, W) flatten order.
* The 1x1 downsample shortcut's last channel passes the incoming checksum
  through (weight 1 on the last input channel at the centre), as in the
  widened construction.
* Zero slices are multiplied, not skipped: the tensors are ordinary
  tensors, as in the paper's engine, so 0 * inf = NaN can leak from an
  overflowing checksum into data channels.
* BatchNorm on the carry-through channel is the identity (scale 1, bias 0).
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence

import numpy as np

import synth

from . import OLayer, ONet, fold_bn, round_to


def streams(layers: Sequence[synth.Layer]) -> Dict[int, int]:
    """Slot -> representative slot of its stream (union over residual adds,
    max-pools and global average pools, which keep channel indices)."""
    parent: Dict[int, int] = {}

    def find(a: int) -> int:
        parent.setdefault(a, a)
        while parent[a] != a:
            parent[a] = parent[parent[a]]
            a = parent[a]
        return a

    def union(a: int, b: int) -> None:
        ra, rb = find(a), find(b)
        if ra != rb:
            parent[max(ra, rb)] = min(ra, rb)

    for L in layers:
        find(L.src)
        find(L.dst)
        if L.op == "conv" and L.res >= 0:
            union(L.dst, L.res)
        if L.op in ("maxpool", "gap"):
            union(L.dst, L.src)
    return {s: find(s) for s in parent}


def _channels_and_hw(layers: Sequence[synth.Layer], in_shape) -> Dict[int, tuple]:
    """Slot -> (channels, H, W) of the original network."""
    shp = {0: tuple(in_shape)}
    for L in layers:
        C, H, W = shp[L.src]
        if L.op == "conv":
            shp[L.dst] = (L.cout, (H + 2 * L.pad - L.k) // L.stride + 1, (W + 2 * L.pad - L.k) // L.stride + 1)
        elif L.op == "maxpool":
            shp[L.dst] = (C, (H + 2 * L.pad - L.k) // L.stride + 1, (W + 2 * L.pad - L.k) // L.stride + 1)
        elif L.op == "gap":
            shp[L.dst] = (C, 1, 1)
        else:
            shp[L.dst] = (L.cout, 1, 1)
    return shp


def prune_indices(layers: Sequence[synth.Layer], params, in_shape) -> Dict[int, int]:
    """Stream representative -> pruned channel index (Sec. II-A, importance
    by combined L1 norm).  The network input and the classifier output are
    never pruned."""
    st = streams(layers)
    shp = _channels_and_hw(layers, in_shape)
    final_dst = [L.dst for L in layers if L.op == "fc" and L.final]
    keep_out = {st[0]} | {st[d] for d in final_dst}
    score: Dict[int, np.ndarray] = {}

    def acc(slot: int, v: np.ndarray) -> None:
        r = st[slot]
        if r in keep_out:
            return
        score[r] = score.get(r, 0.0) + v

    for L, P in zip(layers, params):
        if L.op == "conv":
            w = np.abs(P["w"].astype(np.float64))          # [cout, cin, k, k]
            acc(L.dst, w.sum(axis=(1, 2, 3)))                # writer: the output filters
            acc(L.src, w.sum(axis=(0, 2, 3)))                # reader: the input slices
        elif L.op == "fc":
            w = np.abs(P["w"].astype(np.float64))          # [cout, cin]
            if not L.final:
                acc(L.dst, w.sum(axis=1))
            C, H, W = shp[L.src]
            acc(L.src, w.reshape(L.cout, C, H * W).sum(axis=(0, 2)))
    # np.argmin returns the first minimum: ties go to the lowest index
    return {r: int(np.argmin(v)) for r, v in score.items()}


def _keep(n: int, j: Optional[int]) -> List[int]:
    return [i for i in range(n) if i != j]


def build_replace(layers: Sequence[synth.Layer], params, prec: str, bn_eps: float = 1e-5,
                  in_shape=None, n_classes=None) -> ONet:
    """The replace-mode network in its stored layout (original widths, the
    checksum as the last channel of every pruned tensor); weights rounded to
    ``prec`` as in ``oracle.build``."""
    st = streams(layers)
    shp = _channels_and_hw(layers, in_shape)
    pj = prune_indices(layers, params, in_shape)
    jof = lambda slot: pj.get(st[slot])                        # noqa: E731
    out: List[OLayer] = []
    n_data = {0: in_shape[0]}
    for L, P in zip(layers, params):
        coef = 2.0 ** (-L.ct_shift)
        if L.op == "conv":
            w = P["w"].astype(np.float64)
            b = P["b"].astype(np.float64)
            if L.bn:
                w, b = fold_bn(w, b, P, bn_eps)
            w = round_to(w, prec)
            b = round_to(b, "fp32") if prec != "fp64" else b
            jo, ji = jof(L.dst), jof(L.src)
            K, C = L.cout, L.cin
            W = np.zeros((K, C, L.k, L.k))
            rows = _keep(K, jo)
            if ji is None:
                W[:K - 1] = w[rows]
            else:
                W[:K - 1, :C - 1] = w[rows][:, _keep(C, ji)]   # last input slice (checksum) = 0
            ctr = (L.k - 1) // 2
            if L.ct == "ct":
                W[K - 1, :, ctr, ctr] = coef                  # every input channel, checksum included
            elif L.ct == "pass":
                W[K - 1, C - 1, ctr, ctr] = 1.0               # the incoming checksum only
            bb = np.zeros(K)
            bb[:K - 1] = b[rows]
            n_data[L.dst] = K
            out.append(OLayer("conv", L.src, L.dst, res=L.res, relu=L.relu, stride=L.stride, pad=L.pad,
                              k=L.k, ct=L.ct, W=W, skip=np.zeros(W.shape, np.uint8), b=bb, n_data_out=K,
                              has_ct_out=False))
        elif L.op in ("maxpool", "gap"):
            n_data[L.dst] = n_data[L.src]
            out.append(OLayer(L.op, L.src, L.dst, k=L.k, stride=L.stride, pad=L.pad))
        elif L.op == "fc":
            w = round_to(P["w"].astype(np.float64), prec)
            b = P["b"].astype(np.float64)
            b = round_to(b, "fp32") if prec != "fp64" else b
            Cs, Hs, Ws = shp[L.src]
            hw = Hs * Ws
            ji = jof(L.src)
            # columns in (C, H, W) order; the pruned channel's block leaves, the
            # checksum channel's block (last) is zero in every normal row
            wc = w.reshape(L.cout, Cs, hw)
            W3 = np.zeros((L.cout, Cs, hw))
            if ji is None:
                W3[:] = wc
            else:
                W3[:, :Cs - 1] = wc[:, _keep(Cs, ji)]
            Wn = W3.reshape(L.cout, Cs * hw)
            if L.final:
                Wf = np.zeros((L.cout + 1, L.cin))
                Wf[:L.cout] = Wn
                Wf[L.cout] = coef                              # accumulated-checksum neuron
                bb = np.zeros(L.cout + 1)
                bb[:L.cout] = b
                n_out = L.cout
            else:
                jo = jof(L.dst)
                rows = _keep(L.cout, jo)
                Wf = np.zeros((L.cout, L.cin))
                Wf[:L.cout - 1] = Wn[rows]
                Wf[L.cout - 1] = coef                          # carry-through neuron
                bb = np.zeros(L.cout)
                bb[:L.cout - 1] = b[rows]
                n_out = L.cout
            n_data[L.dst] = L.cout
            out.append(OLayer("fc", L.src, L.dst, relu=L.relu, final=L.final, W=Wf,
                              skip=np.zeros(Wf.shape, np.uint8), b=bb, n_data_out=n_out,
                              has_ct_out=L.final))
        else:
            raise ValueError(L.op)
    has_cs = {s: False for s in n_data}
    return ONet(out, prec, True, tuple(in_shape), n_classes, has_cs, n_data)


def build_replace_workload(wl: synth.Workload, prec: Optional[str] = None, params=None) -> ONet:
    if params is None:
        params = synth.make_params(wl.layers, wl.seed)
    return build_replace(wl.layers, params, prec or wl.precision, wl.bn_eps, wl.in_shape, wl.n_classes)
