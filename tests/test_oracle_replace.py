"""Pins of the replace-mode oracle (Sec. II-A, the paper's own construction).

The pruned index is checked against L1 norms worked out by hand; the
constructed network against the widened construction, which is pinned on
its own in test_oracle.py: replace mode is the widened scheme applied to the
network with the pruned channels removed, so on finite values both give the
same logits and S (the test removes the channels with its own slicing).
"""
import numpy as np
import pytest

import oracle
from oracle import replace as orep
from synth import Layer


def _conv_p(w, b=None):
    w = np.asarray(w, np.float32)
    return {"w": w, "b": np.zeros(w.shape[0], np.float32) if b is None else np.asarray(b, np.float32)}


def _fc_p(w, b=None):
    w = np.asarray(w, np.float32)
    return {"w": w, "b": np.zeros(w.shape[0], np.float32) if b is None else np.asarray(b, np.float32)}


def test_pruned_index_is_the_smallest_combined_l1_norm_by_hand():
    # conv A: 1 -> 3 channels (1x1), conv B: 3 -> 2 (1x1), gap, final FC 2 -> 2
    layers = [Layer("conv", 0, 1, cin=1, cout=3, k=1, ct="ct"),
              Layer("conv", 1, 2, cin=3, cout=2, k=1, ct="ct"),
              Layer("gap", 2, 3),
              Layer("fc", 3, 4, cin=2, cout=2, final=True)]
    wa = np.array([[[[4.]]], [[[-1.]]], [[[2.]]]])                 # |rows| = 4, 1, 2
    wb = np.array([[[[1.]], [[-3.]], [[1.]]],
                   [[[2.]], [[1.]], [[-1.]]]])                      # |cols| = 3, 4, 2
    wf = np.array([[1., -5.], [2., 1.]])                             # |cols| = 3, 6
    params = [_conv_p(wa), _conv_p(wb), {}, _fc_p(wf)]
    pj = orep.prune_indices(layers, params, (1, 2, 2))
    st = orep.streams(layers)
    # channel scores of slot 1: 4+3, 1+4, 2+2 -> channel 2 (score 4)
    assert pj[st[1]] == 2
    # slots 2 and 3 share a stream (gap keeps channels): 2-row norms of wb
    # (5, 4) + final-FC columns (3, 6) -> 8, 10 -> channel 0
    assert st[2] == st[3] and pj[st[2]] == 0
    assert st[0] not in pj and st[4] not in pj
    net = orep.build_replace(layers, params, "fp64", in_shape=(1, 2, 2), n_classes=2)
    A, B, F = net.layers[0], net.layers[1], net.layers[3]
    # A: rows 0, 1 kept, carry-through filter last (the image is not pruned)
    assert np.array_equal(A.W[:, :, 0, 0], [[4.], [-1.], [1.]])
    # B: row 0 pruned; kept row 1 loses input 2 and gets the zero checksum
    # slice; last row is the carry-through filter over all three inputs
    assert np.array_equal(B.W[:, :, 0, 0], [[2., 1., 0.], [1., 1., 1.]])
    # final FC: input 0 pruned, the checksum feature (last) is 0 for classes;
    # the accumulated-checksum neuron sums both features
    assert np.array_equal(F.W, [[-5., 0.], [1., 0.], [1., 1.]])


def test_one_index_per_residual_stream():
    # stem 1 -> 3, block conv1 3 -> 3 (no filter), conv2 3 -> 3 with the
    # stem's output as residual: slots 1 and 3 form one stream
    layers = [Layer("conv", 0, 1, cin=1, cout=3, k=1, ct="ct"),
              Layer("conv", 1, 2, cin=3, cout=3, k=1, ct="none"),
              Layer("conv", 2, 3, cin=3, cout=3, k=1, ct="ct", res=1),
              Layer("gap", 3, 4),
              Layer("fc", 4, 5, cin=3, cout=2, final=True)]
    w0 = np.array([1., 5., 5.]).reshape(3, 1, 1, 1)                 # stem rows: 1, 5, 5
    w1 = np.array([[5., 1., 0.], [5., 1., 0.], [0., 0., 1.]]).reshape(3, 3, 1, 1)
    # conv1 reads the stream (cols 10, 2, 1) and writes slot 2 (rows 6, 6, 1)
    w2 = np.array([[1., 0., 0.], [0., 1., 1.], [0., 0., 9.]]).reshape(3, 3, 1, 1)
    # conv2 reads slot 2 (cols 1, 1, 10) and writes the stream (rows 1, 2, 9)
    wf = np.array([[0., 1., 0.], [0., 0., 1.]])                      # reads the stream: 0, 1, 1
    params = [_conv_p(w0), _conv_p(w1), _conv_p(w2), {}, _fc_p(wf)]
    st = orep.streams(layers)
    assert st[1] == st[3] == st[4] and st[2] != st[1]
    pj = orep.prune_indices(layers, params, (1, 1, 1))
    # stream: writers 1+1, 5+2, 5+9 ; readers 10+0, 2+1, 1+1 -> 12, 10, 16.
    # No single writer or reader picks channel 1: the stem and conv2's rows
    # alone pick 0, conv1's columns 2, the classifier's columns 0.
    assert pj[st[1]] == 1
    # slot 2: conv1 rows 6, 6, 1 + conv2 cols 1, 1, 10 -> 7, 7, 11: a tie, lowest index
    assert pj[st[2]] == 0
    net = orep.build_replace(layers, params, "fp64", in_shape=(1, 1, 1), n_classes=2)
    c1 = net.layers[1]
    # block conv1: last output channel all zero (no carry-through filter)
    assert not c1.W[2].any()


def _prune_params(layers, params, pj, st, shp):
    """The widened construction's input: each pruned channel removed from
    its writers (rows, bias, BatchNorm) and readers (input slices)."""
    new_layers, new_params = [], []
    for L, P in zip(layers, params):
        jo = pj.get(st[L.dst])
        ji = pj.get(st[L.src])
        q = {k: v.copy() for k, v in P.items()}
        kw = dict(L.__dict__)
        if L.op == "conv":
            if ji is not None:
                q["w"] = np.delete(q["w"], ji, axis=1)
                kw["cin"] = L.cin - 1
            if jo is not None:
                q["w"] = np.delete(q["w"], jo, axis=0)
                for k in ("b", "gamma", "beta", "mean", "var"):
                    if k in q:
                        q[k] = np.delete(q[k], jo)
                kw["cout"] = L.cout - 1
        elif L.op == "fc":
            C, H, W = shp[L.src]
            w = q["w"].reshape(L.cout, C, H * W)
            if ji is not None:
                w = np.delete(w, ji, axis=1)
            q["w"] = w.reshape(L.cout, -1)
            kw["cin"] = q["w"].shape[1]
            if jo is not None and not L.final:
                q["w"] = np.delete(q["w"], jo, axis=0)
                q["b"] = np.delete(q["b"], jo)
                kw["cout"] = L.cout - 1
        new_layers.append(Layer(**kw))
        new_params.append(q)
    return new_layers, new_params


@pytest.mark.parametrize("net_kind", ["resnet", "lenet"])
def test_replace_equals_widened_construction_on_pruned_network(net_kind):
    rng = np.random.default_rng(3)
    if net_kind == "resnet":
        layers = [Layer("conv", 0, 1, cin=3, cout=6, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True),
                  Layer("conv", 1, 2, cin=6, cout=6, k=3, stride=1, pad=1, ct="none", bn=True, relu=True),
                  Layer("conv", 2, 3, cin=6, cout=6, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True, res=1),
                  Layer("conv", 3, 4, cin=6, cout=8, k=3, stride=2, pad=1, ct="none", bn=True, relu=True),
                  Layer("conv", 3, 5, cin=6, cout=8, k=1, stride=2, pad=0, ct="pass", bn=True),
                  Layer("conv", 4, 6, cin=8, cout=8, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True, res=5),
                  Layer("gap", 6, 7),
                  Layer("fc", 7, 8, cin=8, cout=5, final=True)]
        in_shape = (3, 8, 8)
    else:
        layers = [Layer("conv", 0, 1, cin=1, cout=4, k=3, stride=1, pad=0, ct="ct", relu=True),
                  Layer("maxpool", 1, 2, k=2, stride=2),
                  Layer("conv", 2, 3, cin=4, cout=5, k=3, stride=1, pad=0, ct="ct", relu=True),
                  Layer("fc", 3, 4, cin=5 * 2 * 2, cout=7, relu=True),
                  Layer("fc", 4, 5, cin=7, cout=3, final=True)]
        in_shape = (1, 10, 10)
    params = []
    for L in layers:
        p = {}
        if L.op == "conv":
            p["w"] = rng.normal(size=(L.cout, L.cin, L.k, L.k)).astype(np.float32)
            p["b"] = rng.normal(size=L.cout).astype(np.float32)
            if L.bn:
                p["gamma"] = rng.uniform(0.5, 1.5, L.cout).astype(np.float32)
                p["beta"] = rng.normal(size=L.cout).astype(np.float32)
                p["mean"] = rng.normal(size=L.cout).astype(np.float32)
                p["var"] = rng.uniform(0.5, 2.0, L.cout).astype(np.float32)
        elif L.op == "fc":
            p["w"] = rng.normal(size=(L.cout, L.cin)).astype(np.float32)
            p["b"] = rng.normal(size=L.cout).astype(np.float32)
        params.append(p)
    x = rng.normal(size=(3,) + in_shape)
    net_r = orep.build_replace(layers, params, "fp64", in_shape=in_shape, n_classes=layers[-1].cout)
    st = orep.streams(layers)
    pj = orep.prune_indices(layers, params, in_shape)
    shp = orep._channels_and_hw(layers, in_shape)
    pl, pp = _prune_params(layers, params, pj, st, shp)
    in_c = in_shape[0]
    net_a = oracle.build(pl, pp, "fp64", True, in_shape=(in_c,) + in_shape[1:], n_classes=layers[-1].cout)
    o_r = oracle.forward(net_r, x, keep=True)
    o_a = oracle.forward(net_a, x)
    assert np.allclose(o_r["logits"], o_a["logits"], rtol=1e-12, atol=1e-12)
    assert np.allclose(o_r["S"], o_a["S"], rtol=1e-12, atol=1e-12)
    # the checksum channel is the last one of every pruned tensor: in the
    # stream after the first CT convolution it equals the centre-tap channel
    # sum of that convolution's input (ReLU of a sum of ReLU outputs is the sum)
    first = layers[0]
    a0 = o_r["acts"][0]
    if first.k == 3 and first.pad == 1:
        xin = oracle.round_to(x[0], "fp64")
        ctr = xin.sum(axis=0)                       # stride 1, pad 1: the centre is the pixel itself
        assert np.allclose(a0[first.dst][-1], np.maximum(ctr, 0.0), rtol=1e-12, atol=1e-12)
