"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these tests compares the oracle with itself: each one checks it
against a closed form, a brute-force loop written separately, an invariant
stated in the paper, or a hand-computed value.
"""
import math
import struct

import numpy as np
import pytest

import oracle
import synth
from synth import Layer

from _cache import params as cached_params, inputs as cached_inputs


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------

def int_params(layers, seed, lo=-2, hi=2, bn=False):
    """Integer-valued parameters so that fp64 sums are exact."""
    rng = np.random.default_rng(seed)
    out = []
    for L in layers:
        p = {}
        if L.op == "conv":
            p["w"] = rng.integers(lo, hi + 1, size=(L.cout, L.cin // L.groups, L.k, L.k)).astype(np.float32)
            p["b"] = rng.integers(-2, 3, size=L.cout).astype(np.float32)
            if L.bn:
                # eps = 0, var = 4, gamma = 1: the folded scale is exactly 0.5
                p["gamma"] = np.ones(L.cout, np.float32)
                p["beta"] = rng.integers(-2, 3, size=L.cout).astype(np.float32)
                p["mean"] = rng.integers(-2, 3, size=L.cout).astype(np.float32)
                p["var"] = np.full(L.cout, 4.0, np.float32)
        elif L.op == "fc":
            p["w"] = rng.integers(lo, hi + 1, size=(L.cout, L.cin)).astype(np.float32)
            p["b"] = rng.integers(-2, 3, size=L.cout).astype(np.float32)
        out.append(p)
    return out


def brute_conv(x, w, stride, pad):
    C, H, W = x.shape
    K, _, R, S = w.shape
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    y = np.zeros((K, P, Q))
    for k in range(K):
        for p in range(P):
            for q in range(Q):
                terms = []
                for c in range(C):
                    for r in range(R):
                        for s in range(S):
                            h, ww = p * stride + r - pad, q * stride + s - pad
                            if 0 <= h < H and 0 <= ww < W:
                                terms.append(w[k, c, r, s] * x[c, h, ww])
                y[k, p, q] = math.fsum(terms)
    return y


def tiny_resnet(ds):
    """stem(ct) -> block[conv1(none), (ds), conv2(ct)+res] -> gap -> fc."""
    L = [Layer("conv", 0, 1, cin=2, cout=3, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True)]
    if ds:
        L += [Layer("conv", 1, 2, cin=3, cout=4, k=3, stride=2, pad=1, ct="none", bn=True, relu=True),
              Layer("conv", 1, 3, cin=3, cout=4, k=1, stride=2, pad=0, ct="pass", bn=True),
              Layer("conv", 2, 4, cin=4, cout=4, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True, res=3),
              Layer("gap", 4, 5), Layer("fc", 5, 6, cin=4, cout=3, final=True)]
    else:
        L += [Layer("conv", 1, 2, cin=3, cout=3, k=3, stride=1, pad=1, ct="none", bn=True, relu=True),
              Layer("conv", 2, 3, cin=3, cout=3, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True, res=1),
              Layer("gap", 3, 4), Layer("fc", 4, 5, cin=3, cout=3, final=True)]
    return L


def tiny_lenet():
    return [Layer("conv", 0, 1, cin=1, cout=2, k=3, stride=1, pad=0, ct="ct", relu=True),
            Layer("maxpool", 1, 2, k=2, stride=2),
            Layer("conv", 2, 3, cin=2, cout=3, k=3, stride=1, pad=1, ct="ct", relu=True),
            Layer("fc", 3, 4, cin=3 * 4 * 4, cout=5, relu=True),
            Layer("fc", 4, 5, cin=5, cout=3, final=True)]


# ---------------------------------------------------------------------------
# primitives
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("stride,pad", [(1, 0), (1, 1), (2, 1), (2, 2), (1, 2)])
def test_conv2d_matches_bruteforce(stride, pad):
    rng = np.random.default_rng(stride * 10 + pad)
    x = rng.standard_normal((3, 7, 6))
    w = rng.standard_normal((4, 3, 3, 3))
    y = oracle.conv2d(x, w, None, stride, pad)
    ref = brute_conv(x, w, stride, pad)
    assert y.shape == ref.shape
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("hw", [(8, 8), (7, 9), (14, 14)])
def test_strided_shortcut_reads_the_centre_tap_of_the_block_convolution(hw):
    """A 1 x 1 stride-2 convolution (pad 0) equals a 3 x 3 stride-2 pad-1
    convolution whose only non-zero tap is the centre: output (p, q) reads
    input (2p, 2q) in both, for every map size (odd ones too).  This is
    why a ResNet downsample can use its block's first convolution's
    centre-tap operand.  Checked against the brute-force loop, integers so
    that the sums are exact."""
    rng = np.random.default_rng(hw[0] * 31 + hw[1])
    x = rng.integers(-3, 4, size=(5,) + hw).astype(np.float64)
    w1 = rng.integers(-3, 4, size=(6, 5, 1, 1)).astype(np.float64)
    w3 = np.zeros((6, 5, 3, 3))
    w3[:, :, 1, 1] = w1[:, :, 0, 0]
    a = brute_conv(x, w1, 2, 0)
    b = brute_conv(x, w3, 2, 1)
    assert a.shape == b.shape == (6, (hw[0] - 1) // 2 + 1, (hw[1] - 1) // 2 + 1)
    assert np.array_equal(a, b)
    assert np.array_equal(oracle.conv2d(x, w1, None, 2, 0), a)


def test_conv2d_skip_is_structural():
    x = np.ones((2, 4, 4))
    x[1, 1, 1] = np.inf
    w = np.ones((1, 2, 3, 3))
    skip = np.zeros((1, 2, 3, 3), np.uint8)
    skip[0, 1] = 1                       # whole channel 1 is a structural zero
    w[0, 1] = 0.0
    y = oracle.conv2d(x, w, skip, 1, 1)
    assert np.isfinite(y).all()
    assert y[0, 1, 1] == 9.0
    y2 = oracle.conv2d(x, w, None, 1, 1)  # multiplying 0 * inf instead leaks NaN
    assert np.isnan(y2[0, 1, 1])


def test_maxpool_bruteforce_and_nan():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((2, 7, 7))
    for k, s, p in [(2, 2, 0), (3, 2, 1)]:
        y = oracle.maxpool(x, k, s, p)
        P = (7 + 2 * p - k) // s + 1
        for c in range(2):
            for i in range(P):
                for j in range(P):
                    vals = [x[c, i * s + a - p, j * s + b - p] for a in range(k) for b in range(k)
                            if 0 <= i * s + a - p < 7 and 0 <= j * s + b - p < 7]
                    assert y[c, i, j] == max(vals)
    x[0, 3, 3] = np.nan
    y = oracle.maxpool(x, 2, 2, 0)
    assert np.isnan(y[0, 1, 1]) and np.isfinite(y[1]).all()


def test_flip_bit_known_words():
    assert oracle.flip_bit(1.0, 31, "fp32") == -1.0
    assert oracle.flip_bit(1.0, 23, "fp32") == 0.5          # 0x3F800000 -> 0x3F000000
    assert oracle.flip_bit(1.0, 30, "fp32") == math.inf     # 0x3F800000 -> 0x7F800000
    assert oracle.flip_bit(0.0, 0, "fp32") == 2.0 ** -149
    assert oracle.flip_bit(1.0, 14, "fp16") == math.inf     # 0x3C00 -> 0x7C00
    assert oracle.flip_bit(1.0, 10, "fp16") == 0.5          # 0x3C00 -> 0x3800
    assert oracle.flip_bit(0.0, 0, "fp16") == 2.0 ** -24
    z = oracle.flip_bit(0.0, 31, "fp32")
    assert z == 0.0 and math.copysign(1.0, z) == -1.0


def test_round_to_nearest_even():
    assert oracle.round_to([65504.0], "fp16")[0] == 65504.0
    assert oracle.round_to([65520.0], "fp16")[0] == math.inf     # tie at the top rounds to inf
    assert oracle.round_to([1 + 2 ** -11], "fp16")[0] == 1.0      # tie -> even
    assert oracle.round_to([1 + 3 * 2 ** -11], "fp16")[0] == 1 + 2 ** -9
    assert oracle.round_to([1 + 2 ** -24], "fp32")[0] == 1.0
    assert oracle.round_to([1 + 3 * 2 ** -24], "fp32")[0] == 1 + 2 ** -22


def test_bn_fold_equals_eq1():
    """Folded conv == conv followed by Eq. 1 applied literally."""
    rng = np.random.default_rng(5)
    w = rng.standard_normal((4, 3, 3, 3))
    b = rng.standard_normal(4)
    p = {"gamma": rng.uniform(0.5, 1.5, 4), "beta": rng.standard_normal(4),
         "mean": rng.standard_normal(4), "var": rng.uniform(0.5, 2.0, 4)}
    x = rng.standard_normal((3, 6, 6))
    y = oracle.conv2d(x, w, None, 1, 1) + b[:, None, None]
    bn = (y - p["mean"][:, None, None]) / np.sqrt(p["var"][:, None, None] + 1e-5) \
        * p["gamma"][:, None, None] + p["beta"][:, None, None]
    wf, bf = oracle.fold_bn(w, b, p, 1e-5)
    yf = oracle.conv2d(x, wf, None, 1, 1) + bf[:, None, None]
    np.testing.assert_allclose(yf, bn, rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------------------
# O-T1: the carry-through channel is the channel sum at the filter centre
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("k,stride,pad", [(3, 1, 1), (5, 1, 0), (3, 2, 1), (1, 2, 0), (7, 2, 3)])
def test_ct_channel_is_centre_channel_sum(k, stride, pad):
    layers = [Layer("conv", 0, 1, cin=3, cout=4, k=3, stride=1, pad=1, ct="ct"),
              Layer("conv", 1, 2, cin=4, cout=2, k=k, stride=stride, pad=pad, ct="ct")]
    params = int_params(layers, 1)
    net = oracle.build(layers, params, "fp64", in_shape=(3, 9, 9), n_classes=2)
    rng = np.random.default_rng(2)
    x = rng.integers(-8, 9, size=(1, 3, 9, 9)).astype(np.float64)
    acts = oracle.forward(net, x, keep=True)["acts"][0] if False else None
    # run layer by layer (no final FC in this net)
    a0 = x[0]
    a1 = oracle.conv2d(a0, net.layers[0].W, net.layers[0].skip, 1, 1) + net.layers[0].b[:, None, None]
    a2 = oracle.conv2d(a1, net.layers[1].W, net.layers[1].skip, stride, pad) + net.layers[1].b[:, None, None]
    # layer 0: checksum = sum of the 3 image channels at the same position
    assert np.array_equal(a1[4], a0.sum(axis=0))
    # layer 1: checksum = sum over the 5 input channels (4 data + checksum) at the centre
    ctr = (k - 1) // 2
    P, Q = a2.shape[1:]
    for p in range(P):
        for q in range(Q):
            h, w = p * stride + ctr - pad, q * stride + ctr - pad
            expect = sum(a1[c, h, w] for c in range(5)) if (0 <= h < 9 and 0 <= w < 9) else 0.0
            assert a2[2, p, q] == expect
    if (k, stride, pad) == (3, 1, 1):
        # non-overlapping: every input element counted exactly once (Sec. II-A)
        assert a2[2].sum() == a1.sum()
    # data channels never see the incoming checksum (zero slice, skipped)
    a1_nocs = a1.copy()
    a1_nocs[4] = 12345.0
    a2b = oracle.conv2d(a1_nocs, net.layers[1].W, net.layers[1].skip, stride, pad)
    assert np.array_equal(a2b[:2], a2[:2] - net.layers[1].b[:2, None, None])


def test_construction_entries():
    layers = synth.workload("resnet18_cifar").layers
    net = oracle.build(layers, synth.make_params(layers, 1), "fp32", in_shape=(3, 32, 32),
                       n_classes=10)
    stem, c1, ds = net.layers[0], net.layers[1], net.layers[6]
    assert stem.W.shape == (65, 3, 3, 3)                   # no checksum input into the stem
    assert (stem.W[64, :, 1, 1] == 1.0).all() and stem.skip[64, :, 1, 1].sum() == 0
    assert stem.skip[64].sum() == 3 * 9 - 3 and stem.b[64] == 0.0
    assert c1.W.shape == (64, 65, 3, 3)                     # block conv1: no CT row
    assert (c1.W[:, 64] == 0).all() and (c1.skip[:, 64] == 1).all()
    assert ds.ct == "pass" and ds.W.shape == (129, 65, 1, 1)
    assert ds.W[128, 64, 0, 0] == 1.0 and ds.skip[128, :64].all() and ds.b[128] == 0.0
    fc = net.layers[-1]
    assert fc.W.shape == (11, 513) and (fc.W[10] == 1.0).all() and fc.skip[:10, 512].all()


# ---------------------------------------------------------------------------
# O-T2: no leakage -- protected data logits equal the unprotected ones bitwise
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name,prec", [("lenet5", "fp32"), ("resnet18_cifar", "fp32"),
                                       ("resnet18_cifar", "fp16"), ("resnet18_imagenet", "fp16"),
                                       ("vgg16", "fp16")])
def test_protected_logits_equal_unprotected(name, prec):
    wl = synth.workload(name)
    params = cached_params(name)
    x = cached_inputs(name, 1)
    p = oracle.forward(oracle.build_workload(wl, prec, True, params=params), x)
    u = oracle.forward(oracle.build_workload(wl, prec, False, params=params), x)
    assert np.array_equal(p["logits"], u["logits"])
    assert np.isfinite(p["S"]).all()


# ---------------------------------------------------------------------------
# O-T3 / O-T4: the checksum equals its closed-form recursion; S sums the FC inputs
# ---------------------------------------------------------------------------

def tiny_mobilenet():
    """Two inverted-residual blocks (the second with a residual input) around
    depthwise 3x3 convolutions, one of them stride 2."""
    return [Layer("conv", 0, 1, cin=2, cout=4, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True),
            Layer("conv", 1, 2, cin=4, cout=8, k=1, ct="ct", bn=True, relu=True),
            Layer("conv", 2, 3, cin=8, cout=8, k=3, stride=2, pad=1, ct="pass", bn=True, relu=True, groups=8),
            Layer("conv", 3, 4, cin=8, cout=4, k=1, ct="ct", bn=True),
            Layer("conv", 4, 5, cin=4, cout=8, k=1, ct="none", bn=True, relu=True),
            Layer("conv", 5, 6, cin=8, cout=8, k=3, stride=1, pad=1, ct="pass", bn=True, relu=True, groups=8),
            Layer("conv", 6, 7, cin=8, cout=4, k=1, ct="ct", bn=True, res=4),
            Layer("gap", 7, 8),
            Layer("fc", 8, 9, cin=4, cout=3, final=True)]


def test_depthwise_equals_block_diagonal_dense_convolution():
    """A depthwise convolution is the dense one whose filter k is zero on
    every input channel but k (brute force through the pinned dense path)."""
    rng = np.random.default_rng(8)
    for stride in (1, 2):
        x = rng.normal(size=(5, 7, 6))
        w = rng.normal(size=(5, 1, 3, 3))
        dense = np.zeros((5, 5, 3, 3))
        for k in range(5):
            dense[k, k] = w[k, 0]
        y = oracle.depthwise2d(x, w, None, stride, 1)
        y_ref = oracle.conv2d(x, dense, None, stride, 1)
        assert np.allclose(y, y_ref, rtol=1e-13, atol=1e-13)
        # a skipped tap is not multiplied: an infinite input there stays out
        sk = np.zeros(w.shape, np.uint8)
        sk[2, 0, 0, 0] = 1
        xi = x.copy()
        xi[2] = np.inf
        assert not np.isfinite(oracle.depthwise2d(xi, w, None, stride, 1)[2]).all()
        w0 = w.copy()
        w0[2, 0, 0, 0] = 0.0
        y_sk = oracle.depthwise2d(x, w, sk, stride, 1)
        assert np.allclose(y_sk, oracle.depthwise2d(x, w0, None, stride, 1), rtol=1e-13, atol=1e-13)


def test_depthwise_passes_the_checksum_through():
    """The depthwise layer's checksum group reads only the incoming checksum:
    its checksum output is the input checksum at the sampled centre (ReLU'd,
    and the input checksum is already >= 0)."""
    layers = tiny_mobilenet()
    params = int_params(layers, 5, bn=True)
    net = oracle.build(layers, params, "fp64", True, bn_eps=0.0, in_shape=(2, 8, 8), n_classes=3)
    x = np.random.default_rng(6).integers(-4, 5, size=(1, 2, 8, 8)).astype(np.float32)
    a = oracle.forward(net, x, keep=True)["acts"][0]
    assert np.array_equal(a[3][-1], a[2][-1][::2, ::2])          # stride 2, pad 1: centre = 2p
    assert a[3].shape[0] == 8 + 1
    # the second block's first convolution has no checksum, so its depthwise
    # layer has nothing to pass: no extra group, no checksum channel
    assert a[5].shape[0] == 8 and a[6].shape[0] == 8
    assert net.layers[5].W.shape == (8, 1, 3, 3) and net.layers[2].W.shape == (9, 1, 3, 3)


@pytest.mark.parametrize("which", ["identity", "downsample-pass", "downsample-zero", "lenet", "mobilenet"])
def test_closed_form_exact_on_integer_nets(which):
    if which == "lenet":
        layers, shape = tiny_lenet(), (1, 10, 10)
    elif which == "mobilenet":
        layers, shape = tiny_mobilenet(), (2, 8, 8)
    else:
        layers, shape = tiny_resnet(ds=which != "identity"), (2, 8, 8)
    ds_mode = "zero" if which.endswith("zero") else "pass"
    params = int_params(layers, 3, bn=True)
    netp = oracle.build(layers, params, "fp64", True, ds_mode, bn_eps=0.0, in_shape=shape, n_classes=3)
    netu = oracle.build(layers, params, "fp64", False, ds_mode, bn_eps=0.0, in_shape=shape, n_classes=3)
    rng = np.random.default_rng(4)
    x = rng.integers(-4, 5, size=(3,) + shape).astype(np.float32)
    rp = oracle.forward(netp, x, keep=True)
    ru = oracle.forward(netu, x, keep=True)
    assert np.array_equal(rp["logits"], ru["logits"])
    for n in range(3):
        cf = oracle.closed_form_S(netu, layers, ru["acts"][n], ds_mode)
        assert cf == rp["S"][n]
        fin = rp["acts"][n][layers[-1].src].reshape(-1)
        assert math.fsum(fin) == rp["S"][n]            # S = sum of every final-FC input
        assert cf != 0.0


@pytest.mark.parametrize("name", ["lenet5", "resnet18_cifar", "resnet18_imagenet", "vgg16", "mobilenetv2_cifar"])
def test_closed_form_gaussian_nets(name):
    wl = synth.workload(name)
    params = cached_params(name)
    x = cached_inputs(name, 1)
    rp = oracle.forward(oracle.build_workload(wl, "fp64", True, params=params), x, keep=True)
    netu = oracle.build_workload(wl, "fp64", False, params=params)
    ru = oracle.forward(netu, x, keep=True)
    cf = oracle.closed_form_S(netu, wl.layers, ru["acts"][0])
    assert abs(cf - rp["S"][0]) <= 1e-12 * abs(cf)
    fin = rp["acts"][0][wl.layers[-1].src].reshape(-1)
    assert abs(math.fsum(fin) * 2.0 ** -wl.layers[-1].ct_shift - rp["S"][0]) <= 1e-12 * abs(cf)


def test_residual_rule_prevents_double_count():
    """With a CT filter in the block's first conv the block input would be summed twice."""
    layers = tiny_resnet(ds=False)
    params = int_params(layers, 6, bn=True)
    x = np.random.default_rng(7).integers(0, 5, size=(1, 2, 8, 8)).astype(np.float32)
    good = oracle.forward(oracle.build(layers, params, "fp64", bn_eps=0.0, in_shape=(2, 8, 8),
                                       n_classes=3), x)["S"][0]
    bad_layers = [Layer(**{**L.__dict__, "ct": "ct"}) if i == 1 else L for i, L in enumerate(layers)]
    bad = oracle.forward(oracle.build(bad_layers, params, "fp64", bn_eps=0.0, in_shape=(2, 8, 8),
                                      n_classes=3), x)["S"][0]
    assert bad != good


def test_residual_roles_hand_built_graphs():
    """Sec. II-A residual rule on hand-built graphs: a tensor read twice gives
    its convolution readers no carry-through filter; the convolution whose
    output is the residual operand is the shortcut."""
    # identity block: slot 1 is read by conv1 (src) and by the add of conv2 (res)
    assert oracle.residual_roles(tiny_resnet(ds=False)) == ["ct", "none", "ct", None, None]
    # downsample block: slot 1 is read by conv1 and by the 1x1 shortcut
    assert oracle.residual_roles(tiny_resnet(ds=True)) == ["ct", "none", "pass", "ct", None, None]
    # no residual anywhere: every convolution carries a filter
    assert oracle.residual_roles(tiny_lenet()) == ["ct", None, "ct", None, None]
    # a tensor read by two convolutions whose outputs meet only in an FC-free
    # branch: both readers lose the filter, the depthwise layer passes through
    L = [Layer("conv", 0, 1, cin=1, cout=2, k=3, pad=1),
         Layer("conv", 1, 2, cin=2, cout=2, k=3, pad=1),
         Layer("conv", 1, 3, cin=2, cout=2, k=3, pad=1, groups=2),
         Layer("conv", 3, 4, cin=2, cout=2, k=3, pad=1, groups=2)]
    assert oracle.residual_roles(L) == ["ct", "none", "none", "pass"]


@pytest.mark.parametrize("name", ["lenet5", "resnet18_cifar", "resnet18_imagenet", "vgg16",
                                  "mobilenetv2_cifar"])
def test_workload_roles_follow_the_residual_rule(name):
    """The roles the workloads declare (and the oracle and the library read)
    are those the residual rule derives from the graph."""
    wl = synth.workload(name)
    declared = [L.ct if L.op == "conv" else None for L in wl.layers]
    assert oracle.residual_roles(wl.layers) == declared


def test_top1_pins():
    """Sec. II-B "change of the golden classification": argmax with ties to the
    lowest index, any NaN logit gives class -1; infinities order as numbers."""
    nan, inf = float("nan"), float("inf")
    rows = [([1.0, 3.0, 2.0], 1), ([5.0, 5.0, 1.0], 0), ([1.0, 5.0, 5.0], 1),
            ([nan, 1.0, 2.0], -1), ([1.0, 2.0, nan], -1), ([nan, nan], -1),
            ([1.0, inf, 2.0], 1), ([inf, inf, 0.0], 0), ([-inf, -inf, -inf], 0), ([-inf, -5.0], 1),
            ([-0.0, 0.0], 0), ([0.0, -0.0], 0), ([7.0], 0), ([-1e30, -1e31, -1e29], 2)]
    for row, want in rows:
        assert oracle.top1(np.array([row]))[0] == want, (row, want)
    # without ties or NaN it is numpy's argmax (first maximum)
    x = np.random.default_rng(3).standard_normal((200, 17))
    assert (oracle.top1(x) == np.argmax(x, axis=1)).all()
    # float32 logits promoted to double keep their order
    assert oracle.top1(np.array([[np.float32(1.0), np.nextafter(np.float32(1.0), np.float32(2.0))]],
                                dtype=np.float32))[0] == 1


# ---------------------------------------------------------------------------
# O-T5: brute-force single-bit flips on a tiny net against a separate scalar model
# ---------------------------------------------------------------------------

def _f32(v):
    with np.errstate(over="ignore"):
        return float(np.float32(v))


def _flip32(v, bit):
    u = struct.unpack("<I", struct.pack("<f", v))[0] ^ (1 << bit)
    return struct.unpack("<f", struct.pack("<I", u))[0]


class ScalarTiny:
    """input 1x5x5 -> conv0 1->2 k3p1 (CT) relu -> conv1 2->2 k3p1 (CT) relu -> fc 50(+25)->3 (+S).

    Written from the paper's construction with explicit scalar loops and its
    own bookkeeping of which literal weights exist; shares nothing with the
    oracle beyond the raw parameters.
    """

    def __init__(self, w0, w1, wfc):
        self.w0, self.w1, self.wfc = w0, w1, wfc

    def literal_w(self, layer, k, c, r, s):
        """(value, structural) of literal weight [k, c, r, s]."""
        if layer == 0:                       # [3, 1, 3, 3]
            if k < 2:
                return _f32(self.w0[k, c, r, s]), False
            return (1.0, False) if (r, s) == (1, 1) else (0.0, True)
        # layer 1: [3, 3, 3, 3]; input channel 2 is the incoming checksum
        if k < 2:
            if c < 2:
                return _f32(self.w1[k, c, r, s]), False
            return 0.0, True
        return (1.0, False) if (r, s) == (1, 1) else (0.0, True)

    def run(self, img, wfault=None, afault=None):
        def conv(x, layer, K, C):
            y = np.zeros((K, 5, 5))
            for k in range(K):
                for p in range(5):
                    for q in range(5):
                        acc = 0.0
                        for c in range(C):
                            for r in range(3):
                                for s in range(3):
                                    v, structural = self.literal_w(layer, k, c, r, s)
                                    if wfault is not None and wfault[:5] == (layer, k, c, r, s):
                                        v, structural = wfault[5], False
                                    if structural:
                                        continue
                                    h, w = p + r - 1, q + s - 1
                                    if 0 <= h < 5 and 0 <= w < 5:
                                        acc += v * x[c][h][w]
                        y[k, p, q] = acc
            return y
        x0 = [[[_f32(img[0, h, w]) for w in range(5)] for h in range(5)]]
        a1 = conv(x0, 0, 3, 1)
        a1 = np.vectorize(_f32)(np.where(a1 < 0, 0.0, a1))
        if afault is not None:
            c, h, w, bit = afault
            a1[c, h, w] = _flip32(a1[c, h, w], bit)
        a2 = conv(a1, 1, 3, 3)
        a2 = np.vectorize(_f32)(np.where(a2 < 0, 0.0, a2))
        feats = a2.reshape(-1)                  # 50 data features then 25 checksum features
        logits = [_f32(sum(self.wfc[j, i] * feats[i] for i in range(50))) for j in range(3)]
        S = _f32(sum(feats))
        return logits, S


def test_bruteforce_flips_match_scalar_model():
    layers = [Layer("conv", 0, 1, cin=1, cout=2, k=3, stride=1, pad=1, ct="ct", relu=True),
              Layer("conv", 1, 2, cin=2, cout=2, k=3, stride=1, pad=1, ct="ct", relu=True),
              Layer("fc", 2, 3, cin=50, cout=3, final=True)]
    params = synth.make_params(layers, 11)
    params[1]["w"] = params[1]["w"]                     # Kaiming-normal, fp32
    net = oracle.build(layers, params, "fp32", in_shape=(1, 5, 5), n_classes=3)
    model = ScalarTiny(params[0]["w"], params[1]["w"], params[2]["w"].astype(np.float64))
    img = synth.normal(11, 99, 25).astype(np.float32).reshape(1, 1, 5, 5)
    clean = oracle.forward(net, img)
    lg, S0 = model.run(img[0])
    assert clean["S"][0] == S0
    np.testing.assert_allclose(clean["logits"][0], lg, rtol=1e-6)
    r, tau = S0, 0.05 * abs(S0)
    n_checked = n_flag = n_same = 0
    rng = np.random.default_rng(0)
    sites = [(0, e, b) for e in range(27) for b in range(32)] + \
            [(1, e, b) for e in range(81) for b in range(32)]
    act_sites = [(e, b) for e in range(75) for b in range(32)]
    # every weight flip; every activation flip of a random quarter of the words
    act_sites = [act_sites[i] for i in rng.permutation(len(act_sites))[:600]]
    for layer, e, bit in sites:
        K, C = (3, 1) if layer == 0 else (3, 3)
        k, rem = divmod(e, C * 9)
        c, rem = divmod(rem, 9)
        rr, ss = divmod(rem, 3)
        v0, _ = model.literal_w(layer, k, c, rr, ss)
        vf = _flip32(v0, bit)
        res = oracle.forward(net, img, oracle.Fault(0, layer, e, bit))
        _, Sm = model.run(img[0], wfault=(layer, k, c, rr, ss, vf))
        So = res["S"][0]
        if math.isnan(Sm):
            assert math.isnan(So)
        else:
            assert So == Sm or abs(So - Sm) <= 1e-6 * max(abs(Sm), 1.0), (layer, e, bit, So, Sm)
        fo = bool(oracle.verdict([So], r, tau)[0])
        fm = not (abs(Sm - r) <= tau)
        if abs(abs(Sm - r) - tau) > 0.01 * tau:
            assert fo == fm
        if vf == v0:                       # +0 -> -0: the same number
            assert So == S0 and not fo
            n_same += 1
        n_flag += fo
        n_checked += 1
    for e, bit in act_sites:
        c, rem = divmod(e, 25)
        h, w = divmod(rem, 5)
        res = oracle.forward(net, img, oracle.Fault(1, 1, e, bit))
        _, Sm = model.run(img[0], afault=(c, h, w, bit))
        So = res["S"][0]
        if math.isnan(Sm):
            assert math.isnan(So)
        else:
            assert So == Sm or abs(So - Sm) <= 1e-6 * max(abs(Sm), 1.0), (e, bit, So, Sm)
    assert n_checked == 27 * 32 + 81 * 32
    assert n_same >= 1 and 0 < n_flag < n_checked


def test_activation_fault_on_input_equals_flipped_input():
    wl = synth.workload("lenet5")
    net = oracle.build_workload(wl)
    x = synth.make_input(wl, batch=2)
    e, bit = 28 * 28 + 14 * 28 + 14, 29          # image 1, centre pixel
    a = oracle.forward(net, x, oracle.Fault(1, 0, e, bit))
    xf = x.copy()
    xf[1, 0, 14, 14] = oracle.flip_bit(float(x[1, 0, 14, 14]), bit, "fp32")
    b = oracle.forward(net, xf)
    assert np.array_equal(a["S"], b["S"]) and np.array_equal(a["logits"], b["logits"])


# ---------------------------------------------------------------------------
# O-T6: distribution-based threshold
# ---------------------------------------------------------------------------

def test_calibrate_hand_example():
    S = np.arange(100, dtype=np.float64)
    r, tau = oracle.calibrate(S, 0.10)
    assert r == 49.5
    assert tau == 44.5                     # 90th smallest of 0.5,0.5,1.5,1.5,...
    assert oracle.verdict(S, r, tau).sum() == 10
    r, tau = oracle.calibrate(S, 0.01)
    assert tau == 49.5 and oracle.verdict(S, r, tau).sum() == 0
    assert oracle.verdict([np.nan, np.inf, r], r, tau).tolist() == [True, True, False]


def test_fault_free_flag_rate_matches_alpha():
    layers = [Layer("conv", 0, 1, cin=1, cout=4, k=3, stride=1, pad=1, ct="ct", relu=True),
              Layer("maxpool", 1, 2, k=2, stride=2),
              Layer("fc", 2, 3, cin=4 * 4 * 4, cout=3, final=True)]
    params = synth.make_params(layers, 21)
    net = oracle.build(layers, params, "fp32", in_shape=(1, 8, 8), n_classes=3)
    n_cal, n_eval, alpha = 2000, 3000, 0.05

    def imgs(seed, n):
        return synth.normal(seed, 5, n * 64).astype(np.float32).reshape(n, 1, 8, 8)
    S_cal = oracle.forward(net, imgs(1, n_cal))["S"]
    r, tau = oracle.calibrate(S_cal, alpha)
    assert oracle.verdict(S_cal, r, tau).mean() <= alpha
    S_ev = oracle.forward(net, imgs(2, n_eval))["S"]
    k = int(oracle.verdict(S_ev, r, tau).sum())
    sd = math.sqrt(n_eval * alpha * (1 - alpha) + n_eval ** 2 * alpha * (1 - alpha) / n_cal)
    assert abs(k - n_eval * alpha) <= 2.576 * sd, k


# ---------------------------------------------------------------------------
# fault buffers
# ---------------------------------------------------------------------------

def test_fault_buffers_resnet18_cifar():
    wl = synth.workload("resnet18_cifar")
    net = oracle.build_workload(wl, params=cached_params("resnet18_cifar"))
    bufs = oracle.fault_buffers(net, 128)
    w = {b[1]: b[2] for b in bufs if b[0] == 0}
    a = {b[1]: b[2] for b in bufs if b[0] == 1}
    assert w[0] == 65 * 3 * 9 and w[1] == 64 * 65 * 9 and w[2] == 65 * 64 * 9
    assert 0 not in a                                # the image is left out
    assert a[1] == 128 * 65 * 32 * 32                # block input, read by conv1 and the residual
    assert a[2] == 128 * 64 * 32 * 32                # conv1 output has no checksum channel
    assert all(b[3] == 32 for b in bufs)
    n_conv = sum(1 for L in wl.layers if L.op == "conv")
    assert len(w) == n_conv


def test_fi_threshold_and_detection_rates_by_hand():
    # Sec. II-C FI-based threshold and the Sec. III-A rates on a worked example
    S = np.array([10.0, 11.0, 9.0, 30.0, np.nan, 12.0, 10.5, 8.0])
    crit = np.array([0, 0, 0, 1, 0, 0, 1, 0])
    r = 10.0
    # non-critical deviations: 0, 1, 1, inf (NaN), 2, 2 -> sorted 0 1 1 2 2 inf
    assert oracle.fi_threshold(S, crit, r, 0.2) == 2.0      # rank ceil(0.8 * 6) = 5
    assert oracle.fi_threshold(S, crit, r, 0.5) == 1.0      # rank 3
    assert oracle.fi_threshold(S, crit, r, 0.0) == np.inf   # rank 6
    tpr, fpr, j = oracle.detection_rates(S, crit, r, 2.0)
    # flagged: 30 (critical) and NaN (non-critical); 12 and 8 sit exactly at tau
    assert tpr == 0.5 and fpr == 1.0 / 6.0 and j == tpr - fpr


def test_fi_threshold_bounds_the_false_alarm_rate():
    rng = np.random.default_rng(4)
    S = rng.normal(100.0, 5.0, 5000)
    S[rng.integers(0, 5000, 40)] = np.inf
    crit = rng.random(5000) < 0.05
    for alpha in (0.001, 0.01, 0.05):
        tau = oracle.fi_threshold(S, crit, 100.0, alpha)
        _, fpr, _ = oracle.detection_rates(S, crit, 100.0, tau)
        assert fpr <= alpha + 1e-12
