"""GPU parity: the CUDA path, called through the C ABI, against the oracle on
the same seeded inputs, element by element (logits, S, verdicts)."""
import numpy as np
import pytest

import oracle
from _cache import inputs
from _gpu import TOL, assert_parity, ct, model, onet, run, same_class

pytestmark = pytest.mark.gpu


def _oracle(name, prec, x, protected=True):
    return oracle.forward(onet(name, prec, protected), x)


def test_lenet5_full_batch():
    m = model("lenet5")
    x = inputs("lenet5", 64)
    lg, S, flag = run(m, x)
    o = _oracle("lenet5", "fp32", x)
    assert_parity(lg, S, o["logits"], o["S"], "fp32", "lenet5")


@pytest.mark.parametrize("simt_only", [False, True])
def test_resnet18_cifar_fp32_full_batch_sampled(simt_only):
    m = model("resnet18_cifar", simt_only=simt_only)
    x = inputs("resnet18_cifar", 128)
    lg, S, _ = run(m, x)
    idx = [0, 1, 64, 127]
    o = _oracle("resnet18_cifar", "fp32", x[idx])
    assert_parity(lg[idx], S[idx], o["logits"], o["S"], "fp32", "resnet18_cifar")


@pytest.mark.parametrize("prec,simt_only", [("fp32", False), ("fp16", False), ("fp16", True)])
@pytest.mark.parametrize("batch", [1, 3])
def test_resnet18_cifar_ragged_batches(prec, simt_only, batch):
    m = model("resnet18_cifar", prec=prec, simt_only=simt_only, max_batch=4)
    x = inputs("resnet18_cifar", batch, 5)
    lg, S, _ = run(m, x)
    o = _oracle("resnet18_cifar", prec, x)
    assert_parity(lg, S, o["logits"], o["S"], prec, "resnet18_cifar %s b%d" % (prec, batch))


def test_resnet18_imagenet_fp16_full_batch_sampled():
    m = model("resnet18_imagenet")
    x = inputs("resnet18_imagenet", 256)
    lg, S, _ = run(m, x)
    idx = [0, 129, 255]
    o = _oracle("resnet18_imagenet", "fp16", x[idx])
    assert_parity(lg[idx], S[idx], o["logits"], o["S"], "fp16", "resnet18_imagenet")


def test_resnet18_imagenet_fp16_odd_tile_count_and_flip():
    """131 images: the 256-channel layers have an odd number of 128-row
    tiles (201 at 14 x 14, 51 at 7 x 7), so the last pair of CTAs that share
    a 256-row tile has its second CTA past the output; the last image's rows
    lie in that pair's first CTA.  Then one weight flip in the first
    256-channel convolution, compared on the same images."""
    name, B = "resnet18_imagenet", 131
    m = model(name, max_batch=B)
    x = inputs(name, B)
    lg, S, _ = run(m, x)
    idx = [0, 130]
    net = onet(name, "fp16")
    o = oracle.forward(net, x[idx])
    assert_parity(lg[idx], S[idx], o["logits"], o["S"], "fp16", "resnet18_imagenet b131")
    layer = [i for i, L in enumerate(net.layers) if L.op == "conv" and L.n_data_out == 256][0]
    n_w = [n for kind, lay, n, bits in ct().ct_buffers(m, B) if kind == 0 and lay == layer][0]
    e, bit = n_w // 3 + 7, 13
    ct().ct_inject(m, 0, layer, e, bit)
    lg, S, _ = run(m, x)
    o = oracle.forward(net, x[idx], oracle.Fault(0, layer, e, bit))
    for j, i in enumerate(idx):
        assert same_class(S[i], o["S"][j]), (i, S[i], o["S"][j])
        if np.isfinite(o["S"][j]):
            assert abs(S[i] - o["S"][j]) <= TOL["fp16"] * max(abs(o["S"][j]), 1e-6), (i, S[i], o["S"][j])
    assert ct().ct_device_error(m) == 0
    m.close()


def test_vgg16_fp16_full_batch_sampled():
    m = model("vgg16")
    x = inputs("vgg16", 64)
    lg, S, _ = run(m, x)
    idx = [0, 63]
    o = _oracle("vgg16", "fp16", x[idx])
    assert_parity(lg[idx], S[idx], o["logits"], o["S"], "fp16", "vgg16")
    assert np.isfinite(S).all() and np.abs(S).max() < 65504


@pytest.mark.parametrize("prec", ["fp32", "fp16"])
def test_protected_data_path_equals_unprotected(prec):
    x = inputs("resnet18_cifar", 8)
    lp, Sp, fp = run(model("resnet18_cifar", prec=prec, max_batch=8), x)
    lu, Su, fu = run(model("resnet18_cifar", prec=prec, protect=False, max_batch=8), x)
    assert np.array_equal(lp, lu)           # the checksum never enters a data channel
    assert np.isnan(Su).all() and (fu == 0).all()
    assert np.isfinite(Sp).all()


def test_downsample_zero_mode():
    x = inputs("resnet18_cifar", 2)
    m = model("resnet18_cifar", max_batch=2, ds_mode="zero")
    lg, S, _ = run(m, x)
    o = oracle.forward(onet("resnet18_cifar", "fp32", True, "zero"), x)
    assert_parity(lg, S, o["logits"], o["S"], "fp32", "ds zero")


def test_verdict_parity_with_shared_threshold():
    x = inputs("resnet18_cifar", 32)
    m = model("resnet18_cifar", max_batch=32)
    o = _oracle("resnet18_cifar", "fp32", x)
    r = float(np.median(o["S"]))
    tau = float(np.median(np.abs(o["S"] - r)))      # about half the images flagged
    ct().ct_set_threshold(m, r, tau)
    _, S, flag = run(m, x)
    of = oracle.verdict(o["S"], r, tau)
    near = np.abs(np.abs(o["S"] - r) - tau) <= 0.01 * tau
    assert (flag[~near].astype(bool) == of[~near]).all()
    assert 0 < flag.sum() < len(flag)


def test_fault_buffers_match_oracle():
    m = model("resnet18_cifar")
    assert ct().ct_buffers(m, 128) == oracle.fault_buffers(onet("resnet18_cifar", "fp32"), 128)
    m16 = model("resnet18_imagenet", max_batch=2)
    assert ct().ct_buffers(m16, 2) == oracle.fault_buffers(onet("resnet18_imagenet", "fp16"), 2)


def test_roles_derived_by_the_library_build_the_same_network():
    """Sec. II-A residual rule: the network built with every role left to the
    library (CT_ROLE_AUTO) is the one built from the declared roles, bit for
    bit."""
    import dataclasses
    import synth
    from _cache import params
    name = "resnet18_cifar"
    wl = synth.workload(name)
    auto = [dataclasses.replace(L, ct="auto") if L.op == "conv" else L for L in wl.layers]
    x = inputs(name, 4)
    ma = ct().ct_build(auto, params(name), wl.in_shape, wl.n_classes, max_batch=4)
    la, Sa, _ = run(ma, x)
    lm, Sm, _ = run(model(name, max_batch=4), x)
    assert np.array_equal(la, lm) and np.array_equal(Sa, Sm)
    ma.close()


def test_vgg16_fused_pool_under_weight_faults():
    """VGG-16's first two stride-1 layers apply the following 2 x 2 max-pool in
    their halo-tile epilogue.  Single-bit flips in conv1_2's weights -- a
    stored data weight, the carry-through row off its centre tap and the
    zero checksum slice (the last two are implicit and enter the epilogue as
    a delta) -- give the oracle's S and logits on the images they touch."""
    name, B = "vgg16", 2
    m = model(name, max_batch=B)
    net = onet(name, "fp16")
    x = inputs(name, B)
    lg, S, _ = run(m, x)
    o = oracle.forward(net, x)
    assert_parity(lg, S, o["logits"], o["S"], "fp16", "vgg16 fused pools")
    with pytest.raises(ct().CtError) as ei:          # the unpooled conv1_2 output is not stored
        ct().ct_copy_activation(m, 2, B)
    assert ei.value.status == 4
    layer = 1                                         # conv1_2: 64 -> 64 (+1), input 64 (+1) channels
    K, C = 64, 64
    def el(k, c, r, s_):
        return ((k * (C + 1) + c) * 3 + r) * 3 + s_
    for e, bit in [(el(5, 7, 1, 1), 14), (el(K, 3, 0, 2), 14), (el(9, C, 1, 1), 13)]:
        ct().ct_inject(m, 0, layer, e, bit)
        lg, S, _ = run(m, x)
        of = oracle.forward(net, x, oracle.Fault(0, layer, e, bit))
        for i in range(B):
            assert same_class(S[i], of["S"][i]), (e, bit, S[i], of["S"][i])
            if np.isfinite(of["S"][i]):
                assert abs(S[i] - of["S"][i]) <= TOL["fp16"] * max(abs(of["S"][i]), 1e-6), (e, bit, S[i], of["S"][i])
            if np.isfinite(of["logits"][i]).all():
                err = np.abs(lg[i] - of["logits"][i]).max() / max(np.abs(of["logits"][i]).max(), 1e-6)
                assert err <= TOL["fp16"], (e, bit, err)
    assert ct().ct_device_error(m) == 0


def test_half_tiles_of_the_last_round_give_whole_tile_bits():
    """A 512 -> 512 3 x 3 convolution on 7 x 7 maps: 256 images make 98
    CTA-pair tiles for 76 pairs, and the 22 tiles of the last round (images
    199-255) run as 44 half tiles of 128 channels; 128 images make 50 tiles,
    all whole.  Each output is the same full-K accumulation either way, so
    images 128-255 give the same bits (data and checksum) in both runs."""
    import synth
    from synth import Layer
    shape = (512, 7, 7)
    layers = [Layer("conv", 0, 1, cin=512, cout=512, k=3, stride=1, pad=1, ct="ct", bn=True, relu=True),
              Layer("gap", 1, 2), Layer("fc", 2, 3, cin=512, cout=10, final=True)]
    params = synth.make_params(layers, 11)
    x = np.random.default_rng(5).standard_normal((256,) + shape).astype(np.float32)
    out = {}
    for B in (256, 128):
        m = ct().ct_build(layers, params, shape, 10, precision="fp16", max_batch=B)
        run(m, x[256 - B:])
        out[B] = ct().ct_copy_activation(m, 1, B)
        assert ct().ct_device_error(m) == 0
        m.close()
    (d256, c256), (d128, c128) = out[256], out[128]
    assert np.isfinite(d256).all() and np.abs(d256).max() > 0
    assert np.array_equal(d256[128:], d128) and np.array_equal(c256[128:], c128)


@pytest.mark.gpu
@pytest.mark.parametrize("batch", [256, 37])
def test_shortcuts_in_the_block_launch_give_separate_launch_bits(batch):
    """ResNet-18 (224 x 224, FP16): each 1 x 1 stride-2 shortcut runs in the
    launch of its block's first 3 x 3 convolution, reading that
    convolution's centre-tap K blocks (stage 2 on single CTAs; stages 3-4 on
    CTA pairs, stage 4 beside half tiles at 256 images); CT_FLAG_LAYERWISE
    runs each shortcut in its own launch.  Every output is the same MMA
    sequence either way, so every stored tensor (data and checksum), the
    logits and S are the same bits; the merged run also launches three
    kernels fewer at 256 images."""
    x = inputs("resnet18_imagenet", batch, 3)
    res = {}
    for lw in (False, True):
        m = model("resnet18_imagenet", layerwise=lw, max_batch=batch)
        lg, S, fl = run(m, x)
        assert ct().ct_device_error(m) == 0
        acts = {}
        for slot in range(2, 23):
            try:
                acts[slot] = ct().ct_copy_activation(m, slot, batch)
            except RuntimeError:
                pass
        res[lw] = (lg, S, fl, acts, ct().ct_launches_per_infer(m))
        m.close()
    (lg0, S0, f0, a0, k0), (lg1, S1, f1, a1, k1) = res[False], res[True]
    assert sorted(a0) == sorted(a1) and len(a0) >= 18
    for slot in a0:
        (d0, c0), (d1, c1) = a0[slot], a1[slot]
        assert np.array_equal(d0, d1, equal_nan=True), slot
        assert (c0 is None) == (c1 is None) and (c0 is None or np.array_equal(c0, c1, equal_nan=True)), slot
    assert np.array_equal(lg0, lg1, equal_nan=True) and np.array_equal(S0, S1, equal_nan=True)
    assert np.array_equal(f0, f1)
    if batch == 256:
        assert k1 - k0 == 3
