"""GPU parity of the replace construction (Sec. II-A, prune and replace):
the CUDA path built with CT_PROTECT_REPLACE against oracle/replace.py on
the same seeded inputs (logits, S, verdicts), and single-bit flips in its
stored tensors (the literal layout has the original widths)."""
import functools

import numpy as np
import pytest

import oracle
import synth
from oracle import replace as orep
from _cache import inputs, params
from _gpu import TOL, assert_parity, ct, run, same_class

pytestmark = pytest.mark.gpu


@functools.lru_cache(maxsize=None)
def rnet(name, prec):
    wl = synth.workload(name)
    return orep.build_replace(wl.layers, params(name), prec, wl.bn_eps, wl.in_shape, wl.n_classes)


def rmodel(name, prec=None, max_batch=None, simt_only=False):
    wl = synth.workload(name)
    return ct().ct_build_workload(wl, params(name), precision=prec or wl.precision, replace=True,
                                  max_batch=max_batch or wl.batch, simt_only=simt_only)


@pytest.mark.parametrize("name,prec,batch,idx", [
    ("lenet5", "fp32", 64, None),
    ("resnet18_cifar", "fp32", 16, None),
    ("resnet18_cifar", "fp16", 16, None),
    ("resnet18_imagenet", "fp16", 20, [0, 7, 19]),
])
def test_replace_matches_oracle(name, prec, batch, idx):
    m = rmodel(name, prec, max_batch=batch)
    x = inputs(name, batch)
    lg, S, fl = run(m, x)
    sel = list(range(batch)) if idx is None else idx
    o = oracle.forward(rnet(name, prec), x[sel])
    assert_parity(lg[sel], S[sel], o["logits"], o["S"], prec, "%s %s replace" % (name, prec))
    # verdicts under a threshold that flags about a third of the images;
    # images within 1% of tau are not compared
    r = float(np.mean(o["S"]))
    dev = np.abs(o["S"] - r)
    tau = float(np.quantile(dev, 0.66))
    ct().ct_set_threshold(m, r, tau)
    _, _, fl = run(m, x)
    want = oracle.verdict(o["S"], r, tau)
    near = np.abs(dev - tau) <= 0.01 * tau
    assert np.array_equal(fl[sel][~near].astype(bool), want[~near].astype(bool))
    m.close()


def test_replace_same_shapes_as_unprotected():
    """Sec. II-A: no tensor grows (the fault buffers have the unprotected
    shapes); the widened construction grows them."""
    name, B = "resnet18_cifar", 4
    wl = synth.workload(name)
    mr = rmodel(name, "fp32", max_batch=B)
    mu = ct().ct_build_workload(wl, params(name), precision="fp32", protect=False, max_batch=B)
    mw = ct().ct_build_workload(wl, params(name), precision="fp32", protect=True, max_batch=B)
    br, bu, bw = (ct().ct_buffers(m, B) for m in (mr, mu, mw))
    assert br == bu
    assert br == oracle.fault_buffers(rnet(name, "fp32"), B)
    assert sum(n for _, _, n, _ in bw) > sum(n for _, _, n, _ in br)
    for m in (mr, mu, mw):
        m.close()


def test_replace_flips_match_oracle():
    name, prec, B = "resnet18_cifar", "fp32", 4
    m = rmodel(name, prec, max_batch=B)
    net = rnet(name, prec)
    x = inputs(name, B)
    bufs = ct().ct_buffers(m, B)
    faults = synth.draw_faults(bufs, 16, seed=21)
    per_img = {layer: n // B for kind, layer, n, bits in bufs if kind == 1}
    for kind, layer, e, bit in faults.tolist():
        ct().ct_inject(m, kind, layer, e, bit)
        lg, S, _ = run(m, x)
        if kind == 0:
            imgs, f = list(range(B)), oracle.Fault(0, layer, e, bit)
        else:
            img, off = divmod(e, per_img[layer])
            imgs, f = [img], oracle.Fault(1, layer, off, bit)
        o = oracle.forward(net, x[imgs], f)
        for j, i in enumerate(imgs):
            so, sg = o["S"][j], S[i]
            assert same_class(sg, so), (kind, layer, e, bit, sg, so)
            if np.isfinite(so):
                assert abs(sg - so) <= TOL[prec] * max(abs(so), 1e-6), (kind, layer, e, bit, sg, so)
    assert ct().ct_device_error(m) == 0
    m.close()


def test_replace_rejects_depthwise_networks():
    """The pruning scores read dense filters; a network with depthwise
    convolutions is refused before any weight is read."""
    with pytest.raises(ct().CtError) as e:
        rmodel("mobilenetv2_cifar", "fp32", max_batch=2)
    assert e.value.status == 6
