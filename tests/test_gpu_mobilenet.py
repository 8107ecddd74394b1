"""MobileNet-V2 (CIFAR shape): depthwise convolutions whose checksum group
passes the incoming checksum through.  GPU path through the C ABI against
the oracle: logits, S, verdicts, fault buffers and single-bit flips."""
import numpy as np
import pytest

import oracle
import synth
from _cache import inputs
from _gpu import TOL, assert_parity, ct, model, onet, run, same_class

pytestmark = pytest.mark.gpu

NAME = "mobilenetv2_cifar"


@pytest.mark.parametrize("prec,batch,idx", [("fp32", 128, [0, 77, 127]), ("fp32", 3, None),
                                            ("fp16", 128, [0, 64, 127]), ("fp16", 5, None)])
def test_mobilenet_matches_oracle(prec, batch, idx):
    m = model(NAME, prec=prec, max_batch=batch)
    x = inputs(NAME, batch)
    lg, S, _ = run(m, x)
    sel = list(range(batch)) if idx is None else idx
    o = oracle.forward(onet(NAME, prec), x[sel])
    assert_parity(lg[sel], S[sel], o["logits"], o["S"], prec, "%s %s b%d" % (NAME, prec, batch))
    assert ct().ct_device_error(m) == 0
    m.close()


def test_mobilenet_unprotected_logits_unchanged():
    """The widened construction leaves the data path alone (here too)."""
    mp = model(NAME, prec="fp32", max_batch=4)
    mu = model(NAME, prec="fp32", protect=False, max_batch=4)
    x = inputs(NAME, 4)
    lp, _, _ = run(mp, x)
    lu, _, _ = run(mu, x)
    assert np.array_equal(lp, lu)
    mp.close()
    mu.close()


def test_mobilenet_flips_match_oracle():
    prec, B = "fp32", 4
    m = model(NAME, prec=prec, max_batch=B)
    net = onet(NAME, prec)
    x = inputs(NAME, B)
    bufs = ct().ct_buffers(m, B)
    assert bufs == oracle.fault_buffers(net, B)
    rng_faults = synth.draw_faults(bufs, 24, seed=41)
    # and one flip in a depthwise filter and one in a depthwise checksum group
    dw = [i for i, L in enumerate(net.layers) if L.op == "conv" and L.groups > 1 and L.has_ct_out][0]
    K = net.layers[dw].n_data_out
    extra = np.array([[0, dw, 3 * 9 + 4, 30], [0, dw, K * 9 + 4, 29], [0, dw, K * 9 + 0, 30]], dtype=np.int64)
    faults = np.concatenate([rng_faults, extra])
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
