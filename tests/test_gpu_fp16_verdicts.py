"""Verdict parity on the FP16 workloads (ResNet-18 at 224 x 224, batch 256;
VGG-16, batch 64): every row's logits and S against the oracle, and the
per-image verdict of Sec. II-B (flag = NOT(|S - r| <= tau)) identical on
both sides for one shared (r, tau), fault-free and under seeded single-bit
flips (Sec. III-A).  The GPU's flag is the rule applied to its own S, on
every image.  Near-threshold images are counted separately, not compared:
the oracle's S within 1% of tau of the threshold, or the two S values on
opposite sides of it while at most two binary16 ulps apart -- with FP16
storage S is an FP32 sum of FP16-rounded features, the largest of which
(the carried checksum) is near S itself, so two correct implementations can
round it one ulp apart (16 at S ~ 3.2e4 on VGG-16, against 1% of tau ~
1.4).  Their number is bounded and reported."""
import numpy as np
import pytest

import oracle
import synth
from _cache import inputs
from _gpu import TOL, assert_parity, ct, model, near_threshold, onet, run, same_class

pytestmark = pytest.mark.gpu

CASES = {"resnet18_imagenet": {"calib": 64, "weight_imgs": 8, "faults": 6},
         "vgg16": {"calib": 16, "weight_imgs": 4, "faults": 4}}


def _verdicts_agree(S_g, flag_g, S_o, r, tau, what):
    """Identical verdicts except near-threshold images; returns (compared, near)."""
    own = oracle.verdict(S_g, r, tau)
    assert (flag_g.astype(bool) == own).all(), (what, np.nonzero(flag_g.astype(bool) != own)[0][:8])
    near = near_threshold(S_o, r, tau, "fp16", S_g)
    want = oracle.verdict(S_o, r, tau)
    bad = np.nonzero((flag_g.astype(bool) != want) & ~near)[0]
    assert bad.size == 0, (what, bad[:8], S_g[bad[:8]], S_o[bad[:8]], r, tau)
    return int((~near).sum()), int(near.sum())


@pytest.mark.parametrize("name", sorted(CASES))
def test_fp16_logits_and_verdicts_every_row(name):
    cfg = CASES[name]
    wl = synth.workload(name)
    B = wl.batch
    net = onet(name, "fp16")
    m = model(name)
    x = inputs(name, B)
    o = oracle.forward(net, x)
    # Sec. II-C distribution-based threshold at alpha = 1% from the oracle's S
    # on seeded calibration images disjoint from the evaluation batch
    xc = synth.make_input(wl, batch=cfg["calib"], seed=wl.calib_seed)
    r, tau = oracle.calibrate(oracle.forward(net, xc)["S"], 0.01)
    # a second threshold that flags about half of the batch exercises both outcomes
    r2 = float(np.median(o["S"]))
    tau2 = float(np.median(np.abs(o["S"] - r2)))
    n_cmp = n_near = 0
    for rr, tt in ((r, tau), (r2, tau2)):
        ct().ct_set_threshold(m, rr, tt)
        lg, S, flag = run(m, x)
        assert_parity(lg, S, o["logits"], o["S"], "fp16", "%s all %d rows" % (name, B))
        c, nn = _verdicts_agree(S, flag, o["S"], rr, tt, name)
        n_cmp += c
        n_near += nn
    assert n_cmp + n_near == 2 * B and n_near <= max(3, 2 * B // 50), (n_cmp, n_near)

    # seeded single-bit flips over the literal layout's conv weights and
    # conv-input activations; a weight flip is compared on the first images,
    # an activation flip on the image it hits
    ct().ct_set_threshold(m, r, tau)
    top_o = oracle.top1(o["logits"])
    bufs = ct().ct_buffers(m, B)
    assert bufs == oracle.fault_buffers(net, B)
    per_img = {layer: n // B for kind, layer, n, bits in bufs if kind == 1}
    faults = synth.draw_faults(bufs, cfg["faults"], seed=23)
    # one exponent flip in a weight of the first 256-channel convolution as well,
    # so that at least one fault is large
    layer256 = [i for i, L in enumerate(net.layers) if L.op == "conv" and L.n_data_out == 256][0]
    n_w = [n for kind, lay, n, bits in bufs if kind == 0 and lay == layer256][0]
    faults = np.vstack([faults, [[0, layer256, n_w // 5 + 3, 14]]])
    n_f = crit_mismatch = 0
    for kind, layer, e, bit in faults.tolist():
        ct().ct_inject(m, kind, layer, e, bit)
        lg, S, flag = run(m, x)
        if kind == 0:
            imgs, f = list(range(cfg["weight_imgs"])), oracle.Fault(0, layer, e, bit)
        else:
            img, off = divmod(e, per_img[layer])
            imgs, f = [img], oracle.Fault(1, layer, off, bit)
        of = oracle.forward(net, x[imgs], f)
        for j, i in enumerate(imgs):
            so, sg = of["S"][j], S[i]
            assert same_class(sg, so), (name, kind, layer, e, bit, sg, so)
            if np.isfinite(so):
                assert abs(sg - so) <= TOL["fp16"] * max(abs(so), 1e-6), (name, kind, layer, e, bit, sg, so)
                lo = of["logits"][j]
                if np.isfinite(lo).all():
                    err = np.abs(lg[i] - lo).max() / max(np.abs(lo).max(), 1e-6)
                    assert err <= TOL["fp16"], (name, kind, layer, e, bit, err)
            c, nn = _verdicts_agree(np.array([sg]), flag[i:i + 1], np.array([so]), r, tau, (name, e, bit))
            n_near += nn
            crit_o = oracle.top1(of["logits"][j][None])[0] != top_o[i]
            crit_g = oracle.top1(lg[i][None])[0] != oracle.top1(o["logits"][i][None])[0]
            if crit_o != crit_g:
                lo = of["logits"][j]
                srt = np.sort(lo[np.isfinite(lo)])
                assert len(srt) > 1 and srt[-1] - srt[-2] <= 2 * TOL["fp16"] * np.abs(lo).max()
                crit_mismatch += 1
            n_f += 1
    assert n_f >= len(faults) and crit_mismatch <= 1
    assert ct().ct_device_error(m) == 0
    print("%s: %d verdicts compared, %d near-threshold, %d fault trials" % (name, n_cmp, n_near, n_f))
    m.close()
