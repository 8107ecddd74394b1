"""The fault-injection campaign of Sec. III-A on the CIFAR ResNet-18: its
first 500 seeded faults against the oracle (per-image critical and flagged
verdicts), and the campaign runner's bookkeeping."""
import numpy as np
import pytest

import oracle
import synth
from _cache import params
from _gpu import TOL, ct, near_threshold, onet, run, same_class

pytestmark = pytest.mark.gpu


def _model(prec, B):
    net = synth.workload("resnet18_cifar")
    return ct().ct_build_workload(net, params("resnet18_cifar"), precision=prec, max_batch=B)


@pytest.mark.parametrize("prec", ["fp32", "fp16"])
def test_campaign_faults_match_oracle(prec):
    """The first 500 faults of the campaign (the same seeded draw as
    campaign.run with seed 0, over the campaign's batch of 128 images)
    against the oracle: per image trial, S within tolerance and the verdict
    identical (near-threshold images counted apart), and the critical
    verdict identical unless the oracle's top two logits are within the
    tolerance of each other.  A weight fault is compared on the first 8
    images, an activation fault on the image it hits."""
    wl = synth.workload("campaign_resnet18_cifar")
    B, n_faults = wl.batch, 500
    m = _model(prec, B)
    net = onet("resnet18_cifar", prec)
    x = synth.make_input(wl, batch=B)
    xc = synth.make_input(wl, batch=128, seed=wl.calib_seed)
    r, tau = oracle.calibrate(oracle.forward(net, xc)["S"], 0.01)
    ct().ct_set_threshold(m, r, tau)
    g_lg, _, _ = run(m, x)
    o_g = oracle.forward(net, x)
    top_o = oracle.top1(o_g["logits"])
    top_g = oracle.top1(g_lg)
    bufs = ct().ct_buffers(m, B)
    assert bufs == oracle.fault_buffers(net, B)
    faults = synth.draw_faults(bufs, n_faults, seed=0)
    per_img = {layer: n // B for kind, layer, n, bits in bufs if kind == 1}
    n_cmp = n_near = crit_mismatch = n_crit = n_flag = 0
    for kind, layer, e, bit in faults.tolist():
        ct().ct_inject(m, kind, layer, e, bit)
        lg, S, fl = run(m, x)
        if kind == 0:
            imgs, f = list(range(8)), oracle.Fault(0, layer, e, bit)
        else:
            img, off = divmod(e, per_img[layer])
            imgs, f = [img], oracle.Fault(1, layer, off, bit)
        o = oracle.forward(net, x[imgs], f)
        for j, i in enumerate(imgs):
            so, sg = o["S"][j], S[i]
            assert same_class(sg, so), (kind, layer, e, bit, sg, so)
            if np.isfinite(so):
                assert abs(sg - so) <= TOL[prec] * max(abs(so), 1e-6), (kind, layer, e, bit, sg, so)
            near = bool(near_threshold([so], r, tau, prec, [sg])[0])
            if near:
                n_near += 1
            else:
                assert bool(fl[i]) == bool(oracle.verdict([so], r, tau)[0]), (kind, layer, e, bit, sg, so)
            lo = o["logits"][j]
            crit_o = oracle.top1(lo[None])[0] != top_o[i]
            crit_g = oracle.top1(lg[i][None])[0] != top_g[i]
            if crit_o != crit_g:
                srt = np.sort(lo[np.isfinite(lo)])
                assert len(srt) > 1 and srt[-1] - srt[-2] <= 2 * TOL[prec] * np.abs(lo).max()
                crit_mismatch += 1
            n_crit += int(crit_o)
            n_flag += int(bool(fl[i]))
            n_cmp += 1
    assert n_cmp >= n_faults and crit_mismatch <= max(2, n_cmp // 500) and n_near <= max(5, n_cmp // 50)
    assert ct().ct_device_error(m) == 0
    print("%s: %d trials, %d critical, %d flagged, %d near-threshold, %d critical mismatches"
          % (prec, n_cmp, n_crit, n_flag, n_near, crit_mismatch))


def test_campaign_runner_bookkeeping():
    from paper_2609_16742_gb300 import campaign
    out = campaign.run("fp16", faults=48, seed=3, calib_images=512)
    assert out["device_error"] == 0
    a = out["all"]
    assert a["detected"] <= a["critical"] <= a["trials"]
    assert a["false_alarms"] <= a["trials"] - a["critical"]
    # a weight flip is one trial per image, an activation flip one trial
    w, act = out["weights"], out["activations"]
    assert w["trials"] % out["batch"] == 0
    assert w["trials"] // out["batch"] + act["trials"] == 48
    assert sum(v["trials"] for v in out["by_bit"].values()) == a["trials"]
    assert out["kernels_launched"] > 48


def test_threshold_sweep_rows():
    """Sec. II-C / III-A: distribution-based and FI-based taus over alpha; each
    row's rates are those the oracle's detection_rates gives for its tau on
    the evaluation trials, and the FI tau keeps the calibration campaign's
    false-alarm rate at or below alpha."""
    from paper_2609_16742_gb300 import campaign
    rec = {}
    orig = campaign._trials

    def spy(m, x, B, sites, stream, reexecute=False):
        out = orig(m, x, B, sites, stream, reexecute)
        rec.setdefault("runs", []).append(out)
        return out

    campaign._trials = spy
    try:
        out = campaign.sweep("fp16", faults=256, calib_images=512)
    finally:
        campaign._trials = orig
    assert out["device_error"] == 0
    (S_c, crit_c, _), (S_e, crit_e, _) = rec["runs"]
    assert S_c.size == out["calibration_trials"] and S_e.size == out["evaluation_trials"]
    assert len(out["table"]) == 6
    assert out["evaluation_critical"] > 0 and out["calibration_critical"] > 0
    for row in out["table"]:
        tpr, fpr, j = oracle.detection_rates(S_e, crit_e, row["reference"], row["tau"])
        assert row["fpr"] == pytest.approx(fpr, abs=1e-12)
        if tpr is not None and row["tpr"] is not None:
            assert row["tpr"] == pytest.approx(tpr, abs=1e-12)
        if row["method"] == "fi":
            assert row["tau"] == oracle.fi_threshold(S_c, crit_c, row["reference"], row["alpha"])
            _, fpr_c, _ = oracle.detection_rates(S_c, crit_c, row["reference"], row["tau"])
            assert fpr_c <= row["alpha"] + 1e-12
    # a larger alpha never raises tau
    for meth in ("distribution", "fi"):
        taus = [row["tau"] for row in out["table"] if row["method"] == meth]
        assert all(a >= b for a, b in zip(taus, taus[1:]))
