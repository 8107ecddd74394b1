"""The batched campaign kernel (ct_campaign_batched, many faults per launch)
against the per-fault path (ct_inject + ct_infer) and against the oracle,
on LeNet-5 (Sec. III-A fault model: conv weights and conv-input
activations)."""
import numpy as np
import pytest

import oracle
import synth
from _cache import inputs
from _gpu import TOL, ct, model, onet, same_class

pytestmark = pytest.mark.gpu


def _batched(m, x, faults):
    import torch
    B, F = x.shape[0], len(faults)
    xd = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()
    S = torch.full((F, B), float("nan"), device="cuda")
    top1 = torch.full((F, B), -7, dtype=torch.int32, device="cuda")
    flag = torch.full((F, B), 9, dtype=torch.uint8, device="cuda")
    ct().ct_campaign_batched(m, xd, B, faults, S, top1, flag)
    torch.cuda.synchronize()
    return S.cpu().numpy(), top1.cpu().numpy(), flag.cpu().numpy()


def _per_fault(m, x, faults):
    import torch
    B = x.shape[0]
    xd = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()
    lg = torch.empty(B, m.n_classes, device="cuda")
    S = torch.empty(B, device="cuda")
    fl = torch.empty(B, dtype=torch.uint8, device="cuda")
    out = []
    for kind, layer, e, bit in faults.tolist():
        ct().ct_inject(m, kind, layer, e, bit)
        ct().ct_infer(m, xd, B, lg, S, fl)
        out.append((lg.cpu().numpy().copy(), S.cpu().numpy().copy(), fl.cpu().numpy().copy()))
    return out


def _top1(lg):
    return oracle.top1(lg)


def _setup(n_faults, seed):
    name, B = "lenet5", 64
    m = model(name, max_batch=B)
    x = inputs(name, B)
    bufs = ct().ct_buffers(m, B)
    faults = synth.draw_faults(bufs, n_faults, seed)
    # a threshold that flags the larger third of the fault-free deviations
    import torch
    xd = torch.from_numpy(x).cuda()
    lg = torch.empty(B, m.n_classes, device="cuda")
    S = torch.empty(B, device="cuda")
    ct().ct_infer(m, xd, B, lg, S, None)
    torch.cuda.synchronize()
    s0 = S.cpu().numpy().astype(np.float64)
    r = float(s0.mean())
    tau = float(np.quantile(np.abs(s0 - r), 0.66))
    ct().ct_set_threshold(m, r, tau)
    return m, x, bufs, faults, r, tau


def test_batched_matches_per_fault_path():
    m, x, bufs, faults, r, tau = _setup(300, seed=31)
    B = x.shape[0]
    per_img = {layer: n // B for kind, layer, n, bits in bufs if kind == 1}
    Sb, tb, fb = _batched(m, x, faults)
    ref = _per_fault(m, x, faults)
    n_cmp = n_near = 0
    for f, (kind, layer, e, bit) in enumerate(faults.tolist()):
        lg, S, fl = ref[f]
        imgs = range(B) if kind == 0 else [e // per_img[layer]]
        for i in imgs:
            assert same_class(Sb[f, i], S[i]), (f, kind, layer, e, bit, i, Sb[f, i], S[i])
            if np.isfinite(S[i]):
                assert abs(Sb[f, i] - S[i]) <= TOL["fp32"] * max(abs(S[i]), 1e-6), (f, i, Sb[f, i], S[i])
            if np.isfinite(S[i]) and abs(abs(S[i] - r) - tau) <= 0.01 * tau:
                n_near += 1
            else:
                assert fb[f, i] == fl[i], (f, i, Sb[f, i], S[i])
            t = _top1(lg[i][None])[0]
            if tb[f, i] != t:
                srt = np.sort(lg[i][np.isfinite(lg[i])])
                assert len(srt) > 1 and srt[-1] - srt[-2] <= 2 * TOL["fp32"] * np.abs(lg[i]).max()
            n_cmp += 1
        if kind == 1:
            # only the hit image's entry is written
            untouched = [j for j in range(B) if j not in imgs]
            assert np.isnan(Sb[f, untouched]).all() and (tb[f, untouched] == -7).all()
    assert n_cmp >= 300 and n_near <= n_cmp // 20
    assert ct().ct_device_error(m) == 0
    m.close()


def test_batched_matches_oracle():
    m, x, bufs, faults, r, tau = _setup(40, seed=32)
    B = x.shape[0]
    net = onet("lenet5", "fp32")
    per_img = {layer: n // B for kind, layer, n, bits in bufs if kind == 1}
    Sb, tb, fb = _batched(m, x, faults)
    o0 = oracle.forward(net, x[:4])
    golden = oracle.top1(o0["logits"])
    for f, (kind, layer, e, bit) in enumerate(faults.tolist()):
        if kind == 0:
            imgs, fo = [0, 1, 2, 3], oracle.Fault(0, layer, e, bit)
        else:
            img, off = divmod(e, per_img[layer])
            if img >= 4:
                continue
            imgs, fo = [img], oracle.Fault(1, layer, off, bit)
        o = oracle.forward(net, x[imgs], fo)
        for j, i in enumerate(imgs):
            so = o["S"][j]
            assert same_class(Sb[f, i], so), (f, kind, layer, e, bit, Sb[f, i], so)
            if np.isfinite(so):
                assert abs(Sb[f, i] - so) <= TOL["fp32"] * max(abs(so), 1e-6)
                if abs(abs(so - r) - tau) > 0.01 * tau:
                    assert fb[f, i] == oracle.verdict([so], r, tau)[0]
            to = oracle.top1(o["logits"][j][None])[0]
            if tb[f, i] != to:
                lo = o["logits"][j]
                srt = np.sort(lo[np.isfinite(lo)])
                assert len(srt) > 1 and srt[-1] - srt[-2] <= 2 * TOL["fp32"] * np.abs(lo).max()
    assert golden.shape == (4,)
    m.close()


def test_batched_rejects_other_networks_and_sites():
    m = model("resnet18_cifar", max_batch=2)
    x = inputs("resnet18_cifar", 2)
    with pytest.raises(ct().CtError):
        _batched(m, x, np.array([[0, 0, 0, 1]]))
    m.close()
    m = model("lenet5", max_batch=4)
    x = inputs("lenet5", 4)
    with pytest.raises(ct().CtError):              # the image is not a fault site
        _batched(m, x, np.array([[1, 0, 0, 1]]))
    m.close()


def test_batched_campaign_runner_bookkeeping():
    from paper_2609_16742_gb300 import campaign
    out = campaign.run_batched(faults=2000, seed=4, calib_images=512)
    assert out["device_error"] == 0
    a, w, act = out["all"], out["weights"], out["activations"]
    assert a["detected"] <= a["critical"] <= a["trials"]
    assert w["trials"] % out["batch"] == 0
    assert w["trials"] // out["batch"] + act["trials"] == 2000
    assert a["trials"] == w["trials"] + act["trials"]
