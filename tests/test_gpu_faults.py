"""GPU fault injection and re-execution against the oracle (Sec. III-A, II-B)."""
import numpy as np
import pytest

import oracle
import synth
from _cache import inputs
from _gpu import TOL, assert_parity, ct, kept_checksum_pixel, model, onet, rel_err_rows, run, same_class

pytestmark = pytest.mark.gpu


def _flip_sites(m, net, B, n, seed):
    bufs = ct().ct_buffers(m, B)
    assert bufs == oracle.fault_buffers(net, B)
    return synth.draw_faults(bufs, n, seed)


def test_lenet5_1000_flips_verdict_parity():
    name, B = "lenet5", 64
    wl = synth.workload(name)
    m = model(name)
    net = onet(name, "fp32")
    x = inputs(name, B)
    xc = synth.make_input(wl, batch=1000, seed=wl.calib_seed)
    r, tau = oracle.calibrate(oracle.forward(net, xc)["S"], 0.01)
    ct().ct_set_threshold(m, r, tau)
    g_lg, g_S, g_fl = run(m, x)
    o_g = oracle.forward(net, x)
    top_g, top_o = oracle.top1(g_lg), oracle.top1(o_g["logits"])
    faults = _flip_sites(m, net, B, 1000, seed=0)
    per_img = {L: int(np.prod(oracle.act_shape(net, L, 1)[1:])) for L in range(len(net.layers))
               if net.layers[L].op == "conv"}
    n_crit = n_det = n_near = crit_mismatch = 0
    for kind, layer, e, bit in faults.tolist():
        ct().ct_inject(m, kind, layer, e, bit)
        lg, S, fl = run(m, x)
        if kind == 0:
            imgs = list(range(8))
            f = oracle.Fault(0, layer, e, bit)
        else:
            img, off = divmod(e, per_img[layer])
            imgs = [img]
            f = oracle.Fault(1, layer, off, bit)
            others = [i for i in range(B) if i != img]
            assert np.array_equal(lg[others], g_lg[others]) and np.array_equal(S[others], g_S[others])
        o = oracle.forward(net, x[imgs], f)
        for j, i in enumerate(imgs):
            so, sg = o["S"][j], S[i]
            assert same_class(sg, so), (kind, layer, e, bit, sg, so)
            if np.isfinite(so):
                assert abs(sg - so) <= TOL["fp32"] * max(abs(so), 1e-6), (kind, layer, e, bit, sg, so)
            lo = o["logits"][j]
            if np.isfinite(lo).all():
                assert rel_err_rows(lg[i], lo)[0] <= TOL["fp32"], (kind, layer, e, bit)
            else:
                assert all(same_class(a, b) for a, b in zip(lg[i], lo))
            dev = abs(so - r)
            near = np.isfinite(so) and abs(dev - tau) <= 0.01 * tau
            of = bool(oracle.verdict([so], r, tau)[0])
            if near:
                n_near += 1
            else:
                assert bool(fl[i]) == of, (kind, layer, e, bit, sg, so, r, tau)
            crit_o = oracle.top1(lo[None])[0] != top_o[i]
            crit_g = oracle.top1(lg[i][None])[0] != top_g[i]
            if crit_o != crit_g:
                srt = np.sort(lo[np.isfinite(lo)])
                assert len(srt) > 1 and srt[-1] - srt[-2] <= 2 * TOL["fp32"] * np.abs(lo).max()
                crit_mismatch += 1
            n_crit += crit_o
            n_det += crit_o and of
    assert n_crit > 0 and n_det > 0
    assert crit_mismatch <= 2


@pytest.mark.parametrize("prec", ["fp32", "fp16"])
def test_weights_and_activations_restored_after_fault(prec):
    m = model("resnet18_cifar", prec=prec, max_batch=4)
    x = inputs("resnet18_cifar", 4)
    g = run(m, x)
    # exponent flips of data weights, a carry-through weight, a data activation
    # and a checksum activation at a position every stride-2 shortcut keeps
    net = onet("resnet18_cifar", prec)
    L = net.layers[2]
    K, C = L.W.shape[:2]
    pix, val = kept_checksum_pixel(net, x[:1], 1)
    assert 2.0 <= val < 256.0
    top = 30 if prec == "fp32" else 14
    raise_exp = 29 if prec == "fp32" else 13     # multiplies values in [2, 256) by 2**64 / 2**8
    for kind, layer, e, bit in [(0, 2, 5, top), (0, 2, (K - 1) * C * 9 + 4, top), (0, 2, 3, top),
                                (1, 2, 1000, top), (1, 1, 64 * 1024 + pix, raise_exp)]:
        ct().ct_inject(m, kind, layer, e, bit)
        f = run(m, x)
        assert not np.array_equal(f[1], g[1]), (kind, layer, e, bit)
        again = run(m, x)
        assert np.array_equal(again[0], g[0]) and np.array_equal(again[1], g[1])


def test_reexecute_restores_flagged_rows():
    import torch
    name = "resnet18_cifar"
    m = model(name, max_batch=16)
    x = inputs(name, 16)
    g_lg, g_S, _ = run(m, x)
    r = float(np.mean(g_S))
    ct().ct_set_threshold(m, r, float(np.abs(g_S - r).max()) * 1.01)
    # one activation fault on image 5: bit 29 of a checksum value of block 1's
    # output (a value in [2, 2**64)) multiplies it by 2**64, so S explodes.
    # (A checksum value at a position that a stride-2 shortcut drops never
    # reaches S: the pass-through shortcut samples the checksum like the data.)
    net = onet(name, "fp32")
    per = int(np.prod(oracle.act_shape(net, 3, 1)[1:]))
    assert per == 65 * 32 * 32
    pix, val = kept_checksum_pixel(net, x[5:6], 3)
    assert 2.0 <= val < 2.0 ** 64
    ct().ct_inject(m, 1, 3, 5 * per + 64 * 1024 + pix, 29)
    xd = torch.from_numpy(x).cuda()
    lg = torch.empty(16, m.n_classes, device="cuda")
    S = torch.empty(16, device="cuda")
    fl = torch.empty(16, dtype=torch.uint8, device="cuda")
    ct().ct_infer(m, xd, 16, lg, S, fl)
    flags = fl.cpu().numpy()
    assert flags[5] == 1 and flags.sum() == 1, flags
    n = ct().ct_reexecute(m, xd, 16, fl, lg, S)
    assert n == 1
    # rows of unflagged images are untouched; the re-run row is a fault-free
    # result (a batch of one image may split K differently, so it equals the
    # batch-16 row up to summation order)
    lgn, Sn = lg.cpu().numpy(), S.cpu().numpy()
    keep = [i for i in range(16) if i != 5]
    assert np.array_equal(lgn[keep], g_lg[keep].astype(np.float32))
    assert np.array_equal(Sn[keep], g_S[keep].astype(np.float32))
    assert rel_err_rows(lgn[5], g_lg[5])[0] <= 1e-5
    assert abs(Sn[5] - g_S[5]) <= 1e-5 * abs(g_S[5])


def test_reexecute_rows_match_oracle_every_bucket():
    """Sec. II-B re-execution against the oracle: with the graphs captured
    ahead of time (ct_reexecute_prepare) and a max_batch that is not a power
    of two (6), 1 to 6 flagged images (padded batches 1, 2, 4 and the capped
    6, which 5 flagged images also use) are re-run into poisoned rows; each
    re-run row matches the oracle and no other row is written."""
    import torch
    name, B = "resnet18_cifar", 6
    m = model(name, max_batch=B)
    ct().ct_reexecute_prepare(m, B)
    x = inputs(name, B)
    o = oracle.forward(onet(name, "fp32"), x)
    xd = torch.from_numpy(x).cuda()
    for n in (1, 2, 3, 5, 6, 5):
        fl = torch.zeros(B, dtype=torch.uint8, device="cuda")
        fl[B - n:] = 1
        lg = torch.full((B, m.n_classes), float("nan"), device="cuda")
        S = torch.full((B,), float("nan"), device="cuda")
        assert ct().ct_reexecute(m, xd, B, fl, lg, S) == n
        torch.cuda.synchronize()
        lgn, Sn = lg.cpu().numpy().astype(np.float64), S.cpu().numpy().astype(np.float64)
        assert np.isnan(lgn[:B - n]).all() and np.isnan(Sn[:B - n]).all()
        assert_parity(lgn[B - n:], Sn[B - n:], o["logits"][B - n:], o["S"][B - n:], "fp32",
                      "re-run of %d images" % n)
    assert ct().ct_device_error(m) == 0


def test_run_host_matches_device_path():
    name = "resnet18_cifar"
    m = model(name, max_batch=8)
    x = inputs(name, 8)
    g_lg, g_S, g_fl = run(m, x)
    lg = np.empty((8, m.n_classes), np.float32)
    S = np.empty(8, np.float32)
    fl = np.empty(8, np.uint8)
    n = ct().ct_run_host(m, x, lg, S, fl)
    assert n == 0 and (fl == 0).all()
    assert np.array_equal(lg, g_lg.astype(np.float32)) and np.array_equal(S, g_S.astype(np.float32))


def test_inject_range_errors():
    m = model("lenet5")
    with pytest.raises(ct().CtError):
        ct().ct_inject(m, 0, 1, 0, 0)            # layer 1 is a max-pool
    with pytest.raises(ct().CtError):
        ct().ct_inject(m, 0, 0, 7 * 1 * 25, 0)   # literal conv0 weights: 7 x 1 x 5 x 5
    with pytest.raises(ct().CtError):
        ct().ct_inject(m, 0, 0, 0, 32)
    ct().ct_inject(m, 0, 0, 7 * 25 - 1, 31)
    ct().ct_clear_faults(m)


def test_faults_in_shortcuts_that_share_their_block_launch():
    """ResNet-18/224, FP16, 64 images: the 1 x 1 shortcuts of stages 2 and 3
    (layers 7 and 12) run in the launch of their block's first convolution
    (layers 6 and 11; single CTAs, CTA pairs).  Weight faults in both layers
    (flipped words, and epilogue deltas for the shortcut's checksum-channel
    weights: its pass-through weight and a zero weight from the incoming
    checksum to a data channel) and activation faults in the tensor both
    read give the same bits as separate launches (CT_FLAG_LAYERWISE)."""
    B = 64
    x = inputs("resnet18_imagenet", B)
    ms = {lw: model("resnet18_imagenet", layerwise=lw, max_batch=B) for lw in (False, True)}
    # the merged pairs' weights (layers 6 + 7, 11 + 12) and the tensors they read
    bufs = [b for b in ct().ct_buffers(ms[False], B) if b[1] in (6, 7, 11, 12)]
    faults = []
    for kind, layers, n in ((0, (6, 11), 8), (0, (7, 12), 16), (1, (6, 11), 8)):
        faults += synth.draw_faults([b for b in bufs if b[0] == kind and b[1] in layers], n, seed=5).tolist()
    for layer, C, K in ((7, 64, 128), (12, 128, 256)):
        faults.append([0, layer, K * (C + 1) + C, 14])      # checksum pass-through weight 1.0 -> inf
        faults.append([0, layer, 5 * (C + 1) + C, 13])      # incoming checksum -> channel 5 (0)
    assert {f[0] for f in faults} == {0, 1}
    for kind, layer, e, bit in faults:
        out = []
        for lw in (False, True):
            ct().ct_inject(ms[lw], kind, layer, e, bit)
            out.append(run(ms[lw], x))
        (l0, s0, f0), (l1, s1, f1) = out
        assert np.array_equal(l0, l1, equal_nan=True), (kind, layer, e, bit)
        assert np.array_equal(s0, s1, equal_nan=True) and np.array_equal(f0, f1), (kind, layer, e, bit)
    assert ct().ct_launches_per_infer(ms[True]) - ct().ct_launches_per_infer(ms[False]) >= 2
    for m in ms.values():
        assert ct().ct_device_error(m) == 0
        m.close()
