"""Deferred re-execution (ct_infer_reexec, Sec. II-B): the previous batch's
flagged images are re-run as extra rows of the next inference.  Checked
against plain ct_infer of the same combined batch, which must agree bit for
bit: within one inference every image's row is computed independently of
the others and the combined batch has the same size, hence the same tiling
and split-K choices.  Covers the fused-stem input path (224x224 FP16) and
the converted-input path (32x32 FP32)."""
import numpy as np
import pytest

import synth
from _cache import inputs
from _gpu import ct, model

pytestmark = pytest.mark.gpu


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _threshold_flagging(m, S, k):
    """(r, tau) under which exactly the k images of largest |S - r| are flagged."""
    r = float(np.mean(S))
    dev = np.sort(np.abs(S - r))
    tau = float(0.5 * (dev[-k - 1] + dev[-k]))
    ct().ct_set_threshold(m, r, tau)
    return r, tau


@pytest.mark.parametrize("name", ["resnet18_imagenet", "resnet18_cifar"])
def test_deferred_rows_equal_combined_batch(name):
    import torch
    B, k = 6, 3
    m = model(name, max_batch=B + 4)
    xa, xb = inputs(name, 2 * B)[:B], inputs(name, 2 * B)[B:]
    nc = m.n_classes
    # previous batch: plain inference under a threshold that flags k images
    xad = _dev(xa)
    la = torch.empty(B, nc, device="cuda"); Sa = torch.empty(B, device="cuda")
    fa = torch.empty(B, dtype=torch.uint8, device="cuda")
    ct().ct_infer(m, xad, B, la, Sa, fa)
    torch.cuda.synchronize()
    _threshold_flagging(m, Sa.cpu().numpy().astype(np.float64), k)
    ct().ct_infer(m, xad, B, la, Sa, fa)
    torch.cuda.synchronize()
    flags = fa.cpu().numpy().copy()
    idx = np.nonzero(flags)[0]
    assert len(idx) == k
    la_before, Sa_before = la.cpu().numpy().copy(), Sa.cpu().numpy().copy()
    # poison the flagged rows: the re-run must overwrite them
    la[torch.from_numpy(idx).cuda()] = float("nan")
    Sa[torch.from_numpy(idx).cuda()] = float("nan")
    # deferred: new batch + the k flagged images of the previous one
    xbd = _dev(xb)
    lb = torch.full((B, nc), float("nan"), device="cuda"); Sb = torch.full((B,), float("nan"), device="cuda")
    fb = torch.full((B,), 7, dtype=torch.uint8, device="cuda")
    n = ct().ct_infer_reexec(m, xbd, B, lb, Sb, fb, xad, B, fa, la, Sa)
    torch.cuda.synchronize()
    assert n == k
    # reference: plain ct_infer of the combined batch [xb; xa[idx]]
    comb = np.concatenate([xb, xa[idx]], axis=0)
    cd = _dev(comb)
    lc = torch.empty(B + k, nc, device="cuda"); Sc = torch.empty(B + k, device="cuda")
    fc = torch.empty(B + k, dtype=torch.uint8, device="cuda")
    ct().ct_infer(m, cd, B + k, lc, Sc, fc)
    torch.cuda.synchronize()
    lcn, Scn, fcn = lc.cpu().numpy(), Sc.cpu().numpy(), fc.cpu().numpy()
    assert np.array_equal(lb.cpu().numpy(), lcn[:B])
    assert np.array_equal(Sb.cpu().numpy(), Scn[:B])
    assert np.array_equal(fb.cpu().numpy(), fcn[:B])
    lan, San = la.cpu().numpy(), Sa.cpu().numpy()
    assert np.array_equal(lan[idx], lcn[B:])
    assert np.array_equal(San[idx], Scn[B:])
    keep = np.setdiff1d(np.arange(B), idx)
    assert np.array_equal(lan[keep], la_before[keep])
    assert np.array_equal(San[keep], Sa_before[keep])
    # the previous flags are not modified (the re-run's flag is ignored)
    assert np.array_equal(fa.cpu().numpy(), flags)
    assert ct().ct_device_error(m) == 0
    m.close()


def test_deferred_without_previous_is_plain_infer():
    import torch
    name, B = "resnet18_cifar", 5
    m = model(name, max_batch=B)
    x = _dev(inputs(name, B))
    l1 = torch.empty(B, m.n_classes, device="cuda"); S1 = torch.empty(B, device="cuda")
    l2 = torch.empty(B, m.n_classes, device="cuda"); S2 = torch.empty(B, device="cuda")
    ct().ct_infer(m, x, B, l1, S1, None)
    assert ct().ct_infer_reexec(m, x, B, l2, S2, None) == 0
    torch.cuda.synchronize()
    assert torch.equal(l1, l2) and torch.equal(S1, S2)
    m.close()


def test_deferred_falls_back_when_rows_do_not_fit():
    """batch + flagged > max_batch: the previous batch is re-run as by
    ct_reexecute, then the new batch as by ct_infer."""
    import torch
    name, B, k = "resnet18_cifar", 6, 3
    m = model(name, max_batch=B + 2)
    xa, xb = inputs(name, 2 * B)[:B], inputs(name, 2 * B)[B:]
    nc = m.n_classes
    xad, xbd = _dev(xa), _dev(xb)
    la = torch.empty(B, nc, device="cuda"); Sa = torch.empty(B, device="cuda")
    fa = torch.empty(B, dtype=torch.uint8, device="cuda")
    ct().ct_infer(m, xad, B, la, Sa, fa)
    torch.cuda.synchronize()
    _threshold_flagging(m, Sa.cpu().numpy().astype(np.float64), k)
    ct().ct_infer(m, xad, B, la, Sa, fa)
    # expected previous rows: a synchronous re-execution on copies
    la_ref, Sa_ref = la.clone(), Sa.clone()
    assert ct().ct_reexecute(m, xad, B, fa, la_ref, Sa_ref) == k
    lb = torch.empty(B, nc, device="cuda"); Sb = torch.empty(B, device="cuda")
    fb = torch.empty(B, dtype=torch.uint8, device="cuda")
    assert ct().ct_infer_reexec(m, xbd, B, lb, Sb, fb, xad, B, fa, la, Sa) == k
    lb_ref = torch.empty(B, nc, device="cuda"); Sb_ref = torch.empty(B, device="cuda")
    ct().ct_infer(m, xbd, B, lb_ref, Sb_ref, None)
    torch.cuda.synchronize()
    assert torch.equal(la, la_ref) and torch.equal(Sa, Sa_ref)
    assert torch.equal(lb, lb_ref) and torch.equal(Sb, Sb_ref)
    m.close()
