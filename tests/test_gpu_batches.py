"""ct_infer_batches / ct_run_host_batches (Sec. II-B over a list of batches):
an image flagged in batch 0 is re-run two batches later, after which every
image's logits and S match the oracle; the host-buffer call gives the
device call's results bit for bit."""
import numpy as np
import pytest

import oracle
from _cache import inputs
from _gpu import TOL, assert_parity, ct, kept_checksum_pixel, model, onet

pytestmark = pytest.mark.gpu

NAME, B, NB = "resnet18_cifar", 16, 5


def _armed_model(max_batch):
    """A model whose threshold flags no fault-free image, with one activation
    fault armed for the next inference: bit 29 of a checksum value of block
    1's output of image 5 (a value in [2, 2**64), so S explodes)."""
    net = onet(NAME, "fp32")
    x = inputs(NAME, B * NB)
    o = oracle.forward(net, x)
    m = model(NAME, max_batch=max_batch)
    r = float(np.mean(o["S"]))
    ct().ct_set_threshold(m, r, float(np.abs(o["S"] - r).max()) * 1.01)
    pix, val = kept_checksum_pixel(net, x[5:6], 3)
    assert 2.0 <= val < 2.0 ** 64
    ct().ct_inject(m, 1, 3, 5 * 65 * 32 * 32 + 64 * 1024 + pix, 29)
    return m, x, o


@pytest.mark.parametrize("room", [8, 0])
def test_batches_rerun_the_flagged_image_and_match_the_oracle(room):
    """room 8: the flagged image rides as an extra row of batch 2's
    inference; room 0: it does not fit max_batch and is re-run on its own."""
    import torch
    m, x, o = _armed_model(B + room)
    xs = [torch.from_numpy(x[i * B:(i + 1) * B]).cuda() for i in range(NB)]
    lg = [torch.full((B, m.n_classes), float("nan"), device="cuda") for _ in range(NB)]
    S = [torch.full((B,), float("nan"), device="cuda") for _ in range(NB)]
    fl = [torch.full((B,), 7, dtype=torch.uint8, device="cuda") for _ in range(NB)]
    n = ct().ct_infer_batches(m, xs, B, lg, S, fl)
    flags = torch.cat(fl).cpu().numpy()
    assert flags[5] == 1 and flags.sum() == 1 and n == 1, (flags.nonzero(), n)
    lgn = torch.cat(lg).cpu().numpy().astype(np.float64)
    Sn = torch.cat(S).cpu().numpy().astype(np.float64)
    assert_parity(lgn, Sn, o["logits"], o["S"], "fp32", "batches, room %d" % room)
    assert ct().ct_device_error(m) == 0


def test_host_batches_equal_device_batches():
    import torch
    m, x, o = _armed_model(B + 8)
    xh = [np.ascontiguousarray(x[i * B:(i + 1) * B]) for i in range(NB)]
    lh = [np.full((B, m.n_classes), np.nan, np.float32) for _ in range(NB)]
    sh = [np.full(B, np.nan, np.float32) for _ in range(NB)]
    fh = [np.full(B, 7, np.uint8) for _ in range(NB)]
    n_h = ct().ct_run_host_batches(m, xh, B, lh, sh, fh)
    # the same batches through the device call, with the same fault armed
    m2, _, _ = _armed_model(B + 8)
    xs = [torch.from_numpy(a).cuda() for a in xh]
    lg = [torch.empty(B, m.n_classes, device="cuda") for _ in range(NB)]
    S = [torch.empty(B, device="cuda") for _ in range(NB)]
    fl = [torch.empty(B, dtype=torch.uint8, device="cuda") for _ in range(NB)]
    n_d = ct().ct_infer_batches(m2, xs, B, lg, S, fl)
    assert n_h == n_d == 1
    for i in range(NB):
        assert np.array_equal(lh[i], lg[i].cpu().numpy()), i
        assert np.array_equal(sh[i], S[i].cpu().numpy()), i
        assert np.array_equal(fh[i], fl[i].cpu().numpy()), i
    assert_parity(np.concatenate(lh).astype(np.float64), np.concatenate(sh).astype(np.float64), o["logits"], o["S"],
                  "fp32", "host batches")
    # a second call reuses the library's slots
    assert ct().ct_run_host_batches(m, xh[:2], B, lh[:2], None, None) == 0


def test_lenet5_whole_network_kernel_reruns_inside_the_kernel():
    """LeNet-5 runs as one whole-network kernel per batch; a flagged image's
    re-run is a row of that same kernel (it reads the image from the earlier
    batch and writes its logits and S there).  An activation flip (bit 30 of
    the largest checksum value of conv2's input, image 5 of batch 0) makes S
    explode; after the call every image matches the oracle."""
    import torch
    name, Bl, nb = "lenet5", 16, 4
    net = onet(name, "fp32")
    x = inputs(name, Bl * nb)
    o = oracle.forward(net, x, keep=True)
    m = model(name, max_batch=Bl + 8)
    r = float(np.mean(o["S"]))
    ct().ct_set_threshold(m, r, float(np.abs(o["S"] - r).max()) * 1.01)
    cs = o["acts"][5][2][-1]                        # checksum plane of conv2's input, image 5
    kept = np.zeros_like(cs, dtype=bool)
    kept[2:-2, 2:-2] = True                         # the centre taps conv2 (5x5, no padding) samples
    pix = int(np.argmax(np.where(kept, cs, -1.0)))
    assert 0.5 <= cs.reshape(-1)[pix] < 2.0
    per = int(np.prod(oracle.act_shape(net, 2, 1)[1:]))
    ct().ct_inject(m, 1, 2, 5 * per + (per - cs.size) + pix, 30)
    xs = [torch.from_numpy(x[i * Bl:(i + 1) * Bl]).cuda() for i in range(nb)]
    lg = [torch.full((Bl, m.n_classes), float("nan"), device="cuda") for _ in range(nb)]
    S = [torch.full((Bl,), float("nan"), device="cuda") for _ in range(nb)]
    fl = [torch.full((Bl,), 7, dtype=torch.uint8, device="cuda") for _ in range(nb)]
    n = ct().ct_infer_batches(m, xs, Bl, lg, S, fl)
    flags = torch.cat(fl).cpu().numpy()
    assert flags[5] == 1 and flags.sum() == 1 and n == 1, (flags.nonzero(), n)
    assert_parity(torch.cat(lg).cpu().numpy().astype(np.float64), torch.cat(S).cpu().numpy().astype(np.float64),
                  o["logits"], o["S"], "fp32", "lenet5 batches")
    assert ct().ct_launches_per_infer(m) == 1
    assert ct().ct_device_error(m) == 0
