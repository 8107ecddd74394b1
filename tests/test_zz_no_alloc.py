"""ct_reexecute_noalloc: re-execution for callers that cannot allocate device
memory at run time (device memory fixed at start-up, or an allocator owned
by the host application).  Its scratch is a static device array instead of
buffers made by ct_build; its results must equal ct_reexecute's.  This file
is collected last on purpose."""
import numpy as np
import pytest

import oracle
from _cache import inputs
from _gpu import TOL, assert_parity, ct, model, onet, run

pytestmark = pytest.mark.gpu


def _flagging_threshold(m, S):
    """A threshold that flags roughly half of the images (both entry points
    then re-run the same, non-trivial set)."""
    r = float(np.median(S))
    ct().ct_set_threshold(m, r, float(np.median(np.abs(S - r))))


def test_noalloc_reexecute_matches_reexecute_twice():
    import torch
    name, B = "resnet18_cifar", 16
    m = model(name, max_batch=B)
    x = inputs(name, B)
    _, S0, _ = run(m, x)
    _flagging_threshold(m, S0)
    xd = torch.from_numpy(x).cuda()
    for call in range(2):                       # two calls in a row
        lg = torch.empty(B, m.n_classes, device="cuda")
        S = torch.empty(B, device="cuda")
        fl = torch.empty(B, dtype=torch.uint8, device="cuda")
        # corrupt the rows first so that a re-run that writes nothing is caught
        ct().ct_infer(m, xd, B, lg, S, fl)
        flags = fl.clone()
        lg_a, S_a = lg.clone(), S.clone()
        lg_a[flags.bool()] = float("nan")
        S_a[flags.bool()] = float("nan")
        lg_b, S_b = lg_a.clone(), S_a.clone()
        n_a = ct().ct_reexecute(m, xd, B, flags, lg_a, S_a)
        n_b = ct().ct_reexecute_noalloc(m, xd, B, flags, lg_b, S_b)
        torch.cuda.synchronize()
        assert 0 < n_a < B and n_b == n_a, (call, n_a, n_b)
        a, b = lg_a.cpu().numpy(), lg_b.cpu().numpy()
        assert np.isfinite(b).all()
        err = np.abs(a - b).max(axis=1) / np.maximum(np.abs(a).max(axis=1), 1e-6)
        assert (err <= TOL["fp32"]).all(), (call, err.max())
        sa, sb = S_a.cpu().numpy(), S_b.cpu().numpy()
        assert (np.abs(sa - sb) <= TOL["fp32"] * np.abs(sa)).all(), call
        # and the re-run rows against the oracle (Sec. II-B: a fault-free
        # re-execution of the flagged images)
        rows = np.nonzero(flags.cpu().numpy())[0][:3]
        o = oracle.forward(onet(name, "fp32"), x[rows])
        assert_parity(b[rows], sb[rows], o["logits"], o["S"], "fp32", "noalloc re-run rows")


def test_noalloc_rejects_a_batch_beyond_its_scratch():
    import torch
    # 3 x 224 x 224 fp32 images are 602,112 bytes: 32 flagged images need
    # about 19 MB of scratch, more than the 16 MiB array
    name, B = "resnet18_imagenet", 32
    m = model(name, max_batch=B)
    xd = torch.from_numpy(inputs(name, B)).cuda()
    fl = torch.ones(B, dtype=torch.uint8, device="cuda")
    lg = torch.zeros(B, m.n_classes, device="cuda")
    S = torch.zeros(B, device="cuda")
    with pytest.raises(ct().CtError) as ei:
        ct().ct_reexecute_noalloc(m, xd, B, fl, lg, S)
    assert ei.value.status == 5                # CT_ERANGE
    assert float(lg.abs().sum()) == 0.0        # nothing ran
    fl[2:] = 0                                  # two images fit
    assert ct().ct_reexecute_noalloc(m, xd, B, fl, lg, S) == 2
    torch.cuda.synchronize()
    assert np.isfinite(lg[:2].cpu().numpy()).all() and float(lg[2:].abs().sum()) == 0.0


def test_noalloc_leaves_device_free_memory_unchanged():
    """The reason the entry point exists: a call takes no device memory.  A
    re-run of 8 flagged 3x224x224 images needs ~5 MB of scratch; after the
    model's kernels have run once (so their modules are loaded), the device's
    free memory is the same before and after two calls."""
    import torch
    name, B = "resnet18_imagenet", 8
    m = model(name, max_batch=B)
    xd = torch.from_numpy(inputs(name, B)).cuda()
    lg = torch.zeros(B, m.n_classes, device="cuda")
    S = torch.zeros(B, device="cuda")
    fl = torch.ones(B, dtype=torch.uint8, device="cuda")
    lg0 = torch.zeros_like(lg)
    ct().ct_infer(m, xd, B, lg0, None, None)       # loads the modules of a batch-8 inference
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(2):
        assert ct().ct_reexecute_noalloc(m, xd, B, fl, lg, S) == B
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    a, b = lg0.cpu().numpy(), lg.cpu().numpy()
    err = np.abs(a - b).max(axis=1) / np.maximum(np.abs(a).max(axis=1), 1e-6)
    assert (err <= TOL["fp16"]).all()
