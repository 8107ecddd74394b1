"""CPU checks of the C-ABI library: it builds, loads and exports every symbol
that include/ct.h declares; host-only entry points behave as specified."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def ct():
    from paper_2609_16742_gb300 import build
    build.build()
    import paper_2609_16742_gb300 as ct
    return ct


def declared_symbols():
    src = ""
    inc = os.path.join(ROOT, "include")
    for f in sorted(os.listdir(inc)):
        if f.endswith(".h"):
            src += open(os.path.join(inc, f)).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ct_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for s in ("ct_build", "ct_infer", "ct_inject", "ct_reexecute", "ct_set_threshold"):
        assert s in syms


def test_library_exports_every_declared_symbol(ct):
    lib = ctypes.CDLL(ct.LIB_PATH)
    missing = [s for s in declared_symbols() if not hasattr(lib, s)]
    assert not missing, missing
    assert sorted(ct.EXPORTS) == declared_symbols()


def test_strerror(ct):
    assert ct.lib().ct_strerror(0) == b"ok"
    assert b"range" in ct.lib().ct_strerror(5)


def test_calibrate_matches_hand_example(ct):
    S = np.arange(100, dtype=np.float32)
    r, tau = ct.ct_calibrate(S, 0.10)
    assert r == 49.5 and tau == 44.5


def test_calibrate_agrees_with_oracle(ct):
    rng = np.random.default_rng(1)
    for n, alpha in [(1, 0.0), (7, 0.3), (1000, 0.01), (4096, 0.05)]:
        S = (rng.standard_normal(n) * 40 + 1000).astype(np.float32)
        r1, t1 = ct.ct_calibrate(S, alpha)
        r2, t2 = oracle.calibrate(S.astype(np.float64), alpha)
        assert abs(r1 - r2) <= 1e-12 * abs(r2)
        assert abs(t1 - t2) <= 1e-9 * max(abs(t2), 1.0)


def test_calibrate_rejects_bad_input(ct):
    with pytest.raises(ct.CtError):
        ct.ct_calibrate(np.array([1.0, np.nan], np.float32), 0.01)
    with pytest.raises(ct.CtError):
        ct.ct_calibrate(np.array([1.0], np.float32), 1.0)


def test_build_without_device_fails_cleanly(ct):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a device is present")
    import synth
    wl = synth.workload("lenet5")
    with pytest.raises(ct.CtError) as ei:
        ct.ct_build_workload(wl)
    assert ei.value.status == 3          # CT_ECUDA


def test_fi_threshold_matches_oracle(ct):
    rng = np.random.default_rng(9)
    S = rng.normal(2000.0, 80.0, 3001).astype(np.float32)
    S[rng.integers(0, 3001, 25)] = np.float32(np.nan)
    S[rng.integers(0, 3001, 5)] = np.float32(np.inf)
    crit = (rng.random(3001) < 0.03).astype(np.uint8)
    for alpha in (0.0, 0.001, 0.01, 0.05, 0.5):
        got = ct.ct_fi_threshold(S, crit, 2001.5, alpha)
        assert got == oracle.fi_threshold(S.astype(np.float64), crit, 2001.5, alpha)
    with pytest.raises(ct.CtError):
        ct.ct_fi_threshold(S, np.ones(3001, np.uint8), 0.0, 0.01)


@pytest.mark.parametrize("name", ["lenet5", "resnet18_cifar", "resnet18_imagenet", "vgg16",
                                  "mobilenetv2_cifar"])
def test_library_derives_the_residual_roles(ct, name):
    """Sec. II-A residual rule in the library (host only): with every role left
    to the library (CT_ROLE_AUTO) it derives the declared roles; the declared
    roles pass unchanged."""
    import dataclasses
    import synth
    wl = synth.workload(name)
    declared = [L.ct if L.op == "conv" else None for L in wl.layers]
    auto = [dataclasses.replace(L, ct="auto") if L.op == "conv" else L for L in wl.layers]
    got = ct.ct_resolve_roles(auto, wl.in_shape, wl.n_classes)
    # depthwise layers: the library keeps the role it is given and decides the
    # pass-through when it builds them; compare the dense convolutions
    dense = [i for i, L in enumerate(wl.layers) if L.op == "conv" and L.groups == 1]
    assert [got[i] for i in dense] == [declared[i] for i in dense]
    assert ct.ct_resolve_roles(wl.layers, wl.in_shape, wl.n_classes) == declared


def test_library_rejects_a_filter_the_residual_rule_forbids(ct):
    """A block whose first convolution is labelled "ct" (its input is also the
    shortcut) is rejected by ct_resolve_roles and by ct_build before any
    device work (CT_EINVAL), GPU or not."""
    import dataclasses
    import synth
    wl = synth.workload("resnet18_cifar")
    first = next(i for i, L in enumerate(wl.layers) if L.op == "conv" and L.ct == "none")
    bad = [dataclasses.replace(L, ct="ct") if i == first else L for i, L in enumerate(wl.layers)]
    with pytest.raises(ct.CtError) as ei:
        ct.ct_resolve_roles(bad, wl.in_shape, wl.n_classes)
    assert ei.value.status == 1
    params = [{} for _ in bad]
    with pytest.raises(ct.CtError) as ei:
        ct.ct_build(bad, params, wl.in_shape, wl.n_classes, max_batch=1)
    assert ei.value.status == 1
    # a downsample shortcut labelled "ct" breaks the rule too
    ds = next(i for i, L in enumerate(wl.layers) if L.op == "conv" and L.ct == "pass")
    bad = [dataclasses.replace(L, ct="ct") if i == ds else L for i, L in enumerate(wl.layers)]
    with pytest.raises(ct.CtError):
        ct.ct_resolve_roles(bad, wl.in_shape, wl.n_classes)


def test_no_multicast_load_in_the_library():
    """The library runs on every rank of a multi-GPU run: no TMA load may use
    cluster multicast (mbarrier arrivals of tcgen05.commit are not loads)."""
    csrc = os.path.join(ROOT, "paper_2609_16742_gb300", "csrc")
    for f in sorted(os.listdir(csrc)):
        txt = open(os.path.join(csrc, f)).read()
        for line in txt.splitlines():
            if "cp.async.bulk" in line:
                assert "multicast" not in line, (f, line)
