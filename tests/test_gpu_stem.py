"""The fused image stem (7x7 stride-2 convolution with the carry-through
filter, ReLU and 3x3 stride-2 max-pool in one kernel) against the oracle:
the pooled tensor and its checksum plane, batches whose CTA ranges start
inside an image and span several images, and faults on the stem's weights."""
import numpy as np
import pytest

import oracle
import synth
from _cache import inputs
from _gpu import TOL, ct, model, onet, rel_err_rows, run, same_class

pytestmark = pytest.mark.gpu

NAME = "resnet18_imagenet"
CT_ESTATE, CT_ERANGE = 4, 5


def _pooled(m, batch):
    wl = synth.workload(NAME)
    assert wl.layers[0].op == "conv" and wl.layers[1].op == "maxpool"
    return ct().ct_copy_activation(m, wl.layers[1].dst, batch)


@pytest.mark.parametrize("batch", [1, 3, 8])
def test_pooled_stem_output_matches_oracle(batch):
    wl = synth.workload(NAME)
    m = model(NAME, max_batch=batch)
    x = inputs(NAME, batch)
    run(m, x)
    assert ct().ct_device_error(m) == 0
    gd, gc = _pooled(m, batch)
    net = onet(NAME, "fp16")
    slot = wl.layers[1].dst
    for n in range(batch):
        a = oracle.forward(net, x[n:n + 1], keep=True)["acts"][0][slot]
        ref, refc = a[:64], a[64]
        # both sides round the same FP32 accumulations to FP16; allow one
        # FP16 ulp of the largest value for accumulation-order differences
        tol = TOL["fp16"] * np.abs(ref).max()
        assert np.abs(gd[n] - ref).max() <= tol
        assert np.abs(gc[n] - refc).max() <= TOL["fp16"] * np.abs(refc).max()
        # ReLU then max-pool: no negative values, the same zero pattern up to
        # values that round differently near zero
        assert (gd[n] >= 0).all()
        assert np.mean((gd[n] == 0) != (ref == 0)) < 1e-3


def test_unstored_tensors_of_the_fused_stem():
    wl = synth.workload(NAME)
    m = model(NAME, max_batch=2)
    for slot in (0, wl.layers[0].dst):
        with pytest.raises(ct().CtError) as ei:
            ct().ct_copy_activation(m, slot, 1)
        assert ei.value.status == CT_ESTATE
    with pytest.raises(ct().CtError) as ei:
        ct().ct_inject(m, 1, 0, 0, 3)          # the image is not a fault-able tensor here
    assert ei.value.status == CT_ERANGE
    assert ct().ct_launches_per_infer(m) == len(wl.layers) - 1


def test_stem_weight_faults_match_oracle():
    wl = synth.workload(NAME)
    B = 2
    m = model(NAME, max_batch=B)
    x = inputs(NAME, B)
    net = onet(NAME, "fp16")
    g_lg, g_S, _ = run(m, x)
    Ct, R = 3, 7

    def el(k, c, r, s):
        return ((k * Ct + c) * R + r) * R + s

    cases = [
        (el(5, 1, 2, 5), 14),      # data filter, exponent bit
        (el(9, 0, 3, 3), 13),      # data filter, centre tap
        (el(40, 2, 6, 0), 12),     # data filter, corner tap
        (el(64, 0, 0, 0), 14),     # carry-through row off the centre (stored 0)
        (el(64, 2, 3, 3), 10),     # carry-through coefficient
        (el(64, 1, 5, 4), 15),     # carry-through row, sign bit of a zero
    ]
    for e, bit in cases:
        ct().ct_inject(m, 0, 0, e, bit)
        lg, S, _ = run(m, x)
        o = oracle.forward(net, x, oracle.Fault(0, 0, e, bit))
        for i in range(B):
            so = o["S"][i]
            assert same_class(S[i], so), (e, bit, S[i], so)
            if np.isfinite(so):
                assert abs(S[i] - so) <= TOL["fp16"] * max(abs(so), 1e-6), (e, bit, S[i], so)
            lo = o["logits"][i]
            if np.isfinite(lo).all():
                assert rel_err_rows(lg[i], lo)[0] <= TOL["fp16"], (e, bit)
        # the fault is transient
        again = run(m, x)
        assert np.array_equal(again[0], g_lg) and np.array_equal(again[1], g_S)
