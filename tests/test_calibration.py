"""Sec. II-C / III-A: the distribution-based threshold is the (1 - alpha)
quantile of |S - r| over fault-free calibration images, so about alpha of
other fault-free images exceed it.  LeNet-5 (FP32): S from the oracle, tau
from the library's host routine ct_calibrate (no GPU), the flag rate on
held-out images of another seed."""
import numpy as np

import oracle
import synth
from _gpu import ct

ALPHA = 0.01
N = 4000


def test_calibrated_threshold_flags_about_alpha_of_held_out_images():
    wl = synth.workload("lenet5")
    net = oracle.build_workload(wl, "fp32")
    Sc = oracle.forward(net, synth.make_input(wl, batch=N, seed=wl.calib_seed))["S"]
    Se = oracle.forward(net, synth.make_input(wl, batch=N))["S"]
    r, tau = ct().ct_calibrate(Sc.astype(np.float32), ALPHA)
    assert r == np.float64(np.mean(Sc.astype(np.float32).astype(np.float64)))
    # on the calibration set itself at most alpha exceed tau (nearest rank)
    assert np.mean(oracle.verdict(Sc, r, tau)) <= ALPHA
    # held out: the quantile estimate (~40 exceedances) and the binomial
    # draw of N images each add ~0.16% of spread; 0.9% is about 4 sigma
    rate = float(np.mean(oracle.verdict(Se, r, tau)))
    assert abs(rate - ALPHA) <= 0.009, rate
