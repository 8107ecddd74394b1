"""Helpers shared by the GPU tests: run the CUDA path through the C ABI and
compare it with the oracle."""
import functools

import numpy as np

import oracle
import synth
from _cache import params

TOL = {"fp32": 1e-4, "fp16": 2e-2}


@functools.lru_cache(maxsize=None)
def onet(name: str, prec: str, protected: bool = True, ds_mode: str = "pass"):
    wl = synth.workload(name)
    return oracle.build_workload(wl, prec, protected, ds_mode, params=params(name))


def ct():
    from paper_2609_16742_gb300 import build
    build.build()
    import paper_2609_16742_gb300 as ct
    return ct


def model(name: str, prec: str = None, protect: bool = True, simt_only: bool = False,
          max_batch: int = None, ds_mode: str = "pass", layerwise: bool = False):
    wl = synth.workload(name)
    return ct().ct_build_workload(wl, params(name), precision=prec or wl.precision,
                                  protect=protect, simt_only=simt_only,
                                  max_batch=max_batch or wl.batch, ds_mode=ds_mode, layerwise=layerwise)


def run(m, x_np):
    import torch
    x = torch.from_numpy(np.ascontiguousarray(x_np, dtype=np.float32)).cuda()
    B = x.shape[0]
    logits = torch.full((B, m.n_classes), float("nan"), device="cuda")
    S = torch.full((B,), float("nan"), device="cuda")
    flag = torch.full((B,), 7, dtype=torch.uint8, device="cuda")
    ct().ct_infer(m, x, B, logits, S, flag)
    torch.cuda.synchronize()
    return logits.cpu().numpy().astype(np.float64), S.cpu().numpy().astype(np.float64), \
        flag.cpu().numpy()


def rel_err_rows(gpu, ref):
    """max_j |gpu - ref| / max(||ref||_inf, 1e-6), per row."""
    gpu = np.atleast_2d(gpu)
    ref = np.atleast_2d(ref)
    norm = np.maximum(np.abs(ref).max(axis=1), 1e-6)
    return np.abs(gpu - ref).max(axis=1) / norm


def assert_parity(lg, Sg, lo, So, prec, what=""):
    tol = TOL[prec]
    e = rel_err_rows(lg, lo)
    assert (e <= tol).all(), "%s logits rel err %s > %g" % (what, e.max(), tol)
    es = np.abs(Sg - So) / np.maximum(np.abs(So), 1e-6)
    assert (es <= tol).all(), "%s S rel err %s > %g" % (what, es.max(), tol)


def same_class(a: float, b: float) -> bool:
    """Both NaN, both the same infinity, or both finite."""
    if np.isnan(a) or np.isnan(b):
        return bool(np.isnan(a) and np.isnan(b))
    if np.isinf(a) or np.isinf(b):
        return a == b
    return True


def kept_checksum_pixel(net, x1, slot, n_ds=3):
    """Flat index of the largest checksum value of `slot` (image x1) among the
    positions that n_ds stride-2 pass-through shortcuts keep (row, col = 0 mod
    2**n_ds); checksum values elsewhere are dropped by the shortcuts before
    they reach S."""
    cs = oracle.forward(net, x1, keep=True)["acts"][0][slot][-1]
    kept = np.zeros_like(cs, dtype=bool)
    kept[::2 ** n_ds, ::2 ** n_ds] = True
    pix = int(np.argmax(np.where(kept, cs, -1.0)))
    return pix, float(cs.reshape(-1)[pix])


def ulp16(x):
    """Spacing of binary16 values at |x| (normal range; 2**-24 below it)."""
    a = np.abs(np.asarray(x, dtype=np.float64))
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -14)))
    return 2.0 ** (e - 10)


def near_threshold(S_o, r, tau, prec, S_g=None):
    """Images on which the GPU and the oracle may legitimately decide
    differently: the oracle's S lies within 1% of tau of the threshold (the
    stated band), or -- FP16 storage only -- the two S values fall on opposite
    sides of the threshold while differing by at most two binary16 ulps of S.
    With FP16 storage S is an FP32 sum of FP16-rounded features, the largest
    of which (the carried checksum) is close to S itself; two correct
    implementations that accumulate in different orders can round it one ulp
    apart (16 at S ~ 3.2e4 on VGG-16, against 1% of tau ~ 1.4)."""
    S_o = np.asarray(S_o, dtype=np.float64)
    near = np.isfinite(S_o) & (np.abs(np.abs(S_o - r) - tau) <= 0.01 * tau)
    if prec == "fp16" and S_g is not None:
        S_g = np.asarray(S_g, dtype=np.float64)
        import oracle
        straddle = oracle.verdict(S_g, r, tau) != oracle.verdict(S_o, r, tau)
        near |= np.isfinite(S_o) & np.isfinite(S_g) & straddle & (np.abs(S_g - S_o) <= 2.0 * ulp16(S_o))
    return near
