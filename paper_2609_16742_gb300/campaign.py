"""Fault-injection campaign (Sec. III-A) on the CIFAR-shaped ResNet-18.

One trial = one seeded single-bit flip, drawn uniformly over the union of
(element, bit) pairs of every convolution weight tensor and every
convolution input activation tensor (ct_buffer_info), injected into one
inference of a fixed batch (ct_inject + ct_infer), followed by
ct_reexecute of the flagged images, as deployed.

A weight flip touches every image of the batch: each image is one trial.
An activation flip touches one image: that image is the trial.  An image is
critical when its top-1 class differs from the fault-free run (a NaN logit
counts as class -1, so it is always critical; ties go to the lowest index),
detected when it is critical and flagged, a false alarm when it is flagged
but not critical.

Weights are those of the CIFAR ResNet-18 workload; evaluation and
calibration inputs use the campaign workload's seeds.  The threshold
(reference r and tau) is calibrated on calib_images fault-free images at
alpha (nearest-rank quantile of |S - r|).

    python -m paper_2609_16742_gb300.campaign --precision fp16 --faults 100000

prints one JSON object.  The bookkeeping runs on the GPU (torch ops on the
library's outputs); the host only draws the fault list and launches.

With --sweep it instead compares the two threshold methods of Sec. II-C
over alpha in {0.1, 1, 5}% (Sec. III-A): the distribution-based tau from
fault-free calibration images, and the FI-based tau from a campaign on the
calibration images (at most alpha of its non-critical trials flagged), each
scored on a campaign with other faults on the evaluation images: TPR, FPR
and Youden's J = TPR - FPR.
"""
import argparse
import json
import os
import sys
import time


def _setup(precision, batch, calib_images, device):
    """Model, workload and fault-free calibration S values."""
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import torch
    import synth
    import paper_2609_16742_gb300 as ct

    torch.cuda.set_device(device)
    net = synth.workload("resnet18_cifar")            # weights
    wl = synth.workload("campaign_resnet18_cifar")    # evaluation and calibration inputs
    B = batch or wl.batch
    m = ct.ct_build_workload(net, synth.make_params(net.layers, net.seed), precision=precision, max_batch=B,
                             device=device)
    stream = torch.cuda.current_stream()
    n_cal = ((calib_images + B - 1) // B) * B
    xc = torch.from_numpy(synth.make_input(wl, batch=n_cal, seed=wl.calib_seed)).cuda()
    Sc = torch.empty(n_cal, device="cuda")
    lc = torch.empty(B, wl.n_classes, device="cuda")
    for i in range(0, n_cal, B):
        ct.ct_infer(m, xc[i:i + B], B, lc, Sc[i:i + B], None, stream)
    torch.cuda.synchronize()
    return m, wl, B, stream, Sc.cpu().numpy(), n_cal


def _top1(lg):
    import torch
    return torch.where(torch.isnan(lg).any(1), torch.full((lg.shape[0],), -1, device=lg.device, dtype=torch.long),
                       lg.argmax(1))


def _trials(m, x, B, sites, stream, reexecute=False):
    """Run one campaign on the batch x: per image trial its S and whether it
    was critical (GPU bookkeeping), plus the counters of run()."""
    import torch
    import paper_2609_16742_gb300 as ct
    n_classes = m.n_classes
    logits = torch.empty(B, n_classes, device="cuda")
    S = torch.empty(B, device="cuda")
    flag = torch.empty(B, dtype=torch.uint8, device="cuda")
    ct.ct_infer(m, x, B, logits, S, flag, stream)
    golden = _top1(logits).clone()
    per_img = {}
    for kind, layer, n_el, bits in ct.ct_buffers(m, B):
        if kind == 1:
            per_img[layer] = n_el // B
    S_rec, c_rec = [], []
    n_rerun = 0
    for kind, layer, e, bit in sites.tolist():
        ct.ct_inject(m, kind, layer, e, bit)
        ct.ct_infer(m, x, B, logits, S, flag, stream)
        crit = _top1(logits) != golden
        if kind == 0:
            S_rec.append(S.clone())
            c_rec.append(crit)
        else:
            i = e // per_img[layer]
            S_rec.append(S[i:i + 1].clone())
            c_rec.append(crit[i:i + 1])
        if reexecute:
            n_rerun += ct.ct_reexecute(m, x, B, flag, logits, S, stream)
    torch.cuda.synchronize()
    return torch.cat(S_rec).cpu().numpy(), torch.cat(c_rec).cpu().numpy(), n_rerun


def sweep(precision="fp32", faults=2000, seed_cal=1, seed_eval=2, alphas=(0.001, 0.01, 0.05), batch=None,
          calib_images=10000, device=0):
    """Distribution-based vs FI-based thresholds over alpha (Sec. II-C, III-A)."""
    import numpy as np
    import torch
    import synth
    import paper_2609_16742_gb300 as ct

    m, wl, B, stream, S_ff, n_cal = _setup(precision, batch, calib_images, device)
    bufs = ct.ct_buffers(m, B)
    # FI campaign on calibration images ("training set") and on evaluation images ("test set")
    x_cal = torch.from_numpy(synth.make_input(wl, batch=B, seed=wl.calib_seed)).cuda()
    x_eval = torch.from_numpy(synth.make_input(wl, batch=B)).cuda()
    S_c, crit_c, _ = _trials(m, x_cal, B, synth.draw_faults(bufs, faults, seed_cal), stream)
    S_e, crit_e, _ = _trials(m, x_eval, B, synth.draw_faults(bufs, faults, seed_eval), stream)
    rows = []
    for alpha in alphas:
        r, tau_d = ct.ct_calibrate(S_ff, alpha)
        tau_f = ct.ct_fi_threshold(S_c, crit_c.astype(np.uint8), r, alpha)
        for method, tau in (("distribution", tau_d), ("fi", tau_f)):
            flag = ~(np.abs(S_e.astype(np.float64) - r) <= tau)
            crit = crit_e.astype(bool)
            tpr = float(flag[crit].mean()) if crit.any() else None
            fpr = float(flag[~crit].mean()) if (~crit).any() else None
            rows.append({"method": method, "alpha": alpha, "tau": tau, "reference": r, "tpr": tpr, "fpr": fpr,
                         "youden_j": (tpr - fpr) if tpr is not None and fpr is not None else None})
    best = {}
    for meth in ("distribution", "fi"):
        scored = [row for row in rows if row["method"] == meth and row["youden_j"] is not None]
        best[meth] = max(scored, key=lambda row: row["youden_j"])["alpha"] if scored else None
    out = {"precision": precision, "faults_per_campaign": faults, "batch": B, "calibration_images": n_cal,
           "calibration_trials": int(S_c.size), "calibration_critical": int(crit_c.sum()),
           "evaluation_trials": int(S_e.size), "evaluation_critical": int(crit_e.sum()),
           "table": rows, "best_alpha_by_youden_j": best, "device_error": ct.ct_device_error(m)}
    m.close()
    return out


def run(precision="fp32", faults=1000, seed=0, batch=None, calib_images=10000, alpha=0.01, device=0,
        reexecute=True):
    import numpy as np
    import torch
    import synth
    import paper_2609_16742_gb300 as ct

    m, wl, B, stream, S_ff, n_cal = _setup(precision, batch, calib_images, device)
    r, tau = ct.ct_calibrate(S_ff, alpha)
    ct.ct_set_threshold(m, r, tau)
    # ---- fault-free evaluation batch ----
    x = torch.from_numpy(synth.make_input(wl, batch=B)).cuda()
    logits = torch.empty(B, wl.n_classes, device="cuda")
    S = torch.empty(B, device="cuda")
    flag = torch.empty(B, dtype=torch.uint8, device="cuda")

    top1 = _top1
    ct.ct_infer(m, x, B, logits, S, flag, stream)
    golden = top1(logits).clone()
    ff_flags = int(flag.sum().item())
    # every re-execution graph is captured before anything is timed
    ct.ct_reexecute_prepare(m, B)

    bufs = ct.ct_buffers(m, B)
    sites = synth.draw_faults(bufs, faults, seed)
    per_img = {}
    for kind, layer, n_el, bits in bufs:
        if kind == 1:
            per_img[layer] = n_el // B
    nb = 32 if precision == "fp32" else 16
    # [kind, bit] counters on the GPU: trials, critical, detected, false alarms
    cnt = torch.zeros(2, nb, 4, dtype=torch.long, device="cuda")
    scratch = torch.zeros_like(cnt)

    def trial(kind, layer, e, bit, counters, inject=True):
        """One inference of the batch (with the fault armed when inject),
        the per-image bookkeeping, and the re-execution of its flagged images."""
        if inject:
            ct.ct_inject(m, kind, layer, e, bit)
        ct.ct_infer(m, x, B, logits, S, flag, stream)
        crit = top1(logits) != golden
        fl = flag != 0
        if kind == 0:
            row = torch.stack([torch.full_like(crit, True).sum(), crit.sum(), (crit & fl).sum(),
                               (~crit & fl).sum()])
        else:
            i = e // per_img[layer]
            c, f = crit[i], fl[i]
            row = torch.stack([torch.ones_like(c, dtype=torch.long), c.long(), (c & f).long(),
                               (~c & f).long()])
        counters[kind, bit] += row
        return ct.ct_reexecute(m, x, B, flag, logits, S, stream) if reexecute else 0

    # fault-free time of the same steps (the same bookkeeping and re-execution,
    # no fault armed) for the relative cost
    n_ff = min(200, max(20, faults // 50))
    ff_sites = sites[np.arange(n_ff) % len(sites)].tolist()
    for kind, layer, e, bit in ff_sites[:5]:
        trial(kind, layer, e, bit, scratch, inject=False)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for kind, layer, e, bit in ff_sites:
        trial(kind, layer, e, bit, scratch, inject=False)
    torch.cuda.synchronize()
    ff_step_s = (time.perf_counter() - t0) / n_ff

    # ---- campaign ----
    n_rerun = 0
    ct.ct_kernel_count(m)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for kind, layer, e, bit in sites.tolist():
        n_rerun += trial(kind, layer, e, bit, cnt)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    kernels = ct.ct_kernel_count(m)
    err = ct.ct_device_error(m)
    c = cnt.cpu().numpy()

    def summary(a):
        trials, crit, det, fa = (int(v) for v in a)
        non = trials - crit
        return {"trials": trials, "critical": crit, "detected": det, "false_alarms": fa,
                "detected_fraction_of_critical": det / crit if crit else None,
                "false_alarm_rate": fa / non if non else None}

    tot = c.sum(axis=(0, 1))
    out = {
        "precision": precision, "faults": int(faults), "seed": int(seed), "batch": B,
        "threshold": {"reference": r, "tau": tau, "alpha": alpha, "calibration_images": n_cal},
        "fault_free_flagged_images": ff_flags,
        "all": summary(tot),
        "weights": summary(c[0].sum(axis=0)),
        "activations": summary(c[1].sum(axis=0)),
        "by_bit": {str(b): summary(c[:, b].sum(axis=0)) for b in range(nb)},
        "wall_s": wall,
        "fault_free_wall_s": ff_step_s * faults,
        "time_relative_to_fault_free": wall / (ff_step_s * faults),
        "reexecuted_images": n_rerun,
        "kernels_launched": kernels,
        "device_error": err,
    }
    m.close()
    return out


def run_batched(faults=100000, seed=0, calib_images=10000, alpha=0.01, device=0):
    """The campaign of run() on LeNet-5 (FP32) with ct_campaign_batched: all
    faults in one launch (no re-execution).  Returns the same counters."""
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import numpy as np
    import torch
    import synth
    import paper_2609_16742_gb300 as ct

    torch.cuda.set_device(device)
    wl = synth.workload("lenet5")
    B = wl.batch
    m = ct.ct_build_workload(wl, synth.make_params(wl.layers, wl.seed), max_batch=B, device=device)
    stream = torch.cuda.current_stream()
    n_cal = ((calib_images + B - 1) // B) * B
    xc = torch.from_numpy(synth.make_input(wl, batch=n_cal, seed=wl.calib_seed)).cuda()
    Sc = torch.empty(n_cal, device="cuda")
    lc = torch.empty(B, wl.n_classes, device="cuda")
    for i in range(0, n_cal, B):
        ct.ct_infer(m, xc[i:i + B], B, lc, Sc[i:i + B], None, stream)
    torch.cuda.synchronize()
    r, tau = ct.ct_calibrate(Sc.cpu().numpy(), alpha)
    ct.ct_set_threshold(m, r, tau)
    x = torch.from_numpy(synth.make_input(wl, batch=B)).cuda()
    logits = torch.empty(B, wl.n_classes, device="cuda")
    ct.ct_infer(m, x, B, logits, None, None, stream)
    golden = _top1(logits).to(torch.int32)
    bufs = ct.ct_buffers(m, B)
    sites = synth.draw_faults(bufs, faults, seed)
    F = len(sites)
    S = torch.full((F, B), float("nan"), device="cuda")
    top1 = torch.full((F, B), -2, dtype=torch.int32, device="cuda")
    flag = torch.zeros((F, B), dtype=torch.uint8, device="cuda")
    ct.ct_campaign_batched(m, x, B, sites[:1], S, top1, flag, stream)      # warm-up
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    ct.ct_campaign_batched(m, x, B, sites, S, top1, flag, stream)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    # trials: every image of a weight fault, the hit image of an activation fault
    valid = top1 != -2
    crit = valid & (top1 != golden[None, :])
    fl = valid & (flag != 0)
    kinds = torch.from_numpy(np.ascontiguousarray(sites[:, 0])).cuda()

    def summary(sel):
        v, c, f_ = valid[sel], crit[sel], fl[sel]
        trials, critical = int(v.sum()), int(c.sum())
        det, fa = int((c & f_).sum()), int((~c & f_ & v).sum())
        non = trials - critical
        return {"trials": trials, "critical": critical, "detected": det, "false_alarms": fa,
                "detected_fraction_of_critical": det / critical if critical else None,
                "false_alarm_rate": fa / non if non else None}

    out = {"network": "lenet5", "precision": "fp32", "faults": F, "seed": seed, "batch": B,
           "threshold": {"reference": r, "tau": tau, "alpha": alpha, "calibration_images": n_cal},
           "all": summary(slice(None)), "weights": summary(kinds == 0), "activations": summary(kinds == 1),
           "wall_s": wall, "faults_per_s": F / wall, "device_error": ct.ct_device_error(m)}
    m.close()
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--precision", default="fp32", choices=["fp32", "fp16"])
    ap.add_argument("--faults", type=int, default=1000)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--calib-images", type=int, default=10000)
    ap.add_argument("--alpha", type=float, default=0.01)
    ap.add_argument("--no-reexecute", action="store_true")
    ap.add_argument("--batched-lenet", action="store_true",
                    help="LeNet-5 FP32 campaign, all faults in one launch (ct_campaign_batched)")
    ap.add_argument("--sweep", action="store_true",
                    help="compare distribution-based and FI-based thresholds over alpha in {0.1, 1, 5}%%")
    args = ap.parse_args(argv)
    if args.batched_lenet:
        out = run_batched(args.faults, args.seed, calib_images=args.calib_images, alpha=args.alpha)
        print(json.dumps(out))
        return 0 if out["device_error"] == 0 else 1
    if args.sweep:
        out = sweep(args.precision, args.faults, seed_cal=args.seed + 1, seed_eval=args.seed + 2,
                    calib_images=args.calib_images)
        print(json.dumps(out))
        return 0 if out["device_error"] == 0 else 1
    out = run(args.precision, args.faults, args.seed, calib_images=args.calib_images, alpha=args.alpha,
              reexecute=not args.no_reexecute)
    print(json.dumps(out))
    return 0 if out["device_error"] == 0 else 1


if __name__ == "__main__":
    sys.exit(main())
