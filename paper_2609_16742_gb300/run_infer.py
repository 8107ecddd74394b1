"""Run protected inferences of a named synthetic workload on cuda:0, as a
fixed target for external profilers (for example a kernel launch list):

    python -m paper_2609_16742_gb300.run_infer --workload resnet18_imagenet \\
        --batch 256 --iters 2

Inputs and weights are the seeded synthetic ones of the workload.  Each
iteration is one ct_infer of the whole batch; with --reexecute, also one
ct_reexecute of its flagged images (threshold from a seeded calibration
set).  Exits non-zero if a kernel reported a device error.
"""
import argparse
import os
import sys


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workload", default="resnet18_imagenet")
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--precision", default=None, choices=[None, "fp32", "fp16"])
    ap.add_argument("--iters", type=int, default=2)
    ap.add_argument("--unprotected", action="store_true")
    ap.add_argument("--reexecute", action="store_true")
    args = ap.parse_args(argv)

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import torch
    import synth
    import paper_2609_16742_gb300 as ct

    wl = synth.workload(args.workload)
    B = args.batch or wl.batch
    m = ct.ct_build_workload(wl, synth.make_params(wl.layers, wl.seed), precision=args.precision or wl.precision,
                             protect=not args.unprotected, max_batch=B)
    x = torch.from_numpy(synth.make_input(wl, batch=B)).cuda()
    logits = torch.empty(B, wl.n_classes, device="cuda")
    S = torch.empty(B, device="cuda")
    flag = torch.empty(B, dtype=torch.uint8, device="cuda")
    if args.reexecute:
        xc = torch.from_numpy(synth.make_input(wl, batch=B, seed=wl.calib_seed)).cuda()
        Sc = torch.empty(B, device="cuda")
        ct.ct_infer(m, xc, B, logits, Sc, None)
        torch.cuda.synchronize()
        r, tau = ct.ct_calibrate(Sc.cpu().numpy(), 0.01)
        ct.ct_set_threshold(m, r, tau)
    n_re = 0
    for _ in range(args.iters):
        ct.ct_infer(m, x, B, logits, S, flag)
        if args.reexecute:
            n_re += ct.ct_reexecute(m, x, B, flag, logits, S)
    torch.cuda.synchronize()
    err = ct.ct_device_error(m)
    print("workload %s batch %d iters %d re-executed %d kernels/inference %d device_error %#x"
          % (args.workload, B, args.iters, n_re, ct.ct_launches_per_infer(m), err))
    return 0 if err == 0 else 1


if __name__ == "__main__":
    sys.exit(main())
