"""Training-time model of dual-batch learning (Sec. 3.2), calibrated on this GPU.

Eq. 2 takes the time of one training batch as a linear function ``a*x + b`` of the
batch size x, so that an epoch over d samples takes ``(a*x + b) * ceil(d/x)``; the
coefficients come from a least-squares line through measured batch times.  With
them the closed forms of Sec. 3.3 (Eqs. 4-8, ``dbl_plan``) give each worker's data
amount, the small batch size B_S and the small worker's update factor.

Here one batch is one single-worker iteration of the training step as the bench
runs it: the resize to the stage resolution, forward and backward of ResNet-18
and the parameter-server merge of its one push, replayed as a CUDA graph and
timed with CUDA events (inputs resident on the device).

    python -m paper_2509_26092_gb300.time_model --variant imagenet --res 128 160 224 \\
        --batches 64 128 192 256 384 512
"""
import argparse
import json
import math


def fit_linear(batches, times):
    """Least-squares a, b of t = a*x + b (Eq. 2) and the coefficient of determination."""
    n = len(batches)
    if n < 2 or len(times) != n:
        raise ValueError("fit_linear: need at least two (batch, time) pairs")
    mx = sum(batches) / n
    mt = sum(times) / n
    sxx = sum((x - mx) ** 2 for x in batches)
    if sxx == 0.0:
        raise ValueError("fit_linear: the batch sizes must not all be equal")
    sxt = sum((x - mx) * (t - mt) for x, t in zip(batches, times))
    a = sxt / sxx
    b = mt - a * mx
    ss_res = sum((a * x + b - t) ** 2 for x, t in zip(batches, times))
    ss_tot = sum((t - mt) ** 2 for t in times)
    r2 = 1.0 - ss_res / ss_tot if ss_tot > 0.0 else 1.0
    return a, b, r2


def epoch_time(a, b, x, d):
    """Eq. 2: the time of an epoch of d samples at batch size x."""
    return (a * x + b) * math.ceil(d / x)


def plan(a, b, k, d, n_small, n_large, batch_large, sqrt_scheme=False):
    """Eqs. 4-8 for the fitted a, b (the library's planner)."""
    from . import dbl as D
    d_l, d_s, b_s, f_s = D.dbl_plan(k, d, n_small, n_large, a, b, batch_large, sqrt_scheme)
    return {"k": k, "d": d, "n_small": n_small, "n_large": n_large, "batch_large": batch_large,
            "d_large": d_l, "d_small": d_s, "batch_small": b_s, "batch_small_floor": math.floor(b_s),
            "f_small": f_s}


def measure(variant, classes, res, native, batches, reps=10, warmup=3, device="cuda"):
    """Seconds per single-worker iteration at each batch size: the mean over ``reps``
    replays of the iteration's CUDA graph after ``warmup`` replays."""
    import torch

    from . import dbl as D
    from . import resnet18 as R
    from . import synth

    spec = R.ResNet18Spec(variant, classes)
    server = R.ServerState(spec, synth.params(spec.table(), seed=0), synth.momentum_state(spec.table(), 0.0, seed=0))
    out = []
    for x in batches:
        worker = R.Worker(spec, x, res, device)
        it = R.DualBatchIteration(server, worker, None, native)
        it.set_inputs(torch.from_numpy(synth.images_u8(x, native, native, 3, seed=1)).to(device),
                      torch.from_numpy(synth.labels(x, classes, seed=1)).to(device))
        it.capture()
        for _ in range(warmup):
            it.run()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            it.run()
        e1.record()
        torch.cuda.synchronize()
        if D.dbl_device_status() != D.DBL_OK:
            raise RuntimeError("time_model: a device-side wait timed out")
        out.append(e0.elapsed_time(e1) * 1e-3 / reps)
        del it, worker
        torch.cuda.empty_cache()
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--variant", default="imagenet", choices=("imagenet", "cifar"))
    ap.add_argument("--res", type=int, nargs="+", default=[128, 160, 224])
    ap.add_argument("--batches", type=int, nargs="+", default=[64, 128, 192, 256, 384, 512])
    ap.add_argument("--k", type=float, nargs="+", default=[1.05, 1.1])
    ap.add_argument("--batch-large", type=int, default=512)
    args = ap.parse_args(argv)
    import torch

    from . import build_lib
    build_lib.build()
    torch.cuda.set_device(0)
    classes, native, d = (1000, 224, 1281167) if args.variant == "imagenet" else (100, 32, 50000)
    for res in args.res:
        times = measure(args.variant, classes, res, native, args.batches)
        a, b, r2 = fit_linear(args.batches, times)
        worst = max(abs(a * x + b - t) / t for x, t in zip(args.batches, times))
        # one large- and one small-batch worker, as in the two-stream step
        plans = []
        for k in args.k:
            try:
                plans.append(plan(a, b, k, d, 1, 1, args.batch_large))
            except Exception as e:  # no positive B_S for this k (DBL_ERR_INVALID)
                plans.append({"k": k, "error": str(e)})
        print(json.dumps({"variant": args.variant, "res": res, "batches": args.batches,
                          "ms_per_batch": [round(t * 1e3, 4) for t in times], "a_ms_per_image": a * 1e3,
                          "b_ms_per_batch": b * 1e3, "b_over_a": b / a, "r2": r2, "max_rel_residual": worst,
                          "plans": plans}), flush=True)
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
