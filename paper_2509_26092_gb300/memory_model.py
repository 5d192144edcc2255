"""Memory model of Sec. 6 (Eq. 9), calibrated on this GPU: the largest batch size B_L.

Eq. 9 takes the device memory of training at batch size B as a constant (the
parameters and everything else that does not grow with the batch) plus B times
the per-sample activation memory, M(B) = P + B*A, fitted by least squares to the
peak memory of training at several batch sizes.  B_max is the largest B with
M(B) <= M_GPU.

Every device buffer of the training step comes from PyTorch's caching allocator
(the library allocates nothing), so the allocator's peak over one iteration is
the step's memory: the parameter server's state, one worker's activations,
gradients and scratch, and the input images.

    python -m paper_2509_26092_gb300.memory_model --variant imagenet --res 128 160 224
"""
import argparse
import json
import math

from .time_model import fit_linear


def fit_memory(batches, peak_bytes):
    """Least-squares P (bytes) and A (bytes per sample) of M(B) = P + B*A, and R^2."""
    a, p, r2 = fit_linear(batches, peak_bytes)
    return p, a, r2


def max_batch(p, a, m_gpu):
    """The largest B with P + B*A <= M_GPU (0 if not even one sample fits)."""
    if a <= 0.0:
        raise ValueError("max_batch: the per-sample memory must be positive")
    return max(0, math.floor((m_gpu - p) / a))


def measure(variant, classes, res, native, batches, device="cuda"):
    """Peak allocator bytes of one eager single-worker iteration (resize, forward,
    backward, merge) at each batch size, the parameter-server state included."""
    import torch

    from . import dbl as D
    from . import resnet18 as R
    from . import synth

    spec = R.ResNet18Spec(variant, classes)
    server = R.ServerState(spec, synth.params(spec.table(), seed=0), synth.momentum_state(spec.table(), 0.0, seed=0))
    out = []
    for x in batches:
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        torch.cuda.reset_peak_memory_stats()
        worker = R.Worker(spec, x, res, device)
        it = R.DualBatchIteration(server, worker, None, native)
        it.set_inputs(torch.from_numpy(synth.images_u8(x, native, native, 3, seed=1)).to(device),
                      torch.from_numpy(synth.labels(x, classes, seed=1)).to(device))
        it.run()
        torch.cuda.synchronize()
        if D.dbl_device_status() != D.DBL_OK:
            raise RuntimeError("memory_model: a device-side wait timed out")
        out.append(float(torch.cuda.max_memory_allocated()))
        del it, worker
    torch.cuda.empty_cache()
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--variant", default="imagenet", choices=("imagenet", "cifar"))
    ap.add_argument("--res", type=int, nargs="+", default=[128, 160, 224])
    ap.add_argument("--batches", type=int, nargs="+", default=[64, 128, 192, 256, 320, 384, 448, 512])
    ap.add_argument("--check", type=int, default=1024,
                    help="a larger batch size measured to check the model's prediction (0: none)")
    args = ap.parse_args(argv)
    import torch

    from . import build_lib
    build_lib.build()
    torch.cuda.set_device(0)
    classes, native = (1000, 224) if args.variant == "imagenet" else (100, 32)
    m_gpu = float(torch.cuda.get_device_properties(0).total_memory)
    for res in args.res:
        peaks = measure(args.variant, classes, res, native, args.batches)
        p, a, r2 = fit_memory(args.batches, peaks)
        rec = {"variant": args.variant, "res": res, "batches": args.batches, "peak_gb": [round(v / 1e9, 4) for v in peaks],
               "p_gb": p / 1e9, "a_mb_per_sample": a / 1e6, "r2": r2, "m_gpu_gb": m_gpu / 1e9,
               "b_max": max_batch(p, a, m_gpu)}
        if args.check:
            got = measure(args.variant, classes, res, native, [args.check])[0]
            pred = p + a * args.check
            rec.update(check_batch=args.check, check_measured_gb=got / 1e9, check_predicted_gb=pred / 1e9,
                       check_rel_error=(pred - got) / got)
        print(json.dumps(rec), flush=True)
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
