"""Asynchronous dual-batch training (ASP, Sec. 2.4 and 3) and the hybrid
cyclic-progressive schedule (Sec. 4) on one GPU.

Under ASP each worker pushes its gradient the moment its step ends; the server
applies that one push at once (the merge of Sec. 3.4 with a single gradient and
the worker's update factor), and the worker pulls the new model and starts its
next step.  A worker's gradient is therefore computed on the model it pulled
after its previous push, while the other worker's pushes keep moving the
server's model (staleness).  With a large-batch worker whose step takes t_L and a
small-batch worker whose step takes t_S, the k-th push of worker X arrives at
k*t_X; ``push_order`` merges the two sequences (a tie goes to the large worker).

``AsyncDualBatch`` runs that order on the GPU: the two workers compute on their
own streams, each from its own pulled copy of the weights, so their steps
overlap; the merges are serialised in push order by CUDA events.  The step times
come from the calibrated time model (``time_model``: t = a*B + b, Eq. 2).

``hybrid_schedule`` gives the paper's hybrid schemes (Table 7 for CIFAR-100 and
Table 9 for ImageNet, Sec. 5.2: three stages of decreasing learning rate, each
cycling through increasing resolutions), and ``run_schedule`` runs one
on synthetic data for a fraction of each epoch; the synthetic source images have
the schedule's largest resolution, so every sub-stage downsamples or passes them
through.  Each sub-stage's workers apply the tables' dropout rate before the FC
layer (inverted dropout with a counter-based mask; each worker has its own seed).
"""
import argparse
import json
import math
from dataclasses import dataclass


def push_order(t_large, t_small, n_large, n_small):
    """Arrival order [(time, 'L'|'S', k)] of n_large pushes at k*t_large and n_small
    pushes at k*t_small (k = 1, 2, ...), by time, the large worker first on a tie."""
    if t_large <= 0.0 or t_small <= 0.0 or n_large < 0 or n_small < 0:
        raise ValueError("push_order: step times must be positive and counts non-negative")
    out, i, j = [], 1, 1
    while i <= n_large or j <= n_small:
        tl = i * t_large if i <= n_large else math.inf
        ts = j * t_small if j <= n_small else math.inf
        if tl <= ts:
            out.append((tl, "L", i))
            i += 1
        else:
            out.append((ts, "S", j))
            j += 1
    return out


class PulledWeights:
    """A worker's copy of the model (fp32 w and the bf16 w16 its convolutions read),
    refreshed by ``pull`` on the worker's stream."""

    def __init__(self, server):
        self.spec, self.precision = server.spec, server.precision
        self.w = server.w.clone()
        self.w16 = server.w16.clone()
        # the loss scale is the server's live state: a worker copies it when its step starts
        self.scaled, self.scale_state = server.scaled, server.scale_state

    def pull(self, server, stream):
        import torch
        with torch.cuda.stream(stream):
            self.w.copy_(server.w, non_blocking=True)
            self.w16.copy_(server.w16, non_blocking=True)


class AsyncDualBatch:
    """Free-running large- and small-batch workers on one GPU, pushes applied in
    arrival order (see the module docstring).  ``images_*``: lists of device image
    batches at the native resolution (uint8 or fp32) with their int32 labels; a
    worker takes them in turn, one per step."""

    def __init__(self, server, large, small, native_res, images_large, labels_large, images_small, labels_small,
                 lr=0.2, momentum=0.9, f_large=1.0, f_small=19.0 / 21.0):
        import torch
        self.server, self.native_res = server, native_res
        self.lr, self.momentum = lr, momentum
        self.workers = {"L": large, "S": small}
        self.factor = {"L": f_large, "S": f_small}
        self.data = {"L": (images_large, labels_large), "S": (images_small, labels_small)}
        self.next_batch = {"L": 0, "S": 0}
        self.streams = {"L": torch.cuda.Stream(), "S": torch.cuda.Stream()}
        self.pulled = {"L": PulledWeights(server), "S": PulledWeights(server)}
        self.losses = {"L": [], "S": []}
        self.done = {}     # tag -> event after the worker's latest step
        self.failed = []   # workers that missed the server's deadline (no further pushes)

    def _launch(self, tag):
        import torch
        wk, s = self.workers[tag], self.streams[tag]
        imgs, labs = self.data[tag]
        b = self.next_batch[tag] % len(imgs)
        self.next_batch[tag] += 1
        with torch.cuda.stream(s):
            wk.labels.copy_(labs[b], non_blocking=True)
        wk.enqueue_step(self.pulled[tag], imgs[b], self.native_res, s)
        self.done[tag] = torch.cuda.Event()
        self.done[tag].record(s)

    def run(self, t_large, t_small, n_large, n_small, on_push=None, deadline_s=None, wait=None):
        """Run n_large + n_small pushes in ``push_order``; returns that order.
        ``on_push(tag, worker, pulled)``, if given, is called when a push has been
        enqueued, after its merge and before the worker pulls (stream ``self.streams[tag]``).
        With ``deadline_s`` the server (the host) waits at most that long for each push's step
        to complete (``wait(event, seconds)``, default ``dbl_event_wait``); a worker that misses
        it is taken as stopped: that push and all its later ones are left out (ASP does not
        wait for it, Sec. 2.4) and its tag is listed in ``self.failed``."""
        import torch

        from . import dbl as D
        from .resnet18 import collect_pushes
        wait = wait or D.dbl_event_wait
        order = push_order(t_large, t_small, n_large, n_small)
        remaining = {"L": n_large, "S": n_small}
        cur = torch.cuda.current_stream()
        srv = self.server
        for tag in ("L", "S"):
            if remaining[tag]:
                self.streams[tag].wait_stream(cur)
                self.pulled[tag].pull(srv, self.streams[tag])
                self._launch(tag)
        last = None  # event after the previous push's merge and pull
        for _, tag, _ in order:
            if tag in self.failed:
                continue
            if deadline_s is not None and collect_pushes({tag: self.done[tag]}, deadline_s, wait)[1]:
                self.failed.append(tag)
                continue
            s, wk = self.streams[tag], self.workers[tag]
            if last is not None:
                s.wait_event(last)
            g_l = wk.grad if tag == "L" else None
            g_s = wk.grad if tag == "S" else None
            srv.apply_pushes(g_l, g_s, wk.scale_used if tag == "L" else None, wk.scale_used if tag == "S" else None,
                             self.lr, self.momentum, self.factor["L"], self.factor["S"], 0, s.cuda_stream)
            with torch.cuda.stream(s):
                self.losses[tag].append(wk.loss.clone())
            if on_push is not None:
                on_push(tag, wk, self.pulled[tag])
            remaining[tag] -= 1
            self.pulled[tag].pull(srv, s)
            last = torch.cuda.Event()
            last.record(s)
            if remaining[tag]:
                self._launch(tag)
        for s in self.streams.values():
            cur.wait_stream(s)
        return order


@dataclass
class SubStage:
    stage: int
    epochs: int
    lr: float
    res: int
    batch_large: int
    dropout: float  # rate of the dropout before the FC layer


def hybrid_schedule(variant):
    """The hybrid scheme's sub-stages: Table 7 (CIFAR-100, 140 epochs at 24 and 32 px) or Table 9
    (ImageNet, 105 epochs at 160, 224 and 288 px)."""
    if variant == "cifar":
        rows = [(1, 40, 0.2, 24, 600, 0.1), (1, 40, 0.2, 32, 560, 0.2), (2, 20, 0.02, 24, 600, 0.1),
                (2, 20, 0.02, 32, 560, 0.2), (3, 10, 0.002, 24, 600, 0.1), (3, 10, 0.002, 32, 560, 0.2)]
    elif variant == "imagenet":
        rows = []
        for stage, ep, lr in ((1, 20, 0.2), (2, 10, 0.02), (3, 5, 0.002)):
            rows += [(stage, ep, lr, 160, 2330, 0.1), (stage, ep, lr, 224, 1110, 0.2), (stage, ep, lr, 288, 740, 0.3)]
    else:
        raise ValueError(f"hybrid_schedule: unknown variant {variant!r}")
    return [SubStage(*r) for r in rows]


def substage_pushes(sub, d, k, a, b, n_small=1, n_large=1, batch_large=None, data_fraction=1.0):
    """Per worker and sub-stage: the planned B_S and f_S (Eqs. 4-8 with the time model a, b),
    the pushes of each worker over the sub-stage's epochs on a fraction of the data, and the
    step times a*B + b."""
    from . import time_model
    bl = batch_large or sub.batch_large
    p = time_model.plan(a, b, k, d, n_small, n_large, bl)
    bs = max(1, p["batch_small_floor"])
    dl, ds = p["d_large"] * data_fraction, p["d_small"] * data_fraction
    return {"batch_large": bl, "batch_small": bs, "f_small": p["f_small"],
            "pushes_large": sub.epochs * max(1, math.ceil(dl / bl)), "pushes_small": sub.epochs * max(1, math.ceil(ds / bs)),
            "t_large": a * bl + b, "t_small": a * bs + b}


def run_schedule(variant, fits, k=1.05, data_fraction=1e-3, batch_large=None, max_batch_small=None, seed=0,
                 momentum=0.9, device="cuda"):
    """Run the hybrid schedule on synthetic data.  fits: {res: (a, b)} of the time model
    (seconds); data_fraction scales each epoch's data.  Returns one record per sub-stage."""
    import torch

    from . import resnet18 as R
    from . import synth
    classes, d = (1000, 1281167) if variant == "imagenet" else (100, 50000)
    native = max(s.res for s in hybrid_schedule(variant))
    spec = R.ResNet18Spec(variant, classes)
    server = R.ServerState(spec, synth.params(spec.table(), seed=seed), synth.momentum_state(spec.table(), 0.0, seed))
    out = []
    for sub in hybrid_schedule(variant):
        a, b = fits[sub.res]
        pl = substage_pushes(sub, d, k, a, b, batch_large=batch_large, data_fraction=data_fraction)
        if max_batch_small:
            pl["batch_small"] = min(pl["batch_small"], max_batch_small)
        bl, bs = pl["batch_large"], pl["batch_small"]
        large = R.Worker(spec, bl, sub.res, device, dropout=sub.dropout, dropout_seed=2 * seed + 1)
        small = R.Worker(spec, bs, sub.res, device, dropout=sub.dropout, dropout_seed=2 * seed + 2)
        imgs = {t: [torch.from_numpy(synth.images_u8(n, native, native, 3, seed=seed + 10 * i + j,
                                                     name=t)).to(device) for i in range(2)]
                for j, (t, n) in enumerate((("L", bl), ("S", bs)))}
        labs = {t: [torch.from_numpy(synth.labels(n, classes, seed=seed + 10 * i + j, name=t)).to(device)
                    for i in range(2)] for j, (t, n) in enumerate((("L", bl), ("S", bs)))}
        run = AsyncDualBatch(server, large, small, native, imgs["L"], labs["L"], imgs["S"], labs["S"], lr=sub.lr,
                             momentum=momentum, f_small=pl["f_small"])
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        order = run.run(pl["t_large"], pl["t_small"], pl["pushes_large"], pl["pushes_small"])
        e1.record()
        torch.cuda.synchronize()
        secs = e0.elapsed_time(e1) * 1e-3
        images = pl["pushes_large"] * bl + pl["pushes_small"] * bs
        loss = {t: [float(x) for x in torch.stack(run.losses[t]).cpu()] for t in ("L", "S")}
        out.append({"stage": sub.stage, "res": sub.res, "lr": sub.lr, "epochs": sub.epochs,
                    "dropout": sub.dropout, **pl, "pushes": len(order),
                    "first_pushes": "".join(t for _, t, _ in order[:12]), "seconds": secs,
                    "images_per_s": images / secs, "loss_first": {t: v[0] for t, v in loss.items() if v},
                    "loss_last": {t: v[-1] for t, v in loss.items() if v}})
        del run, large, small
        torch.cuda.empty_cache()
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--variant", default="cifar", choices=("imagenet", "cifar"))
    ap.add_argument("--k", type=float, default=1.05)
    ap.add_argument("--data-fraction", type=float, default=1e-3)
    ap.add_argument("--batch-large", type=int, default=0, help="override the tables' B_L (0: the tables')")
    ap.add_argument("--max-batch-small", type=int, default=0)
    ap.add_argument("--fits", default="", help='JSON {res: [a_seconds, b_seconds]}; default: measure them here')
    args = ap.parse_args(argv)
    import torch

    from . import build_lib, time_model
    build_lib.build()
    torch.cuda.set_device(0)
    classes = 1000 if args.variant == "imagenet" else 100
    native = max(s.res for s in hybrid_schedule(args.variant))
    if args.fits:
        fits = {int(r): tuple(v) for r, v in json.loads(args.fits).items()}
    else:
        fits = {}
        for res in sorted({s.res for s in hybrid_schedule(args.variant)}):
            bs = [64, 128, 256, 384]
            t = time_model.measure(args.variant, classes, res, native, bs, reps=5)
            a, b, _ = time_model.fit_linear(bs, t)
            fits[res] = (a, b)
    for rec in run_schedule(args.variant, fits, k=args.k, data_fraction=args.data_fraction,
                            batch_large=args.batch_large or None, max_batch_small=args.max_batch_small or None):
        print(json.dumps(rec), flush=True)
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
