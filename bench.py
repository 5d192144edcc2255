#!/usr/bin/env python
"""Benchmark of the ResNet-18 hybrid dual-batch training step on GB300.

Default workload (``imagenet_hybrid``): ImageNet-shaped ResNet-18 (7x7/2 stem,
3x3/2 max pool, 1000 classes), synthetic 224x224 images resized by the
library's bilinear downsampler to the cyclic-progressive sub-stage
resolutions 128, 160 and 224; at each resolution a large-batch worker
(batch 512) and a small-batch worker (batch 128) run concurrently on two CUDA
streams and the parameter server merges both pushes into the fp32 master
weights (11.7 M parameters) with the model-update factor f_S = 19/21.

One benchmark step is one dual-batch iteration at each of the three
resolutions (1920 images).  ``value`` is images/s over the whole job (all
ranks); ``per_resolution`` breaks it down.  Each rank runs an independent
replica (the path has no cross-GPU exchange on one box), so scaling is weak.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl ours|reference]
"""
import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "ResNet-18 train-step images/s per resolution; conv TFLOP/s vs bf16 peak"

CONFIGS = {
    # variant, classes, native resolution, sub-stage resolutions, large / small batch per stage, and the
    # rate of the dropout before the FC layer per stage (Sec. 4.1: it rises with the resolution of the
    # sub-stage, 0.1 / 0.2 / 0.3 in Tables 7 and 9)
    "imagenet_hybrid": dict(variant="imagenet", classes=1000, native=224, stages=(128, 160, 224),
                            large=(512, 512, 512), small=(128, 128, 128), dropout=(0.1, 0.2, 0.3),
                            desc="ImageNet-shaped ResNet-18 hybrid: 224 px images resized to 128/160/224, "
                                 "large worker 512 + small worker 128 on two streams, PS merge each iteration"),
    "imagenet_paper": dict(variant="imagenet", classes=1000, native=288, stages=(160, 224, 288),
                           large=(2330, 1110, 740), small=(582, 277, 185), dropout=(0.1, 0.2, 0.3),
                           desc="the paper's ImageNet hybrid sub-stages (Table 9): 288 px images resized to "
                                "160/224/288, large-batch worker 2330/1110/740 and a small-batch worker of a "
                                "quarter of that on two streams, PS merge each iteration"),
    "cifar_hybrid": dict(variant="cifar", classes=100, native=32, stages=(16, 24, 32), large=(1024, 512, 256),
                         small=(256, 128, 64), dropout=(0.1, 0.1, 0.2),
                         desc="CIFAR-shaped ResNet-18 cyclic progressive sweep 16/24/32 px, dual batch, PS merge"),
    "cifar_step": dict(variant="cifar", classes=100, native=32, stages=(32,), large=(256,), small=(None,),
                       dropout=(0.2,),
                       desc="CIFAR-shaped ResNet-18, one train step at 32x32, batch 256, single push"),
    "imagenet_step": dict(variant="imagenet", classes=1000, native=224, stages=(224,), large=(256,), small=(None,),
                          dropout=(0.2,),
                          desc="ImageNet-shaped ResNet-18, one train step at 224x224, batch 256, single push"),
    "imagenet_small": dict(variant="imagenet", classes=1000, native=224, stages=(224,), large=(32,), small=(8,),
                           dropout=(0.2,), desc="small ImageNet-shaped dual-batch iteration for profiling"),
    "imagenet_profile": dict(variant="imagenet", classes=1000, native=224, stages=(224,), large=(128,), small=(None,),
                             dropout=(0.3,),
                             desc="one 224 px worker of batch 128 (a fifth of the imagenet_hybrid 224 px iteration's "
                                  "640 images), the size DRAM-traffic captures are taken at"),
}
DEFAULT_CONFIG = "imagenet_hybrid"
F_SMALL = 19.0 / 21.0  # d_S/d_L for one large and one small worker at k = 1.05 (Eqs. 4-6)
LR, MOMENTUM = 0.2, 0.9


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", 0)), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def _conv_source_hash():
    h = hashlib.sha256()
    for name in ("conv.cu", "dbl_internal.cuh", "dbl_act.cuh"):
        with open(os.path.join(ROOT, "paper_2509_26092_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def _traffic_record(config):
    """DRAM bytes (read + write) of all conv-kernel launches of one iteration at the largest
    stage of `config`, from a committed ncu summary taken on the current kernel source: the
    capture ran a smaller configuration and is scaled by the images processed (conv traffic
    is per image: activations and their gradients, the weights being a small share)."""
    path = os.path.join(ROOT, "profiles", "conv_traffic_imagenet_hybrid_224.json")
    try:
        with open(path) as f:
            rec = json.load(f)
        if rec.get("source_hash") != _conv_source_hash() or rec.get("applies_to") != config:
            return None
        return int(rec["dram_bytes_per_iteration"] * rec.get("scale", 1.0))
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(mx), "reasons": sorted(reasons), "samples": len(sm)}


def max_over_ranks(x, device="cpu"):
    """The largest of each rank's x (the job's time is its slowest rank's); x itself on one rank."""
    import torch
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(images_per_step, world, steps, ms):
    """images/s of the whole job: every rank's images over the slowest rank's time."""
    return images_per_step * world * steps / (ms / 1000.0)


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


# ------------------------------------------------------------------------------------------ oracle timing
def _oracle_setup(cfg):
    import numpy as np

    import oracle as orc
    from oracle import resnet18 as OR
    from paper_2509_26092_gb300 import synth

    table = OR.layer_table(cfg["variant"], cfg["classes"])
    params = {k: v.astype(np.float64) for k, v in synth.params(table, seed=0).items()}
    vel = {k: np.zeros_like(v) for k, v in params.items()}
    img = synth.images(3, cfg["native"], cfg["native"], 3, seed=0).astype(np.float64)
    lab = synth.labels(3, cfg["classes"], seed=0)
    orc.lib()
    return dict(params=params, vel=vel, img=img, lab=lab)


def _oracle_iteration(cfg, st, res):
    """One dual-batch iteration of the fp64 oracle at resolution res: large batch 2, small batch 1."""
    import numpy as np

    from oracle import resnet18 as OR
    d = float(np.float32(cfg["dropout"][list(cfg["stages"]).index(res)]))
    st["step"] = st.get("step", -1) + 1
    t0 = time.perf_counter()
    st["params"], st["vel"], *_ = OR.dual_batch_iteration(st["params"], st["vel"], st["img"][:2], st["lab"][:2],
                                                          st["img"][2:], st["lab"][2:], res, cfg["variant"], LR,
                                                          MOMENTUM, 1.0, F_SMALL, order=0,
                                                          dropout_large=(d, 2 * res + 1, st["step"]),
                                                          dropout_small=(d, 2 * res + 2, st["step"]))
    return 3, time.perf_counter() - t0


def time_oracle(cfg):
    """The fp64 CPU oracle on a bounded sample of the workload, timed on this
    host's cores: one dual-batch iteration (large batch 2, small batch 1) at
    each sub-stage resolution."""
    st = _oracle_setup(cfg)
    images, secs = 0, 0.0
    for res in cfg["stages"]:
        n, dt = _oracle_iteration(cfg, st, res)
        images += n
        secs += dt
    sample = (f"one dual-batch iteration (large batch 2, small batch 1) at each of "
              f"{', '.join(str(r) for r in cfg['stages'])} px, {cfg['variant']} ResNet-18, fp64")
    return images / secs, secs, images, sample


def run_reference(args, cfg):
    """The reference arm: the fp64 CPU oracle, as it stands, on this host's cores.
    Each step is one dual-batch iteration (large batch 2, small batch 1) at the
    next sub-stage resolution of the cycle."""
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    st = _oracle_setup(cfg)
    stages = cfg["stages"]
    images, secs = 0, 0.0
    for i in range(args.warmup + args.steps):
        n, dt = _oracle_iteration(cfg, st, stages[i % len(stages)])
        if i >= args.warmup:
            images += n
            secs += dt
    value = images / secs
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    sample = (f"{args.steps} dual-batch iterations (large batch 2, small batch 1) cycling through "
              f"{', '.join(str(r) for r in stages)} px, {cfg['variant']} ResNet-18, fp64 CPU oracle")
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "images/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1000.0 * secs / args.steps, 1),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.config, "description": cfg["desc"], "reference": "fp64 CPU oracle"},
            "cpu_baseline": {"value": round(value, 4), "unit": "images/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(value, 4), "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------------------------------ GPU arm
def build_pipeline(cfg, device, precision="bf16", pdl="auto"):
    import torch

    from paper_2509_26092_gb300 import dbl as D
    from paper_2509_26092_gb300 import resnet18 as R
    from paper_2509_26092_gb300 import synth

    spec = R.ResNet18Spec(cfg["variant"], cfg["classes"])
    server = R.ServerState(spec, synth.params(spec.table(), seed=0), synth.momentum_state(spec.table(), 0.0, seed=0),
                           precision=precision)
    bl_max = max(cfg["large"])
    bs_max = max([b for b in cfg["small"] if b] or [0])
    nat = cfg["native"]
    # decoded 8-bit pixels, as an input pipeline hands them over (standardized on the GPU)
    host_l = torch.from_numpy(synth.images_u8(bl_max, nat, nat, 3, seed=1, name="large")).pin_memory()
    host_s = torch.from_numpy(synth.images_u8(bs_max, nat, nat, 3, seed=1, name="small")).pin_memory() if bs_max else None
    lab_l = torch.from_numpy(synth.labels(bl_max, cfg["classes"], seed=1, name="large")).pin_memory()
    lab_s = torch.from_numpy(synth.labels(bs_max, cfg["classes"], seed=1, name="small")).pin_memory() if bs_max else None
    stages = []
    for res, bl, bs, drop in zip(cfg["stages"], cfg["large"], cfg["small"], cfg["dropout"]):
        large = R.Worker(spec, bl, res, device, dropout=drop, dropout_seed=2 * res + 1, precision=precision)
        small = (R.Worker(spec, bs, res, device, dropout=drop, dropout_seed=2 * res + 2, precision=precision)
                 if bs else None)
        if pdl != "auto":  # programmatic dependent launch per worker: on, off, or the large worker only
            large.pdl = pdl in ("on", "large")
            if small is not None:
                small.pdl = pdl == "on"
        it = R.DualBatchIteration(server, large, small, nat, lr=LR, momentum=MOMENTUM, f_large=1.0, f_small=F_SMALL)
        it.set_inputs(host_l[:bl].to(device), lab_l[:bl].to(device),
                      host_s[:bs].to(device) if bs else None, lab_s[:bs].to(device) if bs else None)
        n0 = D.dbl_kernel_launches()
        it.capture()
        launches = D.dbl_kernel_launches() - n0
        # capture() enqueues one eager warm-up iteration and one captured iteration
        stages.append(dict(res=res, it=it, large=large, small=small, launches=launches // 2,
                           images=bl + (bs or 0)))
    return dict(spec=server.spec, server=server, stages=stages, host_l=host_l, host_s=host_s, lab_l=lab_l,
                lab_s=lab_s)


def conv_roofline(stage, reps=4, replays=2, table=None, cold_reps=5):
    """Time each convolution pass of the stage's workers alone with CUDA events, two ways.
    Cold: L2 flushed before each launch (a 512 MB buffer, larger than the 129 MB L2, written on
    the stream first), the pass replayed from a one-call CUDA graph, the median of `cold_reps`
    launches, as in the training step where every pass's operands come from DRAM (its working
    set is many GB).  Warm: `reps` calls of the pass captured in one CUDA graph
    and replayed `replays` times, so repeats 2.. find operands of the smaller layers in L2.
    Return (algorithmic conv FLOPs of one iteration, cold seconds per iteration, warm seconds
    per iteration, algorithmic bytes).  If table is a list, append (worker batch, layer, pass,
    FLOPs, cold seconds, warm seconds) per pass."""
    import torch

    from paper_2509_26092_gb300 import dbl as D
    flops, secs, warm_secs = 0.0, 0.0, 0.0
    # 512 MB: the write takes ~80 us, longer than the host needs to enqueue a pass behind it
    flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
    nbytes = lambda *ts: sum(t.numel() * t.element_size() for t in ts)
    algo_bytes = 0  # unique operand bytes of every pass (inputs + weights + outputs)
    for wk in (stage["large"], stage["small"]):
        if wk is None:
            continue
        stem = wk.spec.stem.name
        bufs = _conv_buffers(wk)
        shapes = dict(wk.conv_shapes())
        for name, shp in wk.conv_shapes():
            x, y, dy, dx, w16, g = bufs[name]
            st_sum = torch.empty(shp.k, device=x.device)
            st_sq = torch.empty(shp.k, device=x.device)
            f1 = float(wk.layer_flops(name, shp))
            if name == stem:
                passes = [("fwd", f1, lambda s: D.dbl_conv_fwd(shp, x, w16, y, st_sum, st_sq, wk.ws, wk.ws.numel(), s))]
            else:
                # as in the training step: the BatchNorm statistics are left as per-CTA partials,
                # which the BatchNorm finalize reduces
                parts = wk.ws
                passes = [("fwd", f1, lambda s: D.dbl_conv_fwd_parts(shp, x, w16, y, parts, parts.numel(), s))]
            algo_bytes += nbytes(x, w16, y)
            proj = name.replace(".conv1", ".down") if name.endswith(".conv1") else None
            if proj in bufs:
                # a downsampling block's input gradient: conv1's and the projection's in one pass
                _, _, dy2, _, w2, _ = bufs[proj]
                fd = f1 + float(wk.layer_flops(proj, shapes[proj]))
                passes.append(("dgrad+proj", fd, lambda s: D.dbl_conv_dgrad_proj(shp, dy, w16, shapes[proj].k, dy2, w2,
                                                                                 dx, None, 0, s)))
                algo_bytes += nbytes(dy, w16, dy2, w2, dx)
            elif name != stem and dx is not None:
                passes.append(("dgrad", f1, lambda s: D.dbl_conv_dgrad(shp, dy, w16, dx, None, 0, s)))
                algo_bytes += nbytes(dy, w16, dx)
            passes.append(("wgrad", f1, lambda s: D.dbl_conv_wgrad(shp, x, dy, g, False, wk.ws, wk.ws.numel(), s)))
            algo_bytes += nbytes(x, dy, g)
            for pname, fp, fn in passes:
                fn(torch.cuda.current_stream())
                torch.cuda.synchronize()
                graph = torch.cuda.CUDAGraph()
                with torch.cuda.graph(graph):
                    for _ in range(reps):
                        fn(torch.cuda.current_stream())
                graph.replay()
                s = torch.cuda.current_stream()
                ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
                ev[0].record(s)
                for _ in range(replays):
                    graph.replay()
                ev[1].record(s)
                torch.cuda.synchronize()
                del graph
                tw = ev[0].elapsed_time(ev[1]) / 1000.0 / (reps * replays)
                # cold: one call of the pass as a CUDA graph (its replay is enqueued in microseconds,
                # so the host never holds up the GPU between the events), after the flush
                one = torch.cuda.CUDAGraph()
                with torch.cuda.graph(one):
                    fn(torch.cuda.current_stream())
                cold = []
                for _ in range(cold_reps):
                    flush.zero_()
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record(s)
                    one.replay()
                    e1.record(s)
                    torch.cuda.synchronize()
                    cold.append(e0.elapsed_time(e1) / 1000.0)
                del one
                tc = sorted(cold)[len(cold) // 2]
                secs += tc
                warm_secs += tw
                flops += fp
                if table is not None:
                    table.append((wk.batch, name, pname, fp, tc, tw))
    return flops, secs, warm_secs, algo_bytes


def bandwidth_kernels(pipe, hbm, reps=10):
    """The HBM-bound kernels timed alone with L2 flushed before each launch (a 256 MB buffer,
    larger than the 129 MB L2, written on the same stream): the parameter-server merge of both
    pushes (26 B per parameter: read w, u, g_L, g_S, write w, u and the bf16 copy; 22 B with one
    push) and, per stage, the large worker's resize of its uint8 source images into the stem's
    unrolled bf16 input (bytes: the source read once plus the unrolled tensor written once).
    Median of `reps` launches, CUDA events on the launching stream."""
    import torch

    from paper_2509_26092_gb300 import dbl as D
    s = torch.cuda.current_stream()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=pipe["server"].w.device)

    def timed(fn):
        out = []
        for _ in range(reps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(s)
            fn()
            e1.record(s)
            torch.cuda.synchronize()
            out.append(e0.elapsed_time(e1) * 1e-3)
        out.sort()
        return out[len(out) // 2]

    srv, top = pipe["server"], pipe["stages"][-1]
    gl, gs = top["large"].grad, top["small"].grad if top["small"] else None
    n = srv.spec.n_flat
    nbytes = n * (26 if gs is not None else 22)
    t = timed(lambda: D.dbl_ps_dual_batch_merge(srv.w, srv.u, srv.w16, gl, gs, n, LR, MOMENTUM, 1.0, F_SMALL, 0, s))
    merge = {"us": round(t * 1e6, 2), "bytes": nbytes, "gbs": round(nbytes / t / 1e9, 1),
             "frac": round(nbytes / t / 1e9 / hbm, 4), "params": n, "pushes": 2 if gs is not None else 1,
             "l2": "flushed before each launch"}
    resize = {}
    for st in pipe["stages"]:
        wk, it = st["large"], st["it"]
        nb = it.images_l.numel() * it.images_l.element_size() + wk.x0.numel() * wk.x0.element_size()
        t = timed(lambda: wk.stem_prepare(it.images_l, it.native_res, s))
        resize[str(st["res"])] = {"us": round(t * 1e6, 2), "bytes": nb, "gbs": round(nb / t / 1e9, 1),
                                  "frac": round(nb / t / 1e9 / hbm, 4), "batch": wk.batch}
    return {"merge": merge, "resize": resize}


def time_oracle_single_thread(config):
    """The oracle on one host thread (OMP_NUM_THREADS=1, a child process): one dual-batch
    iteration (large batch 2, small batch 1) at the smallest sub-stage resolution."""
    code = ("import json, sys; sys.path.insert(0, sys.argv[1]); import bench\n"
            "cfg = bench.CONFIGS[sys.argv[2]]; st = bench._oracle_setup(cfg)\n"
            "n, dt = bench._oracle_iteration(cfg, st, min(cfg['stages']))\n"
            "print(json.dumps({'images': n, 'seconds': dt}))\n")
    env = dict(os.environ, OMP_NUM_THREADS="1")
    try:
        r = subprocess.run([sys.executable, "-c", code, ROOT, config], env=env, capture_output=True, text=True,
                           timeout=600)
        rec = json.loads(r.stdout.strip().splitlines()[-1])
    except Exception as e:  # the figure is a reported baseline; its absence must not fail the bench
        return {"error": str(e)[:200]}
    cfg = CONFIGS[config]
    return {"value": round(rec["images"] / rec["seconds"], 4), "unit": "images/s", "cores": 1,
            "seconds": round(rec["seconds"], 2),
            "sample": f"one dual-batch iteration (large batch 2, small batch 1) at {min(cfg['stages'])} px, fp64"}


def _conv_buffers(wk):
    """Per conv layer: (input, output, output-gradient, input-gradient, bf16 weights, fp32 gradient slice)."""
    spec = wk.spec
    srv_w16 = wk._bench_w16
    out = {}
    st = spec.stem
    out[st.name] = (wk.x0, wk.stem_y, wk.stem_dy, None, spec.view(srv_w16, "conv1.w"), spec.view(wk.grad, "conv1.w"))
    cur = wk.pool_out if spec.variant == "imagenet" else wk.stem_a
    for d in wk.blocks:
        b = d["spec"]
        out[b.pre + ".conv1"] = (cur, d["h1"], d["dh1"], d["din"], spec.view(srv_w16, b.pre + ".conv1.w"),
                                 spec.view(wk.grad, b.pre + ".conv1.w"))
        out[b.pre + ".conv2"] = (d["o1"], d["h2"], d["dh2"], d["do1"], spec.view(srv_w16, b.pre + ".conv2.w"),
                                 spec.view(wk.grad, b.pre + ".conv2.w"))
        if b.proj:
            out[b.pre + ".down"] = (cur, d["hs"], d["dhs"], None, spec.view(srv_w16, b.pre + ".down.w"),
                                    spec.view(wk.grad, b.pre + ".down.w"))
        cur = d["out"]
    return out


def run_profile_iteration(args, cfg):
    """One eager dual-batch iteration per stage and nothing else: the command ncu
    captures for the launch list and the per-kernel captures."""
    import torch

    from paper_2509_26092_gb300 import build_lib
    build_lib.build()
    from paper_2509_26092_gb300 import dbl as D
    from paper_2509_26092_gb300 import resnet18 as R
    from paper_2509_26092_gb300 import synth

    torch.cuda.set_device(0)
    spec = R.ResNet18Spec(cfg["variant"], cfg["classes"])
    server = R.ServerState(spec, synth.params(spec.table(), seed=0))
    nat = cfg["native"]
    n0 = D.dbl_kernel_launches()
    for res, bl, bs, drop in zip(cfg["stages"], cfg["large"], cfg["small"], cfg["dropout"]):
        if args.profile_res and res != args.profile_res:
            continue
        large = R.Worker(spec, bl, res, dropout=drop, dropout_seed=2 * res + 1)
        small = R.Worker(spec, bs, res, dropout=drop, dropout_seed=2 * res + 2) if bs else None
        it = R.DualBatchIteration(server, large, small, nat, lr=LR, momentum=MOMENTUM, f_small=F_SMALL)
        it.set_inputs(torch.from_numpy(synth.images_u8(bl, nat, nat, 3, seed=1)).cuda(),
                      torch.from_numpy(synth.labels(bl, cfg["classes"], seed=1)).cuda(),
                      torch.from_numpy(synth.images_u8(bs, nat, nat, 3, seed=2)).cuda() if bs else None,
                      torch.from_numpy(synth.labels(bs, cfg["classes"], seed=2)).cuda() if bs else None)
        it.run()
        torch.cuda.synchronize()
        del it, large, small
    assert D.dbl_device_status() == D.DBL_OK
    print(json.dumps({"profile_iteration": args.config, "launches": D.dbl_kernel_launches() - n0}), flush=True)
    return 0


def run_profile_conv(args):
    """Three launches of one convolution pass of one ResNet-18 layer (224 px input,
    batch --profile-batch), with only that layer's operands on the device: the
    command ncu captures for the per-kernel profiles (-k regex:conv_igemm -s 2 -c 1
    takes the third, warm launch)."""
    import torch

    from paper_2509_26092_gb300 import build_lib
    build_lib.build()
    from paper_2509_26092_gb300 import dbl as D
    from paper_2509_26092_gb300 import resnet18 as R

    torch.cuda.set_device(0)
    with D.precision(args.precision):
        return _profile_conv(args, D, R)


def _profile_conv(args, D, R):
    import torch
    act = {"bf16": torch.bfloat16, "f16": torch.float16}[args.precision]
    layer, pname = args.profile_conv.split(":")
    spec = R.ResNet18Spec("imagenet", 1000)
    n = args.profile_batch
    h = R.conv_out(R.conv_out(224, spec.stem.r, spec.stem.stride, spec.stem.pad), 3, 2, 1)  # after stem and max-pool
    shapes = {}
    for b in spec.blocks:
        ho = R.conv_out(h, 3, b.stride, 1)
        shapes[b.pre + ".conv1"] = D.conv_shape(n, h, h, b.cin, b.cout, 3, b.stride, 1)
        shapes[b.pre + ".conv2"] = D.conv_shape(n, ho, ho, b.cout, b.cout, 3, 1, 1)
        if b.proj:
            shapes[b.pre + ".down"] = D.conv_shape(n, h, h, b.cin, b.cout, 1, b.stride, 0)
        h = ho
    st_, lay = spec.stem, spec.stem_layout  # the stem as a convolution of its unrolled 224 px input
    hs = R.conv_out(224, st_.r, st_.stride, st_.pad)
    shapes[st_.name] = D.conv_shape(n, lay.rows(224, hs), hs, 64, st_.cout, lay.taps, lay.conv_stride, lay.conv_pad,
                                    s=1, stride_w=1, pad_w=0)
    if layer not in shapes:
        raise SystemExit(f"--profile-conv: unknown layer {layer!r} (one of {', '.join(shapes)})")
    s = shapes[layer]
    P = R.conv_out(s.h, s.r, s.stride, s.pad)
    Q = R.conv_out(s.w, s.s, s.stride_w or s.stride, s.pad_w if s.stride_w else s.pad)
    g = torch.Generator(device="cuda").manual_seed(0)
    x = torch.randn(s.n, s.h, s.w, s.c, device="cuda", generator=g).to(act)
    w = (0.05 * torch.randn(s.k, s.r, s.s, s.c, device="cuda", generator=g)).to(act)
    dy = torch.randn(s.n, P, Q, s.k, device="cuda", generator=g).to(act)
    ps = {"fwd": D.DBL_PASS_FWD, "dgrad": D.DBL_PASS_DGRAD, "wgrad": D.DBL_PASS_WGRAD}[pname]
    ws = torch.empty(max(int(D.dbl_conv_workspace_bytes(s, ps)), 16), dtype=torch.uint8, device="cuda")
    st = torch.cuda.current_stream()
    if pname == "fwd":
        y = torch.empty(s.n, P, Q, s.k, dtype=act, device="cuda")
        ssum, ssq = torch.empty(s.k, device="cuda"), torch.empty(s.k, device="cuda")
        fn = lambda: D.dbl_conv_fwd(s, x, w, y, ssum, ssq, ws, ws.numel(), st)
    elif pname == "dgrad":
        dx = torch.empty_like(x)
        fn = lambda: D.dbl_conv_dgrad(s, dy, w, dx, None, 0, st)
    else:
        dw = torch.empty(s.k * s.r * s.s * s.c, device="cuda")
        fn = lambda: D.dbl_conv_wgrad(s, x, dy, dw, False, ws, ws.numel(), st)
    for _ in range(3):
        fn()
    torch.cuda.synchronize()
    assert D.dbl_device_status() == D.DBL_OK
    print(json.dumps({"profile_conv": args.profile_conv, "batch": n, "precision": args.precision}), flush=True)
    return 0


def run_ours(args, cfg):
    import numpy as np
    import torch
    ws, rank, local = _dist()
    if args.pdl == "auto" and all(b is None for b in cfg["small"]):
        # one worker, one stream: let each convolution's set-up overlap the kernel before it
        # (programmatic dependent launch; with two worker streams it measured slower)
        os.environ.setdefault("DBL_CONV_PDL", "1")
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    device = f"cuda:{local}"
    from paper_2509_26092_gb300 import build_lib
    build_lib.build()
    from paper_2509_26092_gb300 import dbl as D

    pipe = build_pipeline(cfg, device, args.precision, args.pdl)
    stages = pipe["stages"]
    images_per_step = sum(s["images"] for s in stages)

    def step():
        for st in stages:
            st["it"].run()

    def barrier():
        torch.cuda.synchronize()
        if ws > 1:
            torch.distributed.barrier()

    for _ in range(args.warmup):
        step()
    barrier()
    assert D.dbl_device_status() == D.DBL_OK, "a device-side wait timed out during warm-up"
    clocks = ClockSampler(local)
    clocks.start()
    stream = torch.cuda.current_stream()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    t0.record(stream)
    for _ in range(args.steps):
        step()
    t1.record(stream)
    barrier()
    clk = clocks.stop()
    ms = max_over_ranks(t0.elapsed_time(t1), device)
    ms_per_step = ms / args.steps
    value = whole_job_rate(images_per_step, ws, args.steps, ms)
    gpu_launches = sum(s["launches"] for s in stages) * args.steps

    # per-resolution throughput (each stage's graph replayed alone)
    per_res = {}
    for st in stages:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = max(2, args.steps)
        e0.record(stream)
        for _ in range(reps):
            st["it"].run()
        e1.record(stream)
        torch.cuda.synchronize()
        per_res[str(st["res"])] = round(st["images"] * reps / (e0.elapsed_time(e1) / 1000.0), 1)

    # end to end through the public API: pinned host images -> device (on a copy stream, each
    # stage's copy overlapping the compute of the stages before it), iteration, losses back to
    # pinned host memory; step k's losses are read on the host after step k+1 is enqueued
    h2d = d2h = 0
    copy_stream = torch.cuda.Stream()
    loss_host = [torch.zeros(2 * len(stages), dtype=torch.float32).pin_memory() for _ in range(2)]
    loss_seen = []
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    e0.record(stream)
    prev = None
    for k in range(args.steps):
        for st in stages:
            it, bl, bs = st["it"], st["large"].batch, st["small"].batch if st["small"] else 0
            it.set_inputs(pipe["host_l"][:bl], pipe["lab_l"][:bl], pipe["host_s"][:bs] if bs else None,
                          pipe["lab_s"][:bs] if bs else None, non_blocking=True, stream=copy_stream)
        buf = loss_host[k % 2]
        n_out = 0
        for st in stages:
            st["it"].run()
            n_out += st["it"].losses_to_host(buf[n_out:])
        done = torch.cuda.Event()
        done.record(stream)
        if prev is not None:
            prev[0].synchronize()
            loss_seen.append(prev[1][:prev[2]].tolist())
        prev = (done, buf, n_out)
        if h2d == 0:
            for st in stages:
                bl, bs = st["large"].batch, st["small"].batch if st["small"] else 0
                h2d += (bl + bs) * cfg["native"] ** 2 * 3 * pipe["host_l"].element_size() + (bl + bs) * 4
                d2h += 4 * (2 if bs else 1)
    prev[0].synchronize()
    loss_seen.append(prev[1][:prev[2]].tolist())
    e1.record(stream)
    barrier()
    assert len(loss_seen) == args.steps and all(np.isfinite(v).all() for v in map(np.asarray, loss_seen))
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), device)
    e2e_value = whole_job_rate(images_per_step, ws, args.steps, e2e_ms)
    assert D.dbl_device_status() == D.DBL_OK, "a device-side wait timed out during the timed region"

    # roofline of the dominant kernel: the implicit-GEMM convolution, full-resolution stage, timed alone
    hbm, bf16, bf16_sus, src = _peaks()
    top = max(stages, key=lambda s: s["res"])
    for wk in (top["large"], top["small"]):
        if wk is not None:
            wk._bench_w16 = pipe["server"].w16
    table = [] if args.conv_table else None
    with D.precision(args.precision):
        flops, secs, warm_secs, algo_bytes = conv_roofline(top, table=table)
    if table is not None:
        for b, name, pname, f1, tc, tw in table:
            print(f"conv {b:4d} {name:16s} {pname:5s} cold {tc * 1e6:9.1f} us {f1 / tc / 1e12:7.1f} TFLOP/s   "
                  f"warm {tw * 1e6:9.1f} us {f1 / tw / 1e12:7.1f} TFLOP/s", file=sys.stderr)
    achieved = flops / secs / 1e12
    warm = flops / warm_secs / 1e12
    roofline = {"bound": "tensor", "achieved": round(achieved, 1), "peak": bf16, "unit": "TFLOP/s",
                "frac": round(achieved / bf16, 4), "traffic": _traffic_record(args.config),
                "algorithmic_bytes": int(algo_bytes),
                "frac_sustained_peak": round(achieved / bf16_sus, 4) if bf16_sus else None,
                "warm_l2": {"achieved": round(warm, 1), "frac": round(warm / bf16, 4)},
                "scope": f"one dual-batch iteration at {top['res']} px: every conv pass of both workers "
                         "(achieved = algorithmic FLOPs / summed CUDA-event time of the passes, each pass timed "
                         "alone with L2 flushed before it, median of 5; warm_l2: the same passes as back-to-back "
                         "CUDA-graph replays; traffic = ncu DRAM bytes of the same launches, null if the kernel "
                         "changed since the capture)",
                "kernel": "conv_igemm_kernel, conv_win_kernel, conv_wgwin_kernel with their channel-sum and "
                          f"split-K reduce kernels (fwd/dgrad/wgrad, every layer of both workers at {top['res']} px)",
                "peak_source": src}
    with D.precision(args.precision):
        bw = bandwidth_kernels(pipe, hbm)
    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        v, dt, images, sample = time_oracle(cfg)
        cpu = {"value": round(v, 4), "unit": "images/s", "cores": int(os.environ.get("OMP_NUM_THREADS",
                                                                                      os.cpu_count() or 1)),
               "kind": "oracle", "sample": sample, "seconds": round(dt, 2),
               "single_thread": time_oracle_single_thread(args.config)}
    if rank == 0:
        line = {"metric": METRIC, "value": round(value, 1), "unit": "images/s", "n_gpus": ws, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": round(ms_per_step, 3), "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": args.precision, "data": "synthetic",
                "config": {"workload": args.config, "description": cfg["desc"], "precision": args.precision,
                           "loss_scaling": ("dynamic: initial 2^15, halved on overflow, doubled after 2000 good "
                                            "steps" if args.precision == "f16" else None),
                           "stages_px": list(cfg["stages"]), "large_batch": list(cfg["large"]),
                           "small_batch": list(cfg["small"]), "dropout": list(cfg["dropout"]),
                           "images_per_step": images_per_step,
                           "params": pipe["spec"].n_params(), "f_small": F_SMALL, "lr": LR, "momentum": MOMENTUM,
                           "conv_pdl": (args.pdl if args.pdl != "auto" else
                                        "on" if os.environ.get("DBL_CONV_PDL") == "1" else "off"),
                           "l2": "working set (activations, several GB) larger than L2; no explicit flush",
                           "input": f"uint8 images {cfg['native']}x{cfg['native']}x3 from pinned host memory, "
                                    "standardized per channel on the GPU",
                           "parallelism": f"{ws} independent replica(s), 2 worker streams each"},
                "per_resolution": per_res, "roofline": roofline, "merge": bw["merge"], "resize": bw["resize"],
                "cpu_baseline": cpu,
                "e2e": {"value": round(e2e_value, 1), "unit": "images/s", "h2d_bytes_per_step": h2d,
                        "d2h_bytes_per_step": d2h},
                "clocks": clk, "gpu_launches": gpu_launches,
                "conv_tflops_step": round(sum(s["large"].conv_flops() + (s["small"].conv_flops() if s["small"] else 0)
                                              for s in stages) / (ms_per_step / 1000.0) / 1e12, 1)}
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default=DEFAULT_CONFIG, choices=sorted(CONFIGS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--pdl", default="auto", choices=["auto", "off", "on", "large"],
                    help="programmatic dependent launch of the convolutions: auto (one-worker workloads only), "
                         "off, on, or the large worker only")
    ap.add_argument("--precision", default="bf16", choices=["bf16", "f16"],
                    help="16-bit storage format: bf16, or f16 with dynamic loss scaling (the paper's mixed precision)")
    ap.add_argument("--conv-table", action="store_true",
                    help="print each convolution pass's time and TFLOP/s (largest stage) to stderr")
    ap.add_argument("--profile-conv", default=None, metavar="LAYER:PASS",
                    help="run one conv pass of one layer three times (e.g. layer1.0.conv1:fwd) for ncu")
    ap.add_argument("--profile-batch", type=int, default=512)
    ap.add_argument("--profile-res", type=int, default=0,
                    help="with --profile-iteration: run only the stage at this resolution")
    ap.add_argument("--profile-iteration", action="store_true",
                    help="run one eager iteration per stage and exit (the command ncu profiles)")
    args = ap.parse_args()
    cfg = CONFIGS[args.config]
    if args.impl == "reference":
        return run_reference(args, cfg)
    if args.profile_conv:
        return run_profile_conv(args)
    if args.profile_iteration:
        return run_profile_iteration(args, cfg)
    return run_ours(args, cfg)


if __name__ == "__main__":
    sys.exit(main())
