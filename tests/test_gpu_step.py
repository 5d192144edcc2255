"""Whole-step GPU parity: the ResNet-18 training step and the two-stream
dual-batch iteration run through libdbl, against the fp64 oracle.

The loss is compared at the conv-path tolerance (max-norm relative 1e-2).
End-to-end parameter gradients are compared against the oracle with bf16
rounding at the same storage points, within the spread that bf16 storage
itself causes: the gradient of this step at initialisation is ill-conditioned
with respect to storage rounding (ReLU masks flip and BatchNorm backward
subtracts nearly equal terms), so the oracle's own bf16-storage gradients
differ from its fp64 gradients by about 30% (median over tensors).  With
spread = |oracle_bf16 - oracle_fp64| per tensor (max norm), the GPU's error
|gpu - oracle_bf16| must be at most max(2 * spread, 1e-2 * |oracle_bf16|) for
every tensor, and its median ratio to the spread over all tensors at most 1:
the GPU is no further from the oracle than the oracle's own rounding moves it.  Each layer on its own is held to 1e-2 at the same shapes in
test_gpu_step_layers.py.  The merge is compared on the GPU's own pushed
gradients (identical fp32 inputs) at 1e-6.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from conftest import max_norm_rel
from gpu_common import load_dbl
from oracle import resnet18 as OR
from paper_2509_26092_gb300 import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


@pytest.fixture(scope="module")
def R():
    load_dbl()
    from paper_2509_26092_gb300 import resnet18
    return resnet18


def _compare_grads(spec, grad_flat, ref_bf16, ref_f64, tag=""):
    """Every gradient within the bf16-storage spread of the oracle (see the module docstring)."""
    got = spec.unpack(grad_flat)
    rows = []
    for name, g in ref_bf16.items():
        scale = float(np.max(np.abs(g))) or 1.0
        err = float(np.max(np.abs(got[name] - g))) / scale
        spread = float(np.max(np.abs(ref_f64[name] - g))) / scale
        rows.append((name, err, spread, max(2.0 * spread, TOL)))
    ratio = [r[1] / max(r[2], 1e-12) for r in rows]
    print(f"\n{tag}: median gpu-vs-oracle {np.median([r[1] for r in rows]):.2e}, median bf16-vs-fp64 spread "
          f"{np.median([r[2] for r in rows]):.2e}, median ratio {np.median(ratio):.2f}, max ratio {max(ratio):.2f}")
    bad = [r for r in rows if r[1] > r[3]]
    assert not bad, f"{len(bad)} gradients outside the storage-rounding spread: {bad[:4]}"
    assert np.median(ratio) <= 1.0, f"median ratio {np.median(ratio):.2f} > 1"


@pytest.mark.parametrize("variant,classes,batch,res", [("cifar", 100, 8, 32), ("imagenet", 1000, 8, 96)])
def test_train_step_matches_oracle(R, variant, classes, batch, res):
    spec = R.ResNet18Spec(variant, classes)
    params = synth.params(spec.table(), seed=3, random_bn=True)
    img = synth.images(batch, res, res, 3, seed=3)
    lab = synth.labels(batch, classes, seed=3)
    server = R.ServerState(spec, params)
    wk = R.Worker(spec, batch, res)
    it = R.DualBatchIteration(server, wk, None, res)
    it.set_inputs(torch.from_numpy(img).cuda(), torch.from_numpy(lab).cuda())
    s = torch.cuda.current_stream()
    wk.enqueue_step(server, it.images_l, res, s)
    torch.cuda.synchronize()
    D = load_dbl()
    assert D.dbl_device_status() == D.DBL_OK
    p64 = {k: v.astype(np.float64) for k, v in params.items()}
    ref = OR.train_step(p64, img.astype(np.float64), lab, variant, bf16_storage=True)
    ref64 = OR.train_step(p64, img.astype(np.float64), lab, variant, bf16_storage=False)
    print(f"\n{variant}: loss {wk.loss.item():.6f} vs oracle {ref['loss']:.6f}")
    assert abs(wk.loss.item() - ref["loss"]) <= TOL * abs(ref["loss"])
    _compare_grads(spec, wk.grad, ref["grads"], ref64["grads"], variant)


@pytest.mark.parametrize("dropout", [0.0, 0.2])
def test_dual_batch_iteration_matches_oracle(R, dropout):
    # native 32x32 images, sub-stage resolution 24: large worker batch 6, small worker batch 2;
    # with dropout before the FC layer (Sec. 4.1), each worker drawing its own mask
    spec = R.ResNet18Spec("cifar", 100)
    params = synth.params(spec.table(), seed=5, random_bn=True)
    u0 = synth.momentum_state(spec.table(), 0.01, seed=5)
    img = synth.images(8, 32, 32, 3, seed=5)
    lab = synth.labels(8, 100, seed=5)
    server = R.ServerState(spec, params, u0)
    large = R.Worker(spec, 6, 24, dropout=dropout, dropout_seed=101)
    small = R.Worker(spec, 2, 24, dropout=dropout, dropout_seed=202)
    d = float(np.float32(dropout))  # the rate as the fp32 value the library receives
    drops = dict(dropout_large=(d, 101, 0), dropout_small=(d, 202, 0)) if dropout else {}
    fS = 19.0 / 21.0
    it = R.DualBatchIteration(server, large, small, 32, lr=0.2, momentum=0.9, f_large=1.0, f_small=fS, order=0)
    it.set_inputs(torch.from_numpy(img[2:]).cuda(), torch.from_numpy(lab[2:]).cuda(), torch.from_numpy(img[:2]).cuda(),
                  torch.from_numpy(lab[:2]).cuda())
    w_before = server.w.clone()
    u_before = server.u.clone()
    it.run()
    torch.cuda.synchronize()
    p64 = {k: v.astype(np.float64) for k, v in params.items()}
    u64 = {k: v.astype(np.float64) for k, v in u0.items()}
    nw, nu, lL, lS, gL, gS = OR.dual_batch_iteration(p64, u64, img[2:], lab[2:], img[:2], lab[:2], 24, "cifar", 0.2,
                                                     0.9, 1.0, fS, order=0, bf16_storage=True, **drops)
    nw64, _, _, _, gL64, gS64 = OR.dual_batch_iteration(p64, u64, img[2:], lab[2:], img[:2], lab[:2], 24, "cifar",
                                                        0.2, 0.9, 1.0, fS, order=0, bf16_storage=False, **drops)
    if dropout:
        # each worker's step counter advanced once; the FC gradient of a feature no sample kept is zero
        assert int(large.dropout_step.item()) == 1 and int(small.dropout_step.item()) == 1
        keep = orc.dropout_mask(2, 512, d, 202, 0)
        dead = np.where(keep.sum(axis=0) == 0)[0]
        assert dead.size > 0 and np.all(spec.unpack(small.grad)["fc.w"][:, dead] == 0.0)
    assert abs(large.loss.item() - lL) <= TOL * abs(lL)
    assert abs(small.loss.item() - lS) <= TOL * abs(lS)
    _compare_grads(spec, large.grad, gL, gL64, "large worker")
    _compare_grads(spec, small.grad, gS, gS64, "small worker")
    # the server's merge, given the pushes the GPU workers produced
    rw, ru = orc.ps_merge(w_before.double().cpu().numpy(), u_before.double().cpu().numpy(),
                          large.grad.double().cpu().numpy(), small.grad.double().cpu().numpy(), 0.2, 0.9, 1.0, fS, 0)
    assert max_norm_rel(server.w.double().cpu().numpy(), rw) <= 1e-6
    assert max_norm_rel(server.u.double().cpu().numpy(), ru) <= 1e-6
    assert torch.equal(server.w16, server.w.to(torch.bfloat16))
    # and the update against the oracle's own end-to-end iteration, within the storage-rounding spread
    got_w = spec.unpack(server.w)
    for name in nw:
        d_ref, d64 = nw[name] - p64[name], nw64[name] - p64[name]
        scale = float(np.max(np.abs(d_ref))) or 1.0
        spread = float(np.max(np.abs(d64 - d_ref))) / scale
        assert float(np.max(np.abs(got_w[name] - p64[name] - d_ref))) / scale <= max(2 * spread, TOL), name


def test_graph_replay_equals_eager(R):
    spec = R.ResNet18Spec("cifar", 100)
    params = synth.params(spec.table(), seed=7)
    img = torch.from_numpy(synth.images(12, 32, 32, 3, seed=7)).cuda()
    lab = torch.from_numpy(synth.labels(12, 100, seed=7)).cuda()
    outs = []
    for use_graph in (False, True):
        server = R.ServerState(spec, params)
        it = R.DualBatchIteration(server, R.Worker(spec, 8, 16), R.Worker(spec, 4, 16), 32)
        it.set_inputs(img[4:], lab[4:], img[:4], lab[:4])
        if use_graph:
            w0, u0 = server.w.clone(), server.u.clone()
            it.capture()  # runs one eager warm-up iteration first
            server.w.copy_(w0)
            server.u.copy_(u0)
            server.w16.copy_(w0.to(torch.bfloat16))
        for _ in range(2):
            it.run()
        torch.cuda.synchronize()
        outs.append(server.w.clone())
    # deterministic kernels: replay and eager launches give identical bits
    assert torch.equal(outs[0], outs[1])


def test_inputs_on_a_copy_stream_give_the_same_iteration(R):
    """Host inputs copied on a separate stream (overlapping other iterations' compute)
    reach the same model as copies on the compute stream, bit for bit."""
    spec = R.ResNet18Spec("cifar", 100)
    params = synth.params(spec.table(), seed=9)
    img = torch.from_numpy(synth.images(12, 32, 32, 3, seed=9)).pin_memory()
    lab = torch.from_numpy(synth.labels(12, 100, seed=9)).pin_memory()
    outs = []
    for use_copy_stream in (False, True):
        server = R.ServerState(spec, params)
        its = [R.DualBatchIteration(server, R.Worker(spec, 8, res), R.Worker(spec, 4, res), 32) for res in (24, 32)]
        copy = torch.cuda.Stream() if use_copy_stream else None
        losses = torch.zeros(8, dtype=torch.float32).pin_memory()
        for step in range(2):
            for it in its:  # all copies first: with a copy stream they wait only for their buffer's last reader
                it.set_inputs(img[4:], lab[4:], img[:4], lab[:4], non_blocking=True, stream=copy)
            n = 0
            for it in its:
                it.run()
                n += it.losses_to_host(losses[n:])
        torch.cuda.synchronize()
        outs.append((server.w.clone(), losses.clone()))
    assert torch.equal(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1], outs[1][1]) and bool(torch.all(outs[0][1][:4] > 0))  # 2 iterations x 2 workers


def test_8bit_images_give_the_same_iteration_as_standardized_fp32(R):
    """The iteration fed 8-bit pixels equals the iteration fed the same pixels standardized
    on the host (p*PIXEL_SCALE + PIXEL_BIAS in fp32), bit for bit."""
    spec = R.ResNet18Spec("imagenet", 10)
    params = synth.params(spec.table(), seed=4)
    u8 = synth.images_u8(6, 96, 96, 3, seed=4)
    x32 = u8.astype(np.float32) * np.asarray(R.PIXEL_SCALE, np.float32) + np.asarray(R.PIXEL_BIAS, np.float32)
    lab = torch.from_numpy(synth.labels(6, 10, seed=4)).cuda()
    outs = []
    for img in (torch.from_numpy(u8).cuda(), torch.from_numpy(x32).cuda()):
        server = R.ServerState(spec, params)
        it = R.DualBatchIteration(server, R.Worker(spec, 4, 64), R.Worker(spec, 2, 64), 96)
        it.set_inputs(img[2:], lab[2:], img[:2], lab[:2])
        it.run()
        torch.cuda.synchronize()
        outs.append(server.w.clone())
    assert torch.equal(outs[0], outs[1])


def test_a_late_push_is_left_out_of_the_merge(R):
    """A small-batch worker held back on its stream (a straggler) misses the server's deadline:
    the iteration reports DBL_ERR_TIMEOUT with the small worker as failed and merges the large
    worker's push alone, as ASP does (Sec. 2.4).  Released afterwards, the held stream finishes,
    and the next iteration merges both pushes again."""
    D = load_dbl()
    spec = R.ResNet18Spec("cifar", 100)
    params = synth.params(spec.table(), seed=6)
    u0 = synth.momentum_state(spec.table(), 0.01, seed=6)
    img = torch.from_numpy(synth.images(8, 32, 32, 3, seed=6)).cuda()
    lab = torch.from_numpy(synth.labels(8, 100, seed=6)).cuda()
    server = R.ServerState(spec, params, u0)
    large, small = R.Worker(spec, 6, 24), R.Worker(spec, 2, 24)
    fS = 19.0 / 21.0
    it = R.DualBatchIteration(server, large, small, 32, lr=0.2, momentum=0.9, f_large=1.0, f_small=fS, order=0)
    it.set_inputs(img[2:], lab[2:], img[:2], lab[:2])
    it.run()  # warm-up: the first launches load the library's kernels, which waits for every stream
    torch.cuda.synchronize()
    w0, u0d = server.w.double().cpu().numpy(), server.u.double().cpu().numpy()
    flag = torch.zeros(1, dtype=torch.int32).pin_memory()
    status = torch.full((1,), 7, dtype=torch.int32).pin_memory()
    D.dbl_hold(flag, 5.0, status, it.stream_s)  # the small worker's step queues behind this
    rc, failed = it.run_with_deadline(0.5)
    held = int(status[0])  # still 7 while the hold waits
    assert (rc, failed, held) == (D.DBL_ERR_TIMEOUT, ["S"], 7)
    it.stream_l.synchronize()
    torch.cuda.current_stream().synchronize()  # the merge, which did not wait for the held stream
    rw, ru = orc.ps_merge(w0, u0d, large.grad.double().cpu().numpy(), None, 0.2, 0.9, 1.0, fS, 0)
    assert max_norm_rel(server.w.double().cpu().numpy(), rw) <= 1e-6
    assert max_norm_rel(server.u.double().cpu().numpy(), ru) <= 1e-6
    flag[0] = 1  # release the straggler
    torch.cuda.synchronize()
    assert int(status[0]) == D.DBL_OK  # released by the host, not by the hold's own timeout
    assert D.dbl_device_status() == D.DBL_OK
    # a normal iteration afterwards: both pushes arrive and are merged
    w1, u1 = server.w.double().cpu().numpy(), server.u.double().cpu().numpy()
    rc, failed = it.run_with_deadline(60.0)
    torch.cuda.synchronize()
    assert rc == D.DBL_OK and failed == []
    rw, ru = orc.ps_merge(w1, u1, large.grad.double().cpu().numpy(), small.grad.double().cpu().numpy(), 0.2, 0.9,
                          1.0, fS, 0)
    assert max_norm_rel(server.w.double().cpu().numpy(), rw) <= 1e-6
    assert max_norm_rel(server.u.double().cpu().numpy(), ru) <= 1e-6


def test_fp16_dual_batch_iteration_matches_oracle(R):
    """The dual-batch iteration in fp16 mixed precision with loss scaling (Sec. 5.2.3): binary16
    storage, loss scale 2^15, the server's scaled merge.  Losses and the pushed (scaled) gradients
    against the oracle rounding to binary16 at the same storage points, the merge against the
    oracle's scaled merge of the GPU's own pushes, and the dynamic scale's first good step."""
    D = load_dbl()
    spec = R.ResNet18Spec("cifar", 100)
    params = synth.params(spec.table(), seed=8, random_bn=True)
    u0 = synth.momentum_state(spec.table(), 0.01, seed=8)
    img = synth.images(8, 32, 32, 3, seed=8)
    lab = synth.labels(8, 100, seed=8)
    S = 2.0 ** 15
    server = R.ServerState(spec, params, u0, precision="f16", loss_scale=S)
    large = R.Worker(spec, 6, 24, dropout=0.2, dropout_seed=11, precision="f16")
    small = R.Worker(spec, 2, 24, dropout=0.2, dropout_seed=12, precision="f16")
    fS = 19.0 / 21.0
    it = R.DualBatchIteration(server, large, small, 32, lr=0.2, momentum=0.9, f_large=1.0, f_small=fS, order=0)
    it.set_inputs(torch.from_numpy(img[2:]).cuda(), torch.from_numpy(lab[2:]).cuda(), torch.from_numpy(img[:2]).cuda(),
                  torch.from_numpy(lab[:2]).cuda())
    w_before, u_before = server.w.clone(), server.u.clone()
    it.run()
    torch.cuda.synchronize()
    assert D.dbl_device_status() == D.DBL_OK
    assert server.w16.dtype == torch.float16 and large.x0.dtype == torch.float16
    d = float(np.float32(0.2))
    p64 = {k: v.astype(np.float64) for k, v in params.items()}
    u64 = {k: v.astype(np.float64) for k, v in u0.items()}
    kw = dict(order=0, dropout_large=(d, 11, 0), dropout_small=(d, 12, 0), loss_scale=S)
    nw, nu, lL, lS, gL, gS = OR.dual_batch_iteration(p64, u64, img[2:], lab[2:], img[:2], lab[:2], 24, "cifar", 0.2,
                                                     0.9, 1.0, fS, storage="f16", **kw)
    _, _, _, _, gL64, gS64 = OR.dual_batch_iteration(p64, u64, img[2:], lab[2:], img[:2], lab[:2], 24, "cifar", 0.2,
                                                     0.9, 1.0, fS, storage=None, **kw)
    assert abs(large.loss.item() - lL) <= TOL * abs(lL)
    assert abs(small.loss.item() - lS) <= TOL * abs(lS)
    _compare_grads(spec, large.grad, gL, gL64, "fp16 large worker")
    _compare_grads(spec, small.grad, gS, gS64, "fp16 small worker")
    rw, ru, ok = orc.ps_merge_scaled(w_before.double().cpu().numpy(), u_before.double().cpu().numpy(),
                                     large.grad.double().cpu().numpy(), small.grad.double().cpu().numpy(), 0.2, 0.9,
                                     1.0, fS, 0, S, S)
    assert ok
    assert max_norm_rel(server.w.double().cpu().numpy(), rw) <= 1e-6
    assert max_norm_rel(server.u.double().cpu().numpy(), ru) <= 1e-6
    assert torch.equal(server.w16, server.w.to(torch.float16))
    assert server.loss_scale() == (S, 1, 0)


def test_fp16_overflow_skips_the_update_and_halves_the_scale(R):
    """A loss scale far too large makes the scaled gradients overflow binary16: the server finds
    the non-finite push, leaves the model as it was, halves the scale and counts the skip."""
    D = load_dbl()
    spec = R.ResNet18Spec("cifar", 100)
    params = synth.params(spec.table(), seed=9)
    server = R.ServerState(spec, params, precision="f16", loss_scale=2.0 ** 60)
    it = R.DualBatchIteration(server, R.Worker(spec, 6, 24, precision="f16"), R.Worker(spec, 2, 24, precision="f16"),
                              32)
    img = torch.from_numpy(synth.images(8, 32, 32, 3, seed=9)).cuda()
    lab = torch.from_numpy(synth.labels(8, 100, seed=9)).cuda()
    it.set_inputs(img[2:], lab[2:], img[:2], lab[:2])
    w0, u0, w160 = server.w.clone(), server.u.clone(), server.w16.clone()
    it.run()
    torch.cuda.synchronize()
    assert D.dbl_device_status() == D.DBL_OK
    assert not torch.isfinite(it.large.grad).all()
    assert torch.equal(server.w, w0) and torch.equal(server.u, u0) and torch.equal(server.w16, w160)
    assert server.loss_scale() == (2.0 ** 59, 0, 1)


def test_a_hold_that_is_never_released_times_out_on_the_device(R):
    """A bounded device wait that runs out: the hold gives up after its limit, reports
    DBL_ERR_TIMEOUT in its status word, and the stream (and the context) carry on."""
    D = load_dbl()
    flag = torch.zeros(1, dtype=torch.int32).pin_memory()  # nothing ever sets it
    status = torch.full((1,), 7, dtype=torch.int32).pin_memory()
    after = torch.ones(4, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    D.dbl_hold(flag, 0.2, status, s)
    with torch.cuda.stream(s):
        after.mul_(3.0)  # queued behind the hold
    s.synchronize()
    assert int(status[0]) == D.DBL_ERR_TIMEOUT
    assert torch.equal(after, torch.full((4,), 3.0, device="cuda"))
    assert D.dbl_device_status() == D.DBL_OK  # the hold reports through its own word only


_STEP_IN_CHILD = r"""
import sys, torch
sys.path.insert(0, sys.argv[1])
from paper_2509_26092_gb300 import build_lib
build_lib.build()
from paper_2509_26092_gb300 import resnet18 as R, synth
spec = R.ResNet18Spec("imagenet", 1000)
server = R.ServerState(spec, synth.params(spec.table(), seed=21, random_bn=True))
wk = R.Worker(spec, 8, 96)
wk.labels.copy_(torch.from_numpy(synth.labels(8, 1000, seed=21)).cuda())
img = torch.from_numpy(synth.images(8, 96, 96, 3, seed=21)).cuda()
for _ in range(2):
    wk.enqueue_step(server, img, 96, torch.cuda.current_stream())
torch.cuda.synchronize()
torch.save(wk.grad.cpu(), sys.argv[2])
"""


def test_programmatic_dependent_launch_gives_the_same_step(R, tmp_path):
    """Convolutions launched with programmatic stream serialization (DBL_CONV_PDL=1, read once per
    process, hence a child process) give the same gradients, bit for bit, as in plain stream order."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = {}
    for flag in ("0", "1"):
        path = str(tmp_path / f"grad{flag}.pt")
        r = subprocess.run([sys.executable, "-c", _STEP_IN_CHILD, root, path], capture_output=True, text=True,
                           timeout=600, env=dict(os.environ, DBL_CONV_PDL=flag))
        assert r.returncode == 0, r.stderr[-2000:]
        out[flag] = torch.load(path)
    assert torch.isfinite(out["1"]).all() and torch.equal(out["0"], out["1"])
