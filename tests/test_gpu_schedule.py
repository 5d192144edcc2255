"""The asynchronous (ASP) dual-batch driver on the GPU: pushes are merged in arrival
order, each one by the oracle's merge rule, and every pushed gradient was computed
on the model its worker pulled after its own previous push (stale with respect to the
other worker's pushes in between)."""
import numpy as np
import pytest
import torch

import oracle as orc
from conftest import max_norm_rel
from gpu_common import load_dbl
from paper_2509_26092_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def mods():
    load_dbl()
    from paper_2509_26092_gb300 import resnet18, schedule
    return resnet18, schedule


def test_async_pushes_follow_asp(mods):
    R, S = mods
    spec = R.ResNet18Spec("cifar", 100)
    params = synth.params(spec.table(), seed=11, random_bn=True)
    server = R.ServerState(spec, params, synth.momentum_state(spec.table(), 0.01, seed=11))
    w0, u0 = server.w.clone(), server.u.clone()
    large, small = R.Worker(spec, 6, 24), R.Worker(spec, 2, 24)
    imgs = {t: [torch.from_numpy(synth.images(n, 32, 32, 3, seed=s)).cuda() for s in (1, 2)]
            for t, n in (("L", 6), ("S", 2))}
    labs = {t: [torch.from_numpy(synth.labels(n, 100, seed=s)).cuda() for s in (1, 2)] for t, n in (("L", 6), ("S", 2))}
    fS = 19.0 / 21.0
    run = S.AsyncDualBatch(server, large, small, 32, imgs["L"], labs["L"], imgs["S"], labs["S"], lr=0.2, momentum=0.9,
                           f_small=fS)
    rec = []

    def on_push(tag, wk, pulled):
        with torch.cuda.stream(run.streams[tag]):  # snapshots in stream order, right after the merge
            rec.append(dict(tag=tag, grad=wk.grad.clone(), used_w=pulled.w.clone(), used_w16=pulled.w16.clone(),
                            server_w=server.w.clone()))

    order = run.run(3.0, 1.0, 2, 6, on_push)
    torch.cuda.synchronize()
    D = load_dbl()
    assert D.dbl_device_status() == D.DBL_OK
    assert "".join(t for _, t, _ in order) == "SSLSSSLS"
    # 1. the server applied the pushes one by one in this order (the oracle's merge, fp64)
    w, u = w0.double().cpu().numpy(), u0.double().cpu().numpy()
    for r in rec:
        g = r["grad"].double().cpu().numpy()
        w, u = orc.ps_merge(w, u, g if r["tag"] == "L" else None, g if r["tag"] == "S" else None, 0.2, 0.9, 1.0, fS, 0)
    assert max_norm_rel(server.w.double().cpu().numpy(), w) <= 1e-6
    assert max_norm_rel(server.u.double().cpu().numpy(), u) <= 1e-6
    assert torch.equal(server.w16, server.w.to(torch.bfloat16))
    # 2. staleness: a worker's k-th step ran on the model as it was right after its own (k-1)-th push
    last = {"L": w0, "S": w0}
    for r in rec:
        assert torch.equal(r["used_w"], last[r["tag"]]), r["tag"]
        assert torch.equal(r["used_w16"], last[r["tag"]].to(torch.bfloat16))
        last[r["tag"]] = r["server_w"]
    # the large worker's second step saw the small worker's three pushes after its first one
    l_pushes = [i for i, r in enumerate(rec) if r["tag"] == "L"]
    assert not torch.equal(rec[l_pushes[1]]["used_w"], rec[l_pushes[0]]["used_w"])
    # 3. each pushed gradient is the step's gradient on those weights (the kernels are deterministic)
    for tag, n in (("L", 6), ("S", 2)):
        fresh = R.Worker(spec, n, 24)
        for k, r in enumerate([r for r in rec if r["tag"] == tag]):
            pulled = S.PulledWeights(server)
            pulled.w.copy_(r["used_w"])
            pulled.w16.copy_(r["used_w16"])
            fresh.labels.copy_(labs[tag][k % 2])
            fresh.enqueue_step(pulled, imgs[tag][k % 2], 32, torch.cuda.current_stream())
            torch.cuda.synchronize()
            assert torch.equal(fresh.grad, r["grad"]), (tag, k)


def test_async_pushes_in_fp16_unscale_by_each_workers_scale(mods):
    """The free-running schedule in fp16 with loss scaling, the scale growing every two good
    pushes: a worker's gradient carries the scale it copied when its step started, which the
    server may have changed before that push arrives; each push must be unscaled by its own
    worker's scale.  Checked against the oracle's scaled merge and scale update, push by push."""
    R, S = mods
    spec = R.ResNet18Spec("cifar", 100)
    params = synth.params(spec.table(), seed=13, random_bn=True)
    server = R.ServerState(spec, params, synth.momentum_state(spec.table(), 0.01, seed=13), precision="f16",
                           loss_scale=2.0 ** 12, growth_interval=2)
    w0, u0 = server.w.clone(), server.u.clone()
    large = R.Worker(spec, 6, 24, precision="f16")
    small = R.Worker(spec, 2, 24, precision="f16")
    imgs = {t: [torch.from_numpy(synth.images(n, 32, 32, 3, seed=s)).cuda() for s in (3, 4)]
            for t, n in (("L", 6), ("S", 2))}
    labs = {t: [torch.from_numpy(synth.labels(n, 100, seed=s)).cuda() for s in (3, 4)] for t, n in (("L", 6), ("S", 2))}
    fS = 19.0 / 21.0
    run = S.AsyncDualBatch(server, large, small, 32, imgs["L"], labs["L"], imgs["S"], labs["S"], lr=0.2, momentum=0.9,
                           f_small=fS)
    rec = []

    def on_push(tag, wk, pulled):
        with torch.cuda.stream(run.streams[tag]):
            rec.append(dict(tag=tag, grad=wk.grad.clone(), scale=wk.scale_used.clone()))

    run.run(3.0, 1.0, 2, 6, on_push)
    torch.cuda.synchronize()
    D = load_dbl()
    assert D.dbl_device_status() == D.DBL_OK
    w, u = w0.double().cpu().numpy(), u0.double().cpu().numpy()
    s, good = 2.0 ** 12, 0
    for r in rec:
        g, sc = r["grad"].double().cpu().numpy(), float(r["scale"].item())
        w, u, ok = orc.ps_merge_scaled(w, u, g if r["tag"] == "L" else None, g if r["tag"] == "S" else None, 0.2, 0.9,
                                       1.0, fS, 0, sc, sc)
        assert ok
        s, good = orc.loss_scale_update(s, good, not ok, 2)
    assert max_norm_rel(server.w.double().cpu().numpy(), w) <= 1e-6
    assert max_norm_rel(server.u.double().cpu().numpy(), u) <= 1e-6
    assert server.loss_scale() == (s, good, 0)
    used = [float(r["scale"].item()) for r in rec]
    assert len(set(used)) > 1 and s > max(used)  # the scale grew during the run, past what any push used
