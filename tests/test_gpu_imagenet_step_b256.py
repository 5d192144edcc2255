"""Parity of the ImageNet-shaped ResNet-18 training step at its stated shape: one step at
224 x 224 px, batch 256 (one worker, single push), checked layer by layer on the step's own
stored tensors.

Each convolution pass (forward, data gradient, weight gradient) of every layer, the stem
included, is checked on sampled outputs that the oracle computes one by one in fp64 from
the GPU's own stored inputs (the tensor's corners always among the samples); BatchNorm
forward and backward of the largest and the smallest layers and the head are checked over
whole tensors.  Tolerance max-norm relative 1e-2 (bf16 storage), 1e-4 for the fp32 head
gradients and BatchNorm statistics.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from conftest import max_norm_rel
from gpu_common import check_status, load_dbl, rng
from paper_2509_26092_gb300 import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2
SAMPLES = 40


def h(t):
    return t.detach().double().cpu().numpy()


def _indices(shape, g):
    idx = [tuple(0 for _ in shape), tuple(d - 1 for d in shape)]
    while len(idx) < SAMPLES:
        idx.append(tuple(int(g.integers(0, d)) for d in shape))
    return idx


def _sampled(tag, got, fn, shape, g, errs):
    idx = _indices(shape, g)
    a = np.array([got[i] for i in idx], dtype=np.float64)
    b = np.array([fn(*i) for i in idx], dtype=np.float64)
    e = float(np.max(np.abs(a - b))) / max(float(np.max(np.abs(b))), 1e-30)
    errs[tag] = e
    assert e <= TOL, f"{tag}: sampled max-norm relative error {e:.3e}"


def test_imagenet_step_at_batch_256_224px():
    D = load_dbl()
    from paper_2509_26092_gb300 import resnet18 as R
    batch, res, classes = 256, 224, 1000
    spec = R.ResNet18Spec("imagenet", classes)
    params = synth.params(spec.table(), seed=12, random_bn=True)
    server = R.ServerState(spec, params)
    wk = R.Worker(spec, batch, res, dropout=0.2, dropout_seed=5)
    img = torch.from_numpy(synth.images(batch, res, res, 3, seed=12)).cuda()
    wk.labels.copy_(torch.from_numpy(synth.labels(batch, classes, seed=12)).cuda())
    wk.enqueue_step(server, img, res, torch.cuda.current_stream())
    torch.cuda.synchronize()
    check_status(D)
    W16 = {e.name: spec.view(server.w16, e.name) for e in spec.entries}
    P = {e.name: h(spec.view(server.w, e.name)) for e in spec.entries}
    G = {e.name: h(spec.view(wk.grad, e.name)) for e in spec.entries}
    g = rng(256)
    errs = {}
    # ---- stem: the 4 x 1 stride-1 convolution of the unrolled input that the kernels compute
    xu = h(wk.x0)
    ws_ = h(W16["conv1.w"]).reshape(64, 4, 1, 64)
    ys, dys = h(wk.stem_y), h(wk.stem_dy)
    _sampled("stem.fwd", ys, lambda n, p, q, k: orc.conv2d_fwd_at(xu, ws_, 1, 0, n, p, q, k), ys.shape, g, errs)
    # weight gradient on the logical 7 x 7 x 3 filter (stored [k][r][s][c] with r, s < 8, c < 4)
    idx = [(0, 0, 0, 0), (63, 6, 6, 2)] + [(int(g.integers(0, 64)), int(g.integers(0, 7)), int(g.integers(0, 7)),
                                            int(g.integers(0, 3))) for _ in range(SAMPLES - 2)]
    a = np.array([G["conv1.w"][i] for i in idx])
    b = np.array([orc.conv2d_wgrad_at(xu, dys, (64, 4, 1, 64), 1, 0, k, r // 2, 0, (r % 2) * 32 + s * 4 + c)
                  for k, r, s, c in idx])
    errs["stem.wgrad"] = float(np.max(np.abs(a - b))) / float(np.max(np.abs(b)))
    assert errs["stem.wgrad"] <= TOL
    assert np.all(G["conv1.w"][:, 7] == 0.0) and np.all(G["conv1.w"][..., 3] == 0.0)
    # ---- every block convolution, forward / data gradient / weight gradient
    for d in wk.blocks:
        b_ = d["spec"]
        x = h(d["x"])
        for cname, xin, yout, dy, dxo, stride, pad in (
                ("conv1", x, d["h1"], d["dh1"], d["din"], b_.stride, 1),
                ("conv2", h(d["o1"]), d["h2"], d["dh2"], d["do1"], 1, 1)) + (
                (("down", x, d["hs"], d["dhs"], None, b_.stride, 0),) if b_.proj else ()):
            name = f"{b_.pre}.{cname}"
            w = h(W16[name + ".w"])
            yv, dyv = h(yout), h(dy)
            _sampled(name + ".fwd", yv, lambda n, p, q, k: orc.conv2d_fwd_at(xin, w, stride, pad, n, p, q, k),
                     yv.shape, g, errs)
            _sampled(name + ".wgrad", G[name + ".w"],
                     lambda k, r, s, c: orc.conv2d_wgrad_at(xin, dyv, w.shape, stride, pad, k, r, s, c), w.shape, g,
                     errs)
            if cname == "conv2":
                dxv = h(dxo)
                _sampled(name + ".dgrad", dxv,
                         lambda n, hh, ww, c: orc.conv2d_dgrad_at(dyv, w, xin.shape, stride, pad, n, hh, ww, c),
                         dxv.shape, g, errs)
        if b_.proj:
            # the block's input gradient: conv1's data gradient with the projection's fused in
            w1, w2 = h(W16[b_.pre + ".conv1.w"]), h(W16[b_.pre + ".down.w"])
            dh1, dhs, din = h(d["dh1"]), h(d["dhs"]), h(d["din"])
            _sampled(b_.pre + ".conv1+down.dgrad", din,
                     lambda n, hh, ww, c: orc.conv2d_dgrad_at(dh1, w1, x.shape, b_.stride, 1, n, hh, ww, c) +
                     orc.conv2d_dgrad_at(dhs, w2, x.shape, b_.stride, 0, n, hh, ww, c), din.shape, g, errs)
        else:
            w1, dh1, din = h(W16[b_.pre + ".conv1.w"]), h(d["dh1"]), h(d["din"])
            _sampled(b_.pre + ".conv1.dgrad", din,
                     lambda n, hh, ww, c: orc.conv2d_dgrad_at(dh1, w1, x.shape, b_.stride, 1, n, hh, ww, c),
                     din.shape, g, errs)
    # ---- BatchNorm over whole tensors: the largest (layer1.0.bn1) and the smallest (layer4.1.bn2)
    eps = wk.eps
    d0, d7 = wk.blocks[0], wk.blocks[-1]
    o, m, s = orc.bn_fwd(h(d0["h1"]), P["layer1.0.bn1.g"], P["layer1.0.bn1.b"], eps)
    assert max_norm_rel(h(d0["o1"]), o) <= TOL
    assert max_norm_rel(h(d0["bn1"][2]), m) <= 1e-4
    dh, dg, db, _ = orc.bn_bwd(h(d0["do1"]), h(d0["o1"]), h(d0["h1"]), P["layer1.0.bn1.g"], h(d0["bn1"][2]),
                               h(d0["bn1"][3]))
    assert max_norm_rel(h(d0["dh1"]), dh) <= TOL
    assert max_norm_rel(G["layer1.0.bn1.g"], dg) <= 1e-3 and max_norm_rel(G["layer1.0.bn1.b"], db) <= 1e-3
    o, _, _ = orc.bn_fwd(h(d7["h2"]), P["layer4.1.bn2.g"], P["layer4.1.bn2.b"], eps, res=h(d7["x"]))
    assert max_norm_rel(h(d7["out"]), o) <= TOL
    # ---- head with the dropout of its first call (step 0), then the counter moved on
    last = h(d7["out"])
    d_ = float(np.float32(0.2))
    keep = orc.dropout_mask(batch, 512, d_, 5, 0)
    feat = orc.dropout_apply(orc.avgpool_fwd(last), keep, d_)
    logits = orc.fc_fwd(feat, P["fc.w"], P["fc.b"])
    loss, dl = orc.softmax_ce(logits, wk.labels.cpu().numpy())
    dW, db, df = orc.fc_bwd(dl, feat, P["fc.w"])
    assert abs(wk.loss.item() - loss) <= 1e-5 * abs(loss)
    assert max_norm_rel(G["fc.w"], dW) <= 1e-4 and max_norm_rel(G["fc.b"], db) <= 1e-4
    assert max_norm_rel(h(wk.dfeat), orc.avgpool_bwd(orc.dropout_apply(df, keep, d_), last.shape)) <= TOL
    assert int(wk.dropout_step.item()) == 1
    worst = sorted(errs.items(), key=lambda kv: -kv[1])[:5]
    print(f"\n{len(errs)} sampled checks; worst " + ", ".join(f"{k}={v:.2e}" for k, v in worst))
