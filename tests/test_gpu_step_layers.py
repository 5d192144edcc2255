"""Teacher-forced parity of every layer inside a real GPU training step.

After one ResNet-18 step on the GPU, each layer's stored inputs (the GPU's
own bf16 activations, gradients and saved BatchNorm statistics) are fed to
the fp64 oracle's version of that layer, and the oracle's result is compared
with what the GPU stored.  This checks each step of the path at its real
shapes and data distribution, independent of how rounding differences
compound across twenty layers.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from conftest import max_norm_rel
from gpu_common import load_dbl, stem_fold
from paper_2509_26092_gb300 import synth

pytestmark = pytest.mark.gpu

TOL = 1e-2


def h(t):
    return t.detach().double().cpu().numpy()


@pytest.mark.parametrize("variant,classes,batch,res,precision", [
    ("cifar", 100, 8, 32, "bf16"), ("imagenet", 1000, 4, 96, "bf16"),
    ("cifar", 100, 256, 32, "bf16"),                                     # the CIFAR step at its batch
    ("imagenet", 1000, 4, 96, "f16")])                                   # fp16 storage, loss scale 2^15
def test_every_layer_of_the_step(variant, classes, batch, res, precision):
    load_dbl()
    from paper_2509_26092_gb300 import resnet18 as R
    spec = R.ResNet18Spec(variant, classes)
    params = synth.params(spec.table(), seed=11, random_bn=True)
    server = R.ServerState(spec, params, precision=precision)
    wk = R.Worker(spec, batch, res, precision=precision)
    scale = server.loss_scale()[0] if server.scaled else 1.0  # every gradient is the loss's times this
    img = torch.from_numpy(synth.images(batch, res, res, 3, seed=11)).cuda()
    wk.labels.copy_(torch.from_numpy(synth.labels(batch, classes, seed=11)).cuda())
    wk.enqueue_step(server, img, res, torch.cuda.current_stream())
    torch.cuda.synchronize()
    W16 = {e.name: h(spec.view(server.w16, e.name)) for e in spec.entries}
    P = {e.name: h(spec.view(server.w, e.name)) for e in spec.entries}
    G = {e.name: h(spec.view(wk.grad, e.name)) for e in spec.entries}
    errs = {}

    def chk(tag, got, ref, tol=TOL):
        e = max_norm_rel(got, ref)
        errs[tag] = e
        assert e <= tol, f"{tag}: {e:.3e}"

    eps = wk.eps
    # ---------------- forward
    st = spec.stem
    lay = spec.stem_layout
    x0 = stem_fold(h(wk.x0), st.r, st.stride, st.pad, res, lay.rg, lay.pad_h)[..., :3]  # the logical stem input
    assert not np.any(np.isnan(x0))
    w_stem = W16["conv1.w"][:, :st.r, :st.r, :3]
    chk("stem.conv", h(wk.stem_y), orc.conv2d_fwd(x0, w_stem, st.stride, st.pad))
    o, m, s = orc.bn_fwd(h(wk.stem_y), P["bn1.g"], P["bn1.b"], eps, relu=True)
    chk("stem.bn.mean", h(wk.stem_stats[2]), m, 1e-4)
    if variant == "imagenet":
        # the BatchNorm output is pooled on the fly (never stored): pool the oracle's stored values
        stem_a = (orc.round_f16 if precision == "f16" else orc.round_bf16)(o)
        y, arg = orc.maxpool_fwd(stem_a)
        chk("stem.bn.pool", h(wk.pool_out), y)
        agree = np.mean(wk.pool_arg.cpu().numpy().astype(np.int32) == arg)
        assert agree > 0.999, f"argmax agreement {agree}"  # ties may fall either way within one bf16 ulp
    else:
        stem_a = h(wk.stem_a)
        chk("stem.bn", stem_a, o)
    for d in wk.blocks:
        b = d["spec"]
        x = h(d["x"])
        chk(b.pre + ".conv1", h(d["h1"]), orc.conv2d_fwd(x, W16[b.pre + ".conv1.w"], b.stride, 1))
        chk(b.pre + ".bn1", h(d["o1"]), orc.bn_fwd(h(d["h1"]), P[b.pre + ".bn1.g"], P[b.pre + ".bn1.b"], eps)[0])
        chk(b.pre + ".conv2", h(d["h2"]), orc.conv2d_fwd(h(d["o1"]), W16[b.pre + ".conv2.w"], 1, 1))
        if b.proj:
            chk(b.pre + ".down", h(d["hs"]), orc.conv2d_fwd(x, W16[b.pre + ".down.w"], b.stride, 0))
            chk(b.pre + ".downbn", h(d["sc"]),
                orc.bn_fwd(h(d["hs"]), P[b.pre + ".downbn.g"], P[b.pre + ".downbn.b"], eps, relu=False)[0])
            res_ = h(d["sc"])
        else:
            res_ = x
        chk(b.pre + ".bn2", h(d["out"]),
            orc.bn_fwd(h(d["h2"]), P[b.pre + ".bn2.g"], P[b.pre + ".bn2.b"], eps, res=res_)[0])
    # ---------------- head
    last = h(wk.blocks[-1]["out"])
    feat = orc.avgpool_fwd(last)
    logits = orc.fc_fwd(feat, P["fc.w"], P["fc.b"])
    loss, dl = orc.softmax_ce(logits, wk.labels.cpu().numpy())
    dW, db, df = orc.fc_bwd(dl * scale, feat, P["fc.w"])
    assert abs(wk.loss.item() - loss) <= 1e-5 * abs(loss)
    chk("fc.w.grad", G["fc.w"], dW, 1e-4)
    chk("fc.b.grad", G["fc.b"], db, 1e-4)
    chk("head.dx", h(wk.dfeat), orc.avgpool_bwd(df, last.shape))
    # ---------------- backward, block by block, from the GPU's own incoming gradients
    dout, dout2 = h(wk.dfeat), None
    for d in reversed(wk.blocks):
        b = d["spec"]
        x = h(d["x"])
        st2 = [h(t) for t in d["bn2"]]
        dh2, dg2, db2, dres = orc.bn_bwd(dout, h(d["out"]), h(d["h2"]), P[b.pre + ".bn2.g"], st2[2], st2[3],
                                         relu=True, dout2=dout2, want_dres=True)
        chk(b.pre + ".bn2.bwd", h(d["dh2"]), dh2)
        chk(b.pre + ".bn2.g.grad", G[b.pre + ".bn2.g"], dg2, 1e-3)
        chk(b.pre + ".bn2.b.grad", G[b.pre + ".bn2.b"], db2, 1e-3)
        chk(b.pre + ".conv2.wgrad", G[b.pre + ".conv2.w"], orc.conv2d_wgrad(h(d["o1"]), h(d["dh2"]),
                                                                              W16[b.pre + ".conv2.w"].shape, 1, 1))
        chk(b.pre + ".conv2.dgrad", h(d["do1"]), orc.conv2d_dgrad(h(d["dh2"]), W16[b.pre + ".conv2.w"],
                                                                  d["o1"].shape, 1, 1))
        st1 = [h(t) for t in d["bn1"]]
        dh1, dg1, db1, _ = orc.bn_bwd(h(d["do1"]), h(d["o1"]), h(d["h1"]), P[b.pre + ".bn1.g"], st1[2], st1[3])
        chk(b.pre + ".bn1.bwd", h(d["dh1"]), dh1)
        chk(b.pre + ".bn1.g.grad", G[b.pre + ".bn1.g"], dg1, 1e-3)
        chk(b.pre + ".conv1.wgrad", G[b.pre + ".conv1.w"], orc.conv2d_wgrad(x, h(d["dh1"]),
                                                                              W16[b.pre + ".conv1.w"].shape, b.stride,
                                                                              1))
        din_ref = orc.conv2d_dgrad(h(d["dh1"]), W16[b.pre + ".conv1.w"], x.shape, b.stride, 1)
        if b.proj:
            std = [h(t) for t in d["downbn"]]
            dhs, dgs, dbs, _ = orc.bn_bwd(dout, h(d["out"]), h(d["hs"]), P[b.pre + ".downbn.g"], std[2], std[3],
                                          relu=True, dout2=dout2)
            chk(b.pre + ".downbn.bwd", h(d["dhs"]), dhs)
            chk(b.pre + ".down.wgrad", G[b.pre + ".down.w"], orc.conv2d_wgrad(x, h(d["dhs"]),
                                                                                W16[b.pre + ".down.w"].shape,
                                                                                b.stride, 0))
            # the projection's data gradient is accumulated into conv1's in one pass
            din_ref = din_ref + orc.conv2d_dgrad(h(d["dhs"]), W16[b.pre + ".down.w"], x.shape, b.stride, 0)
            chk(b.pre + ".conv1+down.dgrad", h(d["din"]), din_ref)
            dout, dout2 = h(d["din"]), None
        else:
            chk(b.pre + ".conv1.dgrad", h(d["din"]), din_ref)
            chk(b.pre + ".dres", h(d["din2"]), dres)
            dout, dout2 = h(d["din"]), h(d["din2"])
    s_stats = [h(t) for t in wk.stem_stats]
    if variant == "imagenet":
        da = orc.maxpool_bwd(dout + (dout2 if dout2 is not None else 0), wk.pool_arg.cpu().numpy().astype(np.int32), stem_a.shape)
        chk("stem.pool.bwd", h(wk.stem_da), da)
        dys, dgs, dbs, _ = orc.bn_bwd(h(wk.stem_da), stem_a, h(wk.stem_y), P["bn1.g"], s_stats[2], s_stats[3])
    else:
        dys, dgs, dbs, _ = orc.bn_bwd(dout, stem_a, h(wk.stem_y), P["bn1.g"], s_stats[2], s_stats[3], dout2=dout2)
    chk("stem.bn.bwd", h(wk.stem_dy), dys)
    wst = orc.conv2d_wgrad(x0, h(wk.stem_dy), w_stem.shape, st.stride, st.pad)
    chk("stem.wgrad", G["conv1.w"][:, :st.r, :st.r, :3], wst)
    assert np.all(G["conv1.w"][:, st.r:] == 0.0)  # rows of the stored layout past the filter
    # padded filter columns and input channels get no gradient
    assert np.all(G["conv1.w"][:, :, st.r:, :] == 0.0) and np.all(G["conv1.w"][..., 3:] == 0.0)
    worst = sorted(errs.items(), key=lambda kv: -kv[1])[:6]
    print(f"\n{variant}: {len(errs)} layer checks; worst " + ", ".join(f"{k}={v:.2e}" for k, v in worst))
