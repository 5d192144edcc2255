"""fp64 reference ResNet-18 training step and dual-batch iteration.

TEST INFRASTRUCTURE ONLY (see the package docstring).

The network is the ResNet-18 of Sec. 5.1.1: a stem convolution, four stages of
two BasicBlocks (widths 64/128/256/512, the first block of stages 2-4 with
stride 2 and a 1x1 stride-2 projection shortcut followed by BatchNorm), global
average pooling (Sec. 6) and one fully connected layer.  Two stems:

* ``cifar``: 3x3 stride-1 convolution, no max pooling;
* ``imagenet``: 7x7 stride-2 convolution, then 3x3 stride-2 max pooling.

The loss is the batch-mean softmax cross-entropy, so every gradient is the
batch mean of Eq. 1.

``bf16_storage=True`` rounds to bfloat16 exactly where the mixed-precision
GPU step stores a bfloat16 tensor, so that a whole-step comparison compares
like with like:

* the network input after resizing;
* every convolution output (BatchNorm statistics are taken of the rounded
  values), every BatchNorm/ReLU output (the projection shortcut's BatchNorm
  output included), the max-pool output;
* every activation gradient: BatchNorm backward outputs, the residual-branch
  gradient, convolution data gradients, the average-pool backward output and
  the max-pool backward output;
* convolution weights are read as bfloat16 copies of the fp32 master weights.

Everything else (BatchNorm statistics, pooled features, logits, all weight
gradients, BatchNorm and fully connected parameters) stays unrounded.
"""
import math

import numpy as np

from . import (avgpool_bwd, avgpool_fwd, bilinear_resize, bn_bwd, bn_fwd, conv2d_dgrad, conv2d_fwd, conv2d_wgrad,
               dropout_apply, dropout_mask, fc_bwd, fc_fwd, maxpool_bwd, maxpool_fwd, ps_merge, ps_merge_scaled,
               round_bf16, round_f16, softmax_ce)

WIDTHS = (64, 128, 256, 512)


def layer_table(variant, classes, widths=WIDTHS, in_ch=3):
    """List of (name, shape, fan_in) for every parameter tensor, in network order.

    Conv weights are [K, R, S, C]; BatchNorm has '.g' (gamma) and '.b' (beta);
    the fully connected layer has 'fc.w' [classes, C] and 'fc.b' [classes].
    """
    t = []

    def conv(name, k, r, c):
        t.append((name + ".w", (k, r, r, c), r * r * c))

    def bn(name, c):
        t.append((name + ".g", (c,), None))
        t.append((name + ".b", (c,), None))

    stem_r = 3 if variant == "cifar" else 7
    conv("conv1", widths[0], stem_r, in_ch)
    bn("bn1", widths[0])
    c_in = widths[0]
    for li, wdt in enumerate(widths):
        for bi in range(2):
            pre = f"layer{li + 1}.{bi}"
            stride = 2 if (li > 0 and bi == 0) else 1
            conv(pre + ".conv1", wdt, 3, c_in)
            bn(pre + ".bn1", wdt)
            conv(pre + ".conv2", wdt, 3, wdt)
            bn(pre + ".bn2", wdt)
            if stride != 1 or c_in != wdt:
                conv(pre + ".down", wdt, 1, c_in)
                bn(pre + ".downbn", wdt)
            c_in = wdt
    t.append(("fc.w", (classes, c_in), c_in))
    t.append(("fc.b", (classes,), None))
    return t


def n_params(variant, classes, widths=WIDTHS):
    return sum(int(np.prod(s)) for _, s, _ in layer_table(variant, classes, widths))


class _Rounder:
    """Rounding at the points where the GPU stores 16-bit values: bf16, fp16 (IEEE binary16),
    or none (fp64 throughout)."""

    def __init__(self, mode):
        self.fn = {"bf16": round_bf16, "f16": round_f16, None: None}[mode]

    def __call__(self, a):
        return self.fn(a) if self.fn else a


def _check_params(params, variant, classes, widths):
    for name, shape, _ in layer_table(variant, classes, widths):
        if name not in params:
            raise KeyError(f"missing parameter {name}")
        if tuple(params[name].shape) != tuple(shape):
            raise ValueError(f"{name}: shape {params[name].shape} != {shape}")


def train_step(params, img, labels, variant, bf16_storage=True, eps=1e-5, widths=WIDTHS, keep=False, dropout=None,
               storage="", loss_scale=1.0):
    """One worker's forward + backward on a batch.

    params: dict name -> fp32-valued array (the master weights the worker pulled);
    img: [N, H, W, 3] float, already at the training resolution; labels: [N] int.
    dropout: None, or (d, seed, step): dropout of rate d on the pooled features before
    the FC layer (Sec. 4.1), with the mask of ``dropout_mask(N, C, d, seed, step)``.
    storage: "bf16", "f16" or None picks the 16-bit format rounded to at the GPU's storage
    points (the default "" follows bf16_storage).  loss_scale: the backward pass starts from
    loss_scale * dloss, as mixed-precision training with loss scaling does (Sec. 5.2.3), so
    the returned gradients are loss_scale times the loss's; the loss itself is unscaled.
    Returns dict(loss=float, grads={name: array}, acts={...} if keep).
    """
    classes = params["fc.w"].shape[0]
    _check_params(params, variant, classes, widths)
    R = _Rounder(storage if storage != "" else ("bf16" if bf16_storage else None))
    P = {k: np.asarray(v, dtype=np.float64) for k, v in params.items()}
    wq = {k: R(v) for k, v in P.items() if k.endswith(".w") and v.ndim == 4}  # bf16 conv weights
    acts = {}
    tape = []  # (kind, info) records for the backward pass

    def conv_bn(x, cname, bname, stride, pad, relu, res=None):
        w = wq[cname + ".w"]
        y = R(conv2d_fwd(x, w, stride, pad))
        out, mean, invstd = bn_fwd(y, P[bname + ".g"], P[bname + ".b"], eps, res=res, relu=relu)
        out = R(out)
        return y, out, mean, invstd

    x0 = R(np.asarray(img, dtype=np.float64))
    N = x0.shape[0]
    # stem
    sr, sst, spd = (3, 1, 1) if variant == "cifar" else (7, 2, 3)
    y, a, mu, istd = conv_bn(x0, "conv1", "bn1", sst, spd, True)
    stem = dict(x=x0, y=y, out=a, mean=mu, invstd=istd, stride=sst, pad=spd)
    if variant == "imagenet":
        m, arg = maxpool_fwd(a, 3, 2, 1)
        stem["pool_arg"] = arg
        cur = m
    else:
        cur = a
    blocks = []
    c_in = widths[0]
    for li, wdt in enumerate(widths):
        for bi in range(2):
            pre = f"layer{li + 1}.{bi}"
            stride = 2 if (li > 0 and bi == 0) else 1
            blk = dict(pre=pre, x=cur, stride=stride)
            blk["h1"], blk["o1"], blk["m1"], blk["s1"] = conv_bn(cur, pre + ".conv1", pre + ".bn1", stride, 1, True)
            blk["h2"] = R(conv2d_fwd(blk["o1"], wq[pre + ".conv2.w"], 1, 1))
            if stride != 1 or c_in != wdt:
                blk["hs"], blk["sc"], blk["ms"], blk["ss"] = conv_bn(cur, pre + ".down", pre + ".downbn", stride, 0,
                                                                     False)
                res = blk["sc"]
                blk["proj"] = True
            else:
                res = cur
                blk["proj"] = False
            out, blk["m2"], blk["s2"] = bn_fwd(blk["h2"], P[pre + ".bn2.g"], P[pre + ".bn2.b"], eps, res=res,
                                               relu=True)
            blk["out"] = R(out)
            cur = blk["out"]
            blocks.append(blk)
            c_in = wdt
    feat = avgpool_fwd(cur)
    mask = None
    if dropout is not None and dropout[0] > 0.0:
        mask = dropout_mask(feat.shape[0], feat.shape[1], dropout[0], dropout[1], dropout[2])
        feat = dropout_apply(feat, mask, dropout[0])
    logits = fc_fwd(feat, P["fc.w"], P["fc.b"])
    loss, dl = softmax_ce(logits, labels)
    dl = dl * loss_scale

    grads = {}
    grads["fc.w"], grads["fc.b"], dfeat = fc_bwd(dl, feat, P["fc.w"])
    if mask is not None:
        dfeat = dropout_apply(dfeat, mask, dropout[0])
    dout = R(avgpool_bwd(dfeat, cur.shape))
    dout2 = None
    for blk in reversed(blocks):
        pre = blk["pre"]
        dh2, grads[pre + ".bn2.g"], grads[pre + ".bn2.b"], dres = bn_bwd(
            dout, blk["out"], blk["h2"], P[pre + ".bn2.g"], blk["m2"], blk["s2"], relu=True, dout2=dout2,
            want_dres=not blk["proj"])
        dh2 = R(dh2)
        grads[pre + ".conv2.w"] = conv2d_wgrad(blk["o1"], dh2, wq[pre + ".conv2.w"].shape, 1, 1)
        do1 = R(conv2d_dgrad(dh2, wq[pre + ".conv2.w"], blk["o1"].shape, 1, 1))
        dh1, grads[pre + ".bn1.g"], grads[pre + ".bn1.b"], _ = bn_bwd(
            do1, blk["o1"], blk["h1"], P[pre + ".bn1.g"], blk["m1"], blk["s1"], relu=True)
        dh1 = R(dh1)
        x = blk["x"]
        st = blk["stride"]
        grads[pre + ".conv1.w"] = conv2d_wgrad(x, dh1, wq[pre + ".conv1.w"].shape, st, 1)
        din = R(conv2d_dgrad(dh1, wq[pre + ".conv1.w"], x.shape, st, 1))
        if blk["proj"]:
            # the shortcut BatchNorm sees the same masked gradient g as bn2
            dhs, grads[pre + ".downbn.g"], grads[pre + ".downbn.b"], _ = bn_bwd(
                dout, blk["out"], blk["hs"], P[pre + ".downbn.g"], blk["ms"], blk["ss"], relu=True, dout2=dout2)
            dhs = R(dhs)
            grads[pre + ".down.w"] = conv2d_wgrad(x, dhs, wq[pre + ".down.w"].shape, st, 0)
            din2 = R(conv2d_dgrad(dhs, wq[pre + ".down.w"], x.shape, st, 0))
        else:
            din2 = R(dres)
        dout, dout2 = din, din2
    if variant == "imagenet":
        dm = dout + dout2
        da = R(maxpool_bwd(dm, stem["pool_arg"], stem["out"].shape, 3, 2, 1))
        dys, grads["bn1.g"], grads["bn1.b"], _ = bn_bwd(da, stem["out"], stem["y"], P["bn1.g"], stem["mean"],
                                                        stem["invstd"], relu=True)
    else:
        dys, grads["bn1.g"], grads["bn1.b"], _ = bn_bwd(dout, stem["out"], stem["y"], P["bn1.g"], stem["mean"],
                                                        stem["invstd"], relu=True, dout2=dout2)
    dys = R(dys)
    grads["conv1.w"] = conv2d_wgrad(x0, dys, wq["conv1.w"].shape, stem["stride"], stem["pad"])
    res = dict(loss=loss, grads=grads, logits=logits)
    if keep:
        res["acts"] = dict(stem=stem, blocks=blocks, feat=feat, dlogits=dl, dropout_keep=mask)
    return res


def dual_batch_iteration(params, velocity, img_large, labels_large, img_small, labels_small, resolution, variant,
                         lr, momentum, f_large, f_small, order=0, bf16_storage=True, widths=WIDTHS,
                         dropout_large=None, dropout_small=None, storage="", loss_scale=None):
    """One emulated parameter-server iteration of the hybrid scheme (Sec. 3-4).

    Both workers pull the same model version, resize their images to the
    sub-stage resolution (Sec. 4.1), run one training step each, and the server
    applies their pushes with the model-update factors (Sec. 3.4).
    dropout_large / dropout_small: each worker's (d, seed, step) for ``train_step``, or None.
    loss_scale: None, or the scale both workers multiply their loss by (storage then usually
    "f16"); the server divides each push by it and skips the update if a pushed value is not
    finite (``ps_merge_scaled``).
    Returns (new_params, new_velocity, loss_large, loss_small, grads_large, grads_small).
    """
    out = {}
    for tag, img, lab, drop in (("L", img_large, labels_large, dropout_large),
                                ("S", img_small, labels_small, dropout_small)):
        if img is None:
            out[tag] = None
            continue
        x = np.asarray(img, dtype=np.float64)
        if x.shape[1] != resolution or x.shape[2] != resolution:
            x = bilinear_resize(x, resolution, resolution)
        out[tag] = train_step(params, x, lab, variant, bf16_storage=bf16_storage, widths=widths, dropout=drop,
                              storage=storage, loss_scale=1.0 if loss_scale is None else loss_scale)
    new_w, new_u = {}, {}
    if loss_scale is not None:
        # one server decision for the whole push: any non-finite value anywhere skips the update
        finite = all(np.all(np.isfinite(out[t]["grads"][name])) for t in ("L", "S") if out[t] for name in params)
        if not finite:
            return (dict(params), dict(velocity), out["L"]["loss"] if out["L"] else None,
                    out["S"]["loss"] if out["S"] else None, out["L"]["grads"] if out["L"] else None,
                    out["S"]["grads"] if out["S"] else None)
    for name in params:
        gl = out["L"]["grads"][name] if out["L"] else None
        gs = out["S"]["grads"][name] if out["S"] else None
        if loss_scale is not None:
            new_w[name], new_u[name], _ = ps_merge_scaled(params[name], velocity[name], gl, gs, lr, momentum,
                                                          f_large, f_small, order, loss_scale, loss_scale)
        else:
            new_w[name], new_u[name] = ps_merge(params[name], velocity[name], gl, gs, lr, momentum, f_large,
                                                f_small, order)
    return (new_w, new_u, out["L"]["loss"] if out["L"] else None, out["S"]["loss"] if out["S"] else None,
            out["L"]["grads"] if out["L"] else None, out["S"]["grads"] if out["S"] else None)


def conv_flops(variant, batch, res, widths=WIDTHS, in_ch=3):
    """Algorithmic conv FLOPs (2*M*N*K per pass) for fwd + dgrad (not the stem) + wgrad."""
    total = 0
    h = res
    stem_r, sst, spd = (3, 1, 1) if variant == "cifar" else (7, 2, 3)
    p = (h + 2 * spd - stem_r) // sst + 1
    f = 2 * batch * p * p * widths[0] * stem_r * stem_r * in_ch
    total += 2 * f  # fwd + wgrad
    h = p
    if variant == "imagenet":
        h = (h + 2 - 3) // 2 + 1
    c_in = widths[0]
    for li, wdt in enumerate(widths):
        for bi in range(2):
            st = 2 if (li > 0 and bi == 0) else 1
            ho = (h + 2 - 3) // st + 1
            total += 3 * 2 * batch * ho * ho * wdt * 9 * c_in
            total += 3 * 2 * batch * ho * ho * wdt * 9 * wdt
            if st != 1 or c_in != wdt:
                total += 3 * 2 * batch * ho * ho * wdt * c_in
            h, c_in = ho, wdt
    return total


def kaiming_std(fan_in):
    return math.sqrt(2.0 / fan_in)
