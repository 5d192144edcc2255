"""ResNet-18 training step of the hybrid dual-batch / cyclic-progressive scheme
on one GB300, driven through the C ABI of ``libdbl.so``.

What runs where
---------------
Every arithmetic step is a ``libdbl`` kernel; this module only allocates
device memory (through PyTorch), lays out the flat parameter buffers and
enqueues ABI calls on CUDA streams:

* the parameter server (Sec. 2.3) holds fp32 master weights ``w``, the
  momentum buffer ``u`` and the bf16 copy ``w16`` the workers pull, each one
  flat contiguous buffer;
* a worker (Sec. 3.1) owns the activations of one batch size at one
  resolution and writes its batch-mean gradient into its own flat fp32
  buffer (same layout as ``w``);
* a dual-batch iteration runs the large-batch and the small-batch worker on
  two streams of the same GPU, joins them with an event, and merges both
  pushes into the master weights with the model-update factor (Sec. 3.4);
* the resolution of a cyclic-progressive sub-stage (Sec. 4.1) is produced by
  ``dbl_progressive_resize`` from the native-resolution images.

ResNet-18 (Sec. 5.1.1): stem convolution (3x3/1 for CIFAR-shaped inputs,
7x7/2 + 3x3/2 max pooling for ImageNet-shaped inputs), four stages of two
BasicBlocks (64/128/256/512 channels; the first block of stages 2-4 has
stride 2 and a 1x1 stride-2 projection shortcut with BatchNorm), global
average pooling and one fully connected layer.

The stem runs on the tensor cores as a convolution over an unrolled input
(``StemLayout``): the input preparation (``dbl_progressive_resize_stem``)
writes the resized image unrolled along W, 8 filter columns per output column,
and, for the stride-2 ImageNet stem, also groups two input rows per unrolled
row (8 columns x 4 channels each); the 3x3/1 CIFAR stem keeps one row of 8
columns x 8 channels.  The R x R stem then equals a ceil(R/g) x 1 convolution
of 64-channel rows (g = rows per unrolled row), with stride 1 along W, and
the stem weights are stored as [64][g*ceil(R/g)][8][8/g] with the filter
zero-padded in every direction.

Convolutions read the bf16 weights ``w16``; BatchNorm and the fully connected
layer read the fp32 master weights directly (they are tiny).
"""
import time
from dataclasses import dataclass, field

import numpy as np

import torch

from . import dbl as D

WIDTHS = (64, 128, 256, 512)
# 8-bit images are standardized per channel as p*PIXEL_SCALE + PIXEL_BIAS (fp32): the
# usual ImageNet channel means and deviations of decoded pixels (the paper does not give
# its preprocessing constants)
PIXEL_MEAN = (0.485 * 255, 0.456 * 255, 0.406 * 255)
PIXEL_STD = (0.229 * 255, 0.224 * 255, 0.225 * 255)
PIXEL_SCALE = tuple(float(np.float32(1.0) / np.float32(s)) for s in PIXEL_STD)
PIXEL_BIAS = tuple(float(-np.float32(m) / np.float32(s)) for m, s in zip(PIXEL_MEAN, PIXEL_STD))
ALIGN = 64  # parameter tensors start on 256-byte boundaries


@dataclass
class ConvSpec:
    name: str
    cin: int       # channels as stored (the stem's 3 colour channels padded to 8)
    cin_logical: int
    cout: int
    r: int
    stride: int
    pad: int


@dataclass
class StemLayout:
    """How the stem's input is unrolled for the tensor cores (see dbl_progressive_resize_stem)."""
    rg: int           # input rows per unrolled row: 2 for a stride-2 stem, else 1
    taps: int         # filter rows of the unrolled convolution, ceil(R / rg)
    pad_h: int        # zero rows the input preparation writes above the image
    conv_stride: int  # stride of the unrolled convolution along H
    conv_pad: int     # padding of the unrolled convolution along H

    @classmethod
    def of(cls, cs):
        rg = 2 if cs.stride == 2 else 1
        taps = -(-cs.r // rg)
        return cls(rg, taps, cs.pad if rg == 2 else 0, cs.stride // rg, 0 if rg == 2 else cs.pad)

    def rows(self, res, p):
        """Unrolled rows for an image of res rows and p output rows."""
        return p + self.taps - 1 if self.rg == 2 else res

    def stored_shape(self, cs):
        return (cs.cout, self.rg * self.taps, 8, 8 // self.rg)


@dataclass
class BlockSpec:
    pre: str
    cin: int
    cout: int
    stride: int
    proj: bool


@dataclass
class ParamEntry:
    name: str
    shape: tuple          # stored shape
    logical: tuple        # shape the method defines (stem: 3 input channels)
    fan_in: object
    offset: int
    numel: int = field(init=False)

    def __post_init__(self):
        n = 1
        for s in self.shape:
            n *= s
        self.numel = n


class ResNet18Spec:
    """Layer list and flat parameter layout of a ResNet-18 variant."""

    def __init__(self, variant="cifar", classes=100, widths=WIDTHS):
        if variant not in ("cifar", "imagenet"):
            raise ValueError(variant)
        self.variant, self.classes, self.widths = variant, classes, tuple(widths)
        r, st, pad = (3, 1, 1) if variant == "cifar" else (7, 2, 3)
        self.stem = ConvSpec("conv1", 64, 3, widths[0], r, st, pad)  # 64 = one unrolled row of 128 bytes
        self.stem_layout = StemLayout.of(self.stem)
        self.blocks = []
        cin = widths[0]
        for li, wd in enumerate(widths):
            for bi in range(2):
                stride = 2 if (li > 0 and bi == 0) else 1
                self.blocks.append(BlockSpec(f"layer{li + 1}.{bi}", cin, wd, stride, stride != 1 or cin != wd))
                cin = wd
        self.entries = []
        off = 0

        def add(name, shape, logical, fan_in):
            nonlocal off
            e = ParamEntry(name, tuple(shape), tuple(logical), fan_in, off)
            self.entries.append(e)
            off += (e.numel + ALIGN - 1) // ALIGN * ALIGN

        def conv(cs):
            if cs is self.stem:  # stored [k][g*ceil(r/g)][8 columns][8/g channels], logical [k][r][r][3]
                add(cs.name + ".w", self.stem_layout.stored_shape(cs), (cs.cout, cs.r, cs.r, cs.cin_logical),
                    cs.r * cs.r * cs.cin_logical)
                return
            add(cs.name + ".w", (cs.cout, cs.r, cs.r, cs.cin), (cs.cout, cs.r, cs.r, cs.cin_logical),
                cs.r * cs.r * cs.cin_logical)

        def bn(name, c):
            add(name + ".g", (c,), (c,), None)
            add(name + ".b", (c,), (c,), None)

        conv(self.stem)
        bn("bn1", widths[0])
        for b in self.blocks:
            conv(ConvSpec(b.pre + ".conv1", b.cin, b.cin, b.cout, 3, b.stride, 1))
            bn(b.pre + ".bn1", b.cout)
            conv(ConvSpec(b.pre + ".conv2", b.cout, b.cout, b.cout, 3, 1, 1))
            bn(b.pre + ".bn2", b.cout)
            if b.proj:
                conv(ConvSpec(b.pre + ".down", b.cin, b.cin, b.cout, 1, b.stride, 0))
                bn(b.pre + ".downbn", b.cout)
        add("fc.w", (classes, cin), (classes, cin), cin)
        add("fc.b", (classes,), (classes,), None)
        self.n_flat = off
        self.by_name = {e.name: e for e in self.entries}

    def table(self):
        """(name, logical shape, fan_in) of every parameter tensor, for the input generator."""
        return [(e.name, e.logical, e.fan_in) for e in self.entries]

    def n_params(self):
        """Parameters the method defines (without the stem's channel padding)."""
        n = 0
        for e in self.entries:
            k = 1
            for s in e.logical:
                k *= s
            n += k
        return n

    def view(self, flat, name):
        e = self.by_name[name]
        return flat[e.offset:e.offset + e.numel].view(e.shape)

    def pack(self, tensors, device="cuda", dtype=torch.float32):
        """Flat buffer from {name: array of the logical shape} (stem padding zero)."""
        flat = torch.zeros(self.n_flat, dtype=dtype, device=device)
        for e in self.entries:
            t = torch.as_tensor(tensors[e.name], dtype=dtype)
            if tuple(t.shape) != e.logical:
                raise ValueError(f"{e.name}: shape {tuple(t.shape)} != {e.logical}")
            v = self.view(flat, e.name)
            v.zero_()
            v[tuple(slice(0, d) for d in e.logical)].copy_(t)
        return flat

    def unpack(self, flat):
        """{name: host float64 array of the logical shape} from a flat buffer."""
        out = {}
        for e in self.entries:
            v = self.view(flat, e.name)[tuple(slice(0, d) for d in e.logical)]
            out[e.name] = v.detach().double().cpu().numpy().copy()
        return out


def conv_out(n, r, st, pad):
    return (n + 2 * pad - r) // st + 1


ACT_DTYPE = {"bf16": torch.bfloat16, "f16": torch.float16}


class ServerState:
    """The parameter server's global model: fp32 master w, momentum u, and the 16-bit pull copy
    w16 in the storage format of ``precision`` ("bf16", or "f16" for the fp16 mixed precision of
    the paper's ImageNet runs, Sec. 5.2.3).  With ``loss_scale`` (an initial scale, 2^15 for fp16
    by default) the workers scale their loss and the server keeps the dynamic scale state
    (``dbl_loss_scale``: fp32 scale, int32 good steps, found_inf, skipped updates) on the device."""

    def __init__(self, spec, params, momentum_state=None, device="cuda", precision="bf16", loss_scale="auto",
                 growth_interval=2000):
        self.spec, self.precision = spec, precision
        self.w = spec.pack(params, device)
        self.u = (spec.pack(momentum_state, device) if momentum_state is not None
                  else torch.zeros_like(self.w))
        self.w16 = self.w.to(ACT_DTYPE[precision])
        if loss_scale == "auto":
            loss_scale = 2.0 ** 15 if precision == "f16" else None
        self.scaled = loss_scale is not None
        self.growth_interval = int(growth_interval)
        self.scale_state = torch.zeros(4, dtype=torch.int32, device=device)
        if self.scaled:
            self.scale_state[0:1].view(torch.float32).fill_(float(loss_scale))

    def loss_scale(self):
        """(scale, good steps, skipped updates), read back from the device (synchronous)."""
        st = self.scale_state.cpu()
        return float(st[0:1].view(torch.float32).item()), int(st[1]), int(st[3])

    def apply_pushes(self, g_large, g_small, scale_large, scale_small, lr, momentum, f_large, f_small, order, stream):
        """The server's update from the pushed gradients (either may be None): the merge of Sec. 3.4,
        and under loss scaling first the finiteness check of the pushes, the merge of the unscaled
        pushes (skipped when a value is not finite) and the dynamic scale's update."""
        n = self.spec.n_flat
        with D.precision(self.precision):
            if not self.scaled:
                D.dbl_ps_dual_batch_merge(self.w, self.u, self.w16, g_large, g_small, n, lr, momentum, f_large,
                                          f_small, order, stream)
                return
            found_inf = self.scale_state.data_ptr() + 8
            for g in (g_large, g_small):
                if g is not None:
                    D.dbl_grads_finite(g, n, found_inf, stream)
            D.dbl_ps_dual_batch_merge_scaled(self.w, self.u, self.w16, g_large, g_small, n, lr, momentum, f_large,
                                             f_small, order, scale_large, scale_small, found_inf, stream)
            D.dbl_loss_scale_update(self.scale_state, self.growth_interval, stream)


class Worker:
    """Activations, gradients and scratch of one worker at one (batch, resolution)."""

    def __init__(self, spec, batch, res, device="cuda", eps=1e-5, dropout=0.0, dropout_seed=0, precision="bf16"):
        self.spec, self.batch, self.res, self.eps = spec, batch, res, eps
        self.precision = precision
        # programmatic dependent launch of this worker's convolutions: None leaves the library's
        # setting (DBL_CONV_PDL), True / False override it while the step is enqueued
        self.pdl = None
        # under loss scaling: the scale this worker's step used, copied from the server's at its start
        self.scale_used = torch.ones(1, dtype=torch.float32, device=device)
        # dropout before the FC layer (Sec. 4.1): rate, the worker's seed, and the device step
        # counter the head reads and advances once per step
        self.dropout, self.dropout_seed = float(dropout), int(dropout_seed)
        self.dropout_step = torch.zeros(1, dtype=torch.int64, device=device)
        dev = device
        bf = ACT_DTYPE[precision]
        B = batch

        def act(h, c):
            return torch.empty((B, h, h, c), dtype=bf, device=dev)

        def vec(c):
            return torch.empty(c, dtype=torch.float32, device=dev)

        st = spec.stem
        p = conv_out(res, st.r, st.stride, st.pad)
        self.stem_hw = p
        # stem input unrolled (StemLayout): [B, rows, P, 64]
        self.stem_rows = spec.stem_layout.rows(res, p)
        self.x0 = torch.empty((B, self.stem_rows, p, 64), dtype=bf, device=dev)
        # the ImageNet stem's BatchNorm output is pooled on the fly and never stored
        self.stem_a = act(p, st.cout) if spec.variant != "imagenet" else None
        self.stem_y, self.stem_da, self.stem_dy = act(p, st.cout), None, act(p, st.cout)
        self.stem_stats = [vec(st.cout) for _ in range(4)]  # sum, sumsq, mean, invstd
        h = p
        if spec.variant == "imagenet":
            q = conv_out(p, 3, 2, 1)
            self.pool_out = act(q, st.cout)
            self.pool_arg = torch.empty((B, q, q, st.cout), dtype=torch.uint8, device=dev)
            self.stem_da = act(p, st.cout)
            h = q
        self.blocks = []
        for b in spec.blocks:
            ho = conv_out(h, 3, b.stride, 1)
            d = dict(spec=b, hin=h, hout=ho)
            # din: the block input's gradient through conv1 (with the projection shortcut's gradient
            # fused in, for a downsampling block); din2: the identity shortcut's gradient
            for k in ("h1", "o1", "h2", "out", "dh2", "do1", "dh1", "din") + (() if b.proj else ("din2",)):
                d[k] = act(ho if k not in ("din", "din2") else h, b.cout if k not in ("din", "din2") else b.cin)
            if b.proj:
                d["hs"], d["sc"], d["dhs"] = act(ho, b.cout), act(ho, b.cout), act(ho, b.cout)
                d["gout"] = act(ho, b.cout)  # the masked output gradient, input of the shortcut BatchNorm
            for k in ("bn1", "bn2", "downbn"):
                d[k] = [vec(b.cout) for _ in range(4)]
                # the BatchNorm's per-CTA partial statistics from its convolution (dbl_conv_fwd_parts)
                d[k + ".parts"] = torch.empty(D.dbl_conv_stats_parts_bytes(D.conv_shape(1, 8, 8, 64, b.cout, 1, 1, 0))
                                              // 4, dtype=torch.float32, device=dev)
            self.blocks.append(d)
            h = ho
        self.final_hw = h
        self.dfeat = act(h, spec.widths[-1])
        self.grad = torch.zeros(spec.n_flat, dtype=torch.float32, device=dev)
        self.loss = torch.zeros(1, dtype=torch.float32, device=dev)
        self.labels = torch.zeros(B, dtype=torch.int32, device=dev)
        self.ws = torch.empty(self._ws_bytes(), dtype=torch.uint8, device=dev)

    # ------------------------------------------------------------------ shapes
    def conv_shapes(self):
        """(name, dbl_conv_shape) of every convolution of this worker, in forward order."""
        B, spec = self.batch, self.spec
        out = [(self.spec.stem.name, self.stem_shape())]
        for d in self.blocks:
            b = d["spec"]
            out.append((b.pre + ".conv1", D.conv_shape(B, d["hin"], d["hin"], b.cin, b.cout, 3, b.stride, 1)))
            out.append((b.pre + ".conv2", D.conv_shape(B, d["hout"], d["hout"], b.cout, b.cout, 3, 1, 1)))
            if b.proj:
                out.append((b.pre + ".down", D.conv_shape(B, d["hin"], d["hin"], b.cin, b.cout, 1, b.stride, 0)))
        return out

    def _ws_bytes(self):
        need = D.dbl_head_workspace_bytes(self.batch, self.spec.widths[-1], self.spec.classes)
        for _, s in self.conv_shapes():
            for ps in (D.DBL_PASS_FWD, D.DBL_PASS_DGRAD, D.DBL_PASS_WGRAD):
                need = max(need, D.dbl_conv_workspace_bytes(s, ps))
        for d in self.blocks:
            need = max(need, D.dbl_bn_workspace_bytes(D.bn_shape(self.batch * d["hout"] ** 2, d["spec"].cout)))
        need = max(need, D.dbl_bn_workspace_bytes(D.bn_shape(self.batch * self.stem_hw ** 2, self.spec.stem.cout)))
        return int(need) + 256

    def stem_shape(self):
        """The stem as a ceil(R/g) x 1 convolution of the unrolled input (StemLayout)."""
        st, lay = self.spec.stem, self.spec.stem_layout
        return D.conv_shape(self.batch, self.stem_rows, self.stem_hw, 64, st.cout, lay.taps, lay.conv_stride,
                            lay.conv_pad, s=1, stride_w=1, pad_w=0)

    def stem_prepare(self, images, native_res, stream):
        """Resize the native images (fp32 values, or uint8 pixels standardized with
        PIXEL_SCALE / PIXEL_BIAS) to this worker's resolution, in the stem's unrolled layout."""
        st, lay = self.spec.stem, self.spec.stem_layout
        if images.dtype == torch.uint8:
            D.dbl_progressive_resize_stem_u8(images, self.batch, native_res, native_res, 3, PIXEL_SCALE, PIXEL_BIAS,
                                             self.x0, self.res, self.res, st.r, st.stride, st.pad, lay.rg, lay.pad_h,
                                             self.stem_rows, stream)
        else:
            D.dbl_progressive_resize_stem(images, self.batch, native_res, native_res, 3, self.x0, self.res, self.res,
                                          st.r, st.stride, st.pad, lay.rg, lay.pad_h, self.stem_rows, stream)

    def stem_wgrad(self, dy, grad_w, ws, wsb, stream):
        """Stem weight gradient into grad_w (stored layout); rows past the filter stay zero."""
        st, lay = self.spec.stem, self.spec.stem_layout
        D.dbl_conv_wgrad(self.stem_shape(), self.x0, dy, grad_w, False, ws, wsb, stream)
        rows = lay.rg * lay.taps
        if rows > st.r:  # padding rows of the row-grouped layout: not filter weights
            k, per_row = grad_w.shape[0], grad_w[0, 0].numel()
            D.dbl_zero_f32_2d(grad_w[:, st.r:].data_ptr(), k, (rows - st.r) * per_row, rows * per_row, stream)

    def layer_flops(self, name, s):
        """Algorithmic FLOPs of one pass of a conv layer: 2*M*N*K over the unpadded problem
        (for the stem: R x R taps of 3 colour channels)."""
        st = self.spec.stem
        if name == st.name:
            return 2 * self.batch * self.stem_hw * self.stem_hw * st.cout * st.r * st.r * st.cin_logical
        P = conv_out(s.h, s.r, s.stride, s.pad)
        Q = conv_out(s.w, s.s, s.stride_w or s.stride, s.pad_w if s.stride_w else s.pad)
        return 2 * s.n * P * Q * s.k * s.r * s.s * s.c

    def conv_flops(self):
        """Algorithmic conv FLOPs of one step: forward + data gradient (not the stem) + weight gradient."""
        return sum(self.layer_flops(name, s) * (2 if name == self.spec.stem.name else 3)
                   for name, s in self.conv_shapes())

    # ------------------------------------------------------------------ the step
    def enqueue_step(self, server, images, native_res, stream):
        """Resize, forward, loss, backward; gradients land in self.grad (batch means, times the
        loss scale under loss scaling).

        images: fp32 [B, native_res, native_res, 3] (or uint8 pixels) on the device; labels in
        self.labels.  server: the model to compute on (a ServerState or a worker's pulled copy).
        """
        if server.precision != self.precision:
            raise ValueError(f"worker stores {self.precision}, the model's copy is {server.precision}")
        with D.precision(self.precision):
            if server.scaled:
                st = stream if isinstance(stream, torch.cuda.Stream) else torch.cuda.ExternalStream(stream)
                with torch.cuda.stream(st):
                    self.scale_used.copy_(server.scale_state[0:1].view(torch.float32))
            if self.pdl is not None:
                D.dbl_set_conv_pdl(1 if self.pdl else 0)
            try:
                self._enqueue_step(server, images, native_res, stream)
            finally:
                if self.pdl is not None:
                    D.dbl_set_conv_pdl(-1)

    def _enqueue_step(self, server, images, native_res, stream):
        spec, B, eps = self.spec, self.batch, self.eps
        s = stream.cuda_stream if hasattr(stream, "cuda_stream") else stream
        ws, wsb = self.ws, self.ws.numel()
        W16, W, G = server.w16, server.w, self.grad

        def wv(name):
            return spec.view(W16, name)

        def pv(name):
            return spec.view(W, name)

        def gv(name):
            return spec.view(G, name)

        st = spec.stem
        self.stem_prepare(images, native_res, s)
        # ---- forward
        shp = self.stem_shape()
        s_sum, s_sq, s_mean, s_istd = self.stem_stats
        D.dbl_conv_fwd(shp, self.x0, wv("conv1.w"), self.stem_y, s_sum, s_sq, ws, wsb, s)
        bns = D.bn_shape(B * self.stem_hw ** 2, st.cout, eps, True)
        if spec.variant == "imagenet":
            # BatchNorm + ReLU + max pool in one pass: the BatchNorm output is never stored (its
            # ReLU mask is recomputed in the backward pass)
            D.dbl_bn_relu_maxpool_fwd(bns, B, self.stem_hw, self.stem_hw, self.stem_y, s_sum, s_sq, pv("bn1.g"),
                                      pv("bn1.b"), s_mean, s_istd, self.pool_out, self.pool_arg, s)
            cur = self.pool_out
        else:
            D.dbl_bn_relu_fused(bns, self.stem_y, s_sum, s_sq, pv("bn1.g"), pv("bn1.b"), None, self.stem_a, s_mean,
                                s_istd, s)
            cur = self.stem_a
        for d in self.blocks:
            b = d["spec"]
            d["x"] = cur
            cnt = B * d["hout"] ** 2
            # each convolution leaves its BatchNorm statistics as per-CTA partials, which the
            # BatchNorm's finalize reduces (one launch per layer fewer than reducing them apart)
            s1 = D.conv_shape(B, d["hin"], d["hin"], b.cin, b.cout, 3, b.stride, 1)
            st1, p1 = d["bn1"], d["bn1.parts"]
            n1 = D.dbl_conv_fwd_parts(s1, cur, wv(b.pre + ".conv1.w"), d["h1"], p1, p1.numel() * 4, s)
            D.dbl_bn_relu_fused_parts(D.bn_shape(cnt, b.cout, eps, True), d["h1"], p1, n1, pv(b.pre + ".bn1.g"),
                                      pv(b.pre + ".bn1.b"), None, d["o1"], st1[2], st1[3], s)
            s2 = D.conv_shape(B, d["hout"], d["hout"], b.cout, b.cout, 3, 1, 1)
            st2, p2 = d["bn2"], d["bn2.parts"]
            n2 = D.dbl_conv_fwd_parts(s2, d["o1"], wv(b.pre + ".conv2.w"), d["h2"], p2, p2.numel() * 4, s)
            if b.proj:
                sd = D.conv_shape(B, d["hin"], d["hin"], b.cin, b.cout, 1, b.stride, 0)
                std, pd = d["downbn"], d["downbn.parts"]
                nd = D.dbl_conv_fwd_parts(sd, cur, wv(b.pre + ".down.w"), d["hs"], pd, pd.numel() * 4, s)
                D.dbl_bn_relu_fused_parts(D.bn_shape(cnt, b.cout, eps, False), d["hs"], pd, nd,
                                          pv(b.pre + ".downbn.g"), pv(b.pre + ".downbn.b"), None, d["sc"], std[2],
                                          std[3], s)
                res = d["sc"]
            else:
                res = cur
            D.dbl_bn_relu_fused_parts(D.bn_shape(cnt, b.cout, eps, True), d["h2"], p2, n2, pv(b.pre + ".bn2.g"),
                                      pv(b.pre + ".bn2.b"), res, d["out"], st2[2], st2[3], s)
            cur = d["out"]
        # ---- head: pooling, FC, softmax cross-entropy and their backward
        C = spec.widths[-1]
        if self.dropout > 0.0 or server.scaled:
            opts = D.head_opts(self.dropout, self.dropout_seed, self.dropout_step if self.dropout > 0.0 else None,
                               self.scale_used if server.scaled else None)
            D.dbl_head_fwd_bwd_ex(B, self.final_hw ** 2, C, spec.classes, cur, pv("fc.w"), pv("fc.b"), self.labels,
                                  opts, self.loss, gv("fc.w"), gv("fc.b"), self.dfeat, ws, wsb, s)
        else:
            D.dbl_head_fwd_bwd(B, self.final_hw ** 2, C, spec.classes, cur, pv("fc.w"), pv("fc.b"), self.labels,
                               self.loss, gv("fc.w"), gv("fc.b"), self.dfeat, ws, wsb, s)
        # ---- backward
        dout, dout2 = self.dfeat, None
        for d in reversed(self.blocks):
            b = d["spec"]
            cnt = B * d["hout"] ** 2
            st1, st2, std = d["bn1"], d["bn2"], d["downbn"]
            # g = (dout + dout2) * [out > 0] is kept: the identity shortcut's gradient, or the
            # projection shortcut BatchNorm's incoming gradient
            g = d["gout"] if b.proj else d["din2"]
            D.dbl_bn_relu_fused_bwd(D.bn_shape(cnt, b.cout, eps, True), dout, dout2, d["h2"], d["out"],
                                    pv(b.pre + ".bn2.g"), st2[2], st2[3], d["dh2"], g, gv(b.pre + ".bn2.g"),
                                    gv(b.pre + ".bn2.b"), ws, wsb, s)
            s2 = D.conv_shape(B, d["hout"], d["hout"], b.cout, b.cout, 3, 1, 1)
            D.dbl_conv_wgrad(s2, d["o1"], d["dh2"], gv(b.pre + ".conv2.w"), False, ws, wsb, s)
            D.dbl_conv_dgrad(s2, d["dh2"], wv(b.pre + ".conv2.w"), d["do1"], None, 0, s)
            # bn1 has no residual: its ReLU mask is recomputed from h1 (o1 is not read again)
            D.dbl_bn_relu_fused_bwd(D.bn_shape(cnt, b.cout, eps, True), d["do1"], None, d["h1"], None,
                                    pv(b.pre + ".bn1.g"), st1[2], st1[3], d["dh1"], None, gv(b.pre + ".bn1.g"),
                                    gv(b.pre + ".bn1.b"), ws, wsb, s, beta=pv(b.pre + ".bn1.b"))
            s1 = D.conv_shape(B, d["hin"], d["hin"], b.cin, b.cout, 3, b.stride, 1)
            D.dbl_conv_wgrad(s1, d["x"], d["dh1"], gv(b.pre + ".conv1.w"), False, ws, wsb, s)
            if b.proj:
                # the shortcut BatchNorm sees the same masked gradient g as bn2 (no ReLU of its own)
                D.dbl_bn_relu_fused_bwd(D.bn_shape(cnt, b.cout, eps, False), g, None, d["hs"], None,
                                        pv(b.pre + ".downbn.g"), std[2], std[3], d["dhs"], None,
                                        gv(b.pre + ".downbn.g"), gv(b.pre + ".downbn.b"), ws, wsb, s)
                sd = D.conv_shape(B, d["hin"], d["hin"], b.cin, b.cout, 1, b.stride, 0)
                D.dbl_conv_wgrad(sd, d["x"], d["dhs"], gv(b.pre + ".down.w"), False, ws, wsb, s)
                # the block input's gradient through conv1 and the projection, in one pass
                D.dbl_conv_dgrad_proj(s1, d["dh1"], wv(b.pre + ".conv1.w"), b.cout, d["dhs"], wv(b.pre + ".down.w"),
                                      d["din"], None, 0, s)
                dout, dout2 = d["din"], None
            else:
                D.dbl_conv_dgrad(s1, d["dh1"], wv(b.pre + ".conv1.w"), d["din"], None, 0, s)
                dout, dout2 = d["din"], d["din2"]
        bns = D.bn_shape(B * self.stem_hw ** 2, st.cout, eps, True)
        if spec.variant == "imagenet":
            D.dbl_maxpool_bwd(B, self.stem_hw, self.stem_hw, st.cout, dout, dout2, self.pool_arg, self.stem_da, s)
            D.dbl_bn_relu_fused_bwd(bns, self.stem_da, None, self.stem_y, None, pv("bn1.g"), s_mean, s_istd,
                                    self.stem_dy, None, gv("bn1.g"), gv("bn1.b"), ws, wsb, s, beta=pv("bn1.b"))
        else:
            D.dbl_bn_relu_fused_bwd(bns, dout, dout2, self.stem_y, None, pv("bn1.g"), s_mean, s_istd,
                                    self.stem_dy, None, gv("bn1.g"), gv("bn1.b"), ws, wsb, s, beta=pv("bn1.b"))
        self.stem_wgrad(self.stem_dy, gv("conv1.w"), ws, wsb, s)


def collect_pushes(done, deadline_s, wait, clock=time.monotonic):
    """The server's side of a deadline (host): ``done`` maps worker tags to their step
    events, in the order the server checks them; all share one deadline of ``deadline_s``
    seconds from the call.  ``wait(event, seconds)`` returns DBL_OK once the event has
    completed or DBL_ERR_TIMEOUT if it has not within the given seconds.  Returns
    (arrived, failed): lists of tags."""
    t0 = clock()
    arrived, failed = [], []
    for tag, ev in done.items():
        left = max(0.0, deadline_s - (clock() - t0))
        rc = wait(ev, left)
        if rc == D.DBL_OK:
            arrived.append(tag)
        elif rc == D.DBL_ERR_TIMEOUT:
            failed.append(tag)
        else:
            raise D.DblError(rc, f"waiting for worker {tag}")
    return arrived, failed


class DualBatchIteration:
    """One parameter-server iteration of the hybrid scheme on one GPU.

    The large-batch worker runs on stream L and the small-batch worker on
    stream S, concurrently; the merge (Sec. 3.4) runs on stream L once both
    have pushed, in the arrival order given by ``order``.  Either worker may be
    None (a single push).  ``capture()`` records the iteration as a CUDA graph.
    """

    def __init__(self, server, large, small, native_res, lr=0.2, momentum=0.9, f_large=1.0, f_small=19.0 / 21.0,
                 order=0):
        self.server, self.large, self.small = server, large, small
        self.native_res = native_res
        self.lr, self.momentum, self.f_large, self.f_small, self.order = lr, momentum, f_large, f_small, order
        self.stream_l = torch.cuda.Stream()
        self.stream_s = torch.cuda.Stream()
        self.images_l = self.images_s = None
        self.graph = None
        self._inputs_ready = None  # copy-stream event the next run() waits for
        self._consumed = None      # compute-stream event: the last run() has read its inputs

    def set_inputs(self, images_l, labels_l, images_s=None, labels_s=None, non_blocking=False, stream=None):
        """Images at the native resolution (fp32 values, or uint8 pixels) and int32 labels
        (device or pinned host tensors), copied into the iteration's device buffers.  Without ``stream`` the
        copies go on the current stream.  With a (copy) ``stream`` they are issued there
        once the previous run() has consumed the buffers, and the next run() waits for
        them, so that host-to-device copies overlap the compute of other iterations."""
        dev = self.server.w.device
        for have, new_t in ((self.images_l, images_l), (self.images_s, images_s)):
            if self.graph is not None and have is not None and new_t is not None and have.dtype != new_t.dtype:
                raise ValueError("set_inputs: the captured graph reads images of another dtype")
        cs = stream if stream is not None else torch.cuda.current_stream()
        if stream is not None and self._consumed is not None:
            stream.wait_event(self._consumed)
        with torch.cuda.stream(cs):
            if self.large is not None:
                if self.images_l is None or self.images_l.dtype != images_l.dtype:
                    self.images_l = torch.empty(images_l.shape, dtype=images_l.dtype, device=dev)
                self.images_l.copy_(images_l, non_blocking=non_blocking)
                self.large.labels.copy_(labels_l, non_blocking=non_blocking)
            if self.small is not None:
                if self.images_s is None or self.images_s.dtype != images_s.dtype:
                    self.images_s = torch.empty(images_s.shape, dtype=images_s.dtype, device=dev)
                self.images_s.copy_(images_s, non_blocking=non_blocking)
                self.small.labels.copy_(labels_s, non_blocking=non_blocking)
        if stream is not None:
            self._inputs_ready = torch.cuda.Event()
            self._inputs_ready.record(stream)

    def losses_to_host(self, out):
        """Queue the workers' losses (large, then small) into ``out`` (pinned host fp32)
        on the current stream; read them after that stream has passed this point."""
        workers = [w for w in (self.large, self.small) if w is not None]
        for i, w in enumerate(workers):
            out[i:i + 1].copy_(w.loss, non_blocking=True)
        return len(workers)

    def _enqueue(self):
        cur = torch.cuda.current_stream()
        sL, sS = self.stream_l, self.stream_s
        sL.wait_stream(cur)
        sS.wait_stream(cur)
        if self.large is not None:
            self.large.enqueue_step(self.server, self.images_l, self.native_res, sL)
        if self.small is not None:
            self.small.enqueue_step(self.server, self.images_s, self.native_res, sS)
        sL.wait_stream(sS)  # the server applies the pushes once both have arrived
        self._merge(["L", "S"], sL)
        cur.wait_stream(sL)

    def _merge(self, tags, stream):
        wl = self.large if "L" in tags else None
        ws_ = self.small if "S" in tags else None
        self.server.apply_pushes(wl.grad if wl else None, ws_.grad if ws_ else None,
                                 wl.scale_used if wl else None, ws_.scale_used if ws_ else None, self.lr,
                                 self.momentum, self.f_large, self.f_small, self.order, stream.cuda_stream)

    def run(self):
        cur = torch.cuda.current_stream()
        if self._inputs_ready is not None:
            cur.wait_event(self._inputs_ready)
            self._inputs_ready = None
        if self.graph is not None:
            self.graph.replay()
        else:
            self._enqueue()
        self._consumed = torch.cuda.Event()
        self._consumed.record(cur)

    def run_with_deadline(self, deadline_s, wait=None):
        """One iteration in which the server waits at most ``deadline_s`` seconds of host time
        (counted from when both workers' steps are enqueued) for the pushes, and merges those
        that arrived: under ASP the server does not wait for a worker that has stopped
        (Sec. 2.4).  A worker whose step has not completed by then is reported failed and its
        push is left out of this iteration; its stream finishes in its own time, and the next
        iteration's steps queue behind it.  Runs eagerly, not as the captured graph.
        Returns (status, failed): (DBL_OK, []) when every worker pushed, otherwise
        (DBL_ERR_TIMEOUT, tags) with the tags ('L', 'S') of the workers that missed the
        deadline.  ``wait(event, seconds) -> status`` defaults to ``dbl_event_wait``.
        Run the iteration once (``run`` or ``capture``) before the first call: the first launch
        of a kernel loads it, and loading waits for every stream, a stalled one included."""
        wait = wait or D.dbl_event_wait
        cur = torch.cuda.current_stream()
        if self._inputs_ready is not None:
            cur.wait_event(self._inputs_ready)
            self._inputs_ready = None
        done = {}
        for tag, wk, st, img in (("L", self.large, self.stream_l, self.images_l),
                                 ("S", self.small, self.stream_s, self.images_s)):
            if wk is None:
                continue
            st.wait_stream(cur)
            wk.enqueue_step(self.server, img, self.native_res, st)
            ev = torch.cuda.Event()
            ev.record(st)
            done[tag] = ev
        arrived, failed = collect_pushes(done, deadline_s, wait)
        if arrived:
            for tag in arrived:
                cur.wait_event(done[tag])
            self._merge(arrived, cur)
        self._consumed = torch.cuda.Event()
        self._consumed.record(cur)
        return (D.DBL_OK if not failed else D.DBL_ERR_TIMEOUT), failed

    def capture(self):
        """Record one iteration (both workers, the join and the merge) as a CUDA graph."""
        self._enqueue()  # warm-up outside capture: kernel attributes, lazy loading
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            with torch.cuda.graph(g, stream=s):
                self._enqueue()
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        self.graph = g
        return g

    def images_per_iteration(self):
        return (self.large.batch if self.large else 0) + (self.small.batch if self.small else 0)
