"""GPU parity of each C-ABI kernel against the fp64 oracle, on seeded inputs
that both sides see identically (bf16-rounded where the GPU reads bf16).

Tolerances (max|gpu - ref| / max|ref|): 1e-2 for bf16-input / fp32-accumulate
convolutions and the bf16 outputs of BatchNorm and the head; 1e-6 for the
fp32 merge; resize taps bit-exact and values within one bf16 ulp.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from conftest import max_norm_rel
from gpu_common import bf16_values, check_status, host, load_dbl, rng, stem_fold, to_bf16_dev, to_f32_dev, ws

pytestmark = pytest.mark.gpu

CONV_TOL = 1e-2
# fp32 weight gradients: the products of two bf16 values are exact in fp32, so the only error
# against the fp64 oracle is that of fp32 summation (relative ~1e-6 at these sizes)
WGRAD_TOL = 1e-4
MERGE_TOL = 1e-6


@pytest.fixture(scope="module")
def D():
    return load_dbl()


# ----------------------------------------------------------------------------- merge
@pytest.mark.parametrize("n", [36_864, 1_001, 11_220_132])
@pytest.mark.parametrize("order", [0, 1, 2])
def test_merge_matches_oracle(D, n, order):
    g = rng(n + order)
    w0 = g.standard_normal(n).astype(np.float32)
    u0 = (0.01 * g.standard_normal(n)).astype(np.float32)
    gl = (0.1 * g.standard_normal(n)).astype(np.float32)
    gs = (0.1 * g.standard_normal(n)).astype(np.float32)
    w, u, gL, gS = (to_f32_dev(a) for a in (w0, u0, gl, gs))
    w16 = torch.empty(n, dtype=torch.bfloat16, device="cuda")
    D.dbl_ps_dual_batch_merge(w, u, w16, gL, gS, n, 0.2, 0.9, 1.0, 19 / 21, order)
    rw, ru = orc.ps_merge(w0, u0, gl, gs, 0.2, 0.9, 1.0, 19 / 21, order)
    assert max_norm_rel(host(w), rw) <= MERGE_TOL
    assert max_norm_rel(host(u), ru) <= MERGE_TOL
    # the pulled copy is the bf16 rounding of the new fp32 master weights
    assert torch.equal(w16, w.to(torch.bfloat16))
    check_status(D)


def test_merge_single_push_and_no_w16(D):
    n = 4099
    g = rng(7)
    w0, u0, gl = (g.standard_normal(n).astype(np.float32) for _ in range(3))
    w, u, gL = to_f32_dev(w0), to_f32_dev(u0), to_f32_dev(gl)
    D.dbl_ps_dual_batch_merge(w, u, None, gL, None, n, 0.1, 0.9, 1.0, 0.5, 0)
    rw, ru = orc.ps_merge(w0, u0, gl, None, 0.1, 0.9, 1.0, 0.5, 0)
    assert max_norm_rel(host(w), rw) <= MERGE_TOL
    assert max_norm_rel(host(u), ru) <= MERGE_TOL


# ----------------------------------------------------------------------------- resize
@pytest.mark.parametrize("n,hin,hout", [(3, 32, 16), (3, 32, 24), (2, 32, 32), (2, 224, 128), (2, 224, 160),
                                        (1, 17, 5)])
def test_resize_matches_oracle(D, n, hin, hout):
    x = rng(hin + hout).standard_normal((n, hin, hin, 3)).astype(np.float32)
    ref = orc.bilinear_resize(x, hout, hout)
    xd = to_f32_dev(x)
    out = torch.full((n, hout, hout, 8), 7.0, dtype=torch.bfloat16, device="cuda")
    D.dbl_progressive_resize(xd, D.DBL_F32, n, hin, hin, 3, out, D.DBL_BF16, hout, hout, 8)
    got = host(out)
    assert np.all(got[..., 3:] == 0.0)
    # within one bf16 ulp of the exact value
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(ref), 1e-30))) - 7)
    assert np.all(np.abs(got[..., :3] - ref) <= ulp + 1e-30)
    out32 = torch.empty((n, hout, hout, 3), dtype=torch.float32, device="cuda")
    D.dbl_progressive_resize(xd, D.DBL_F32, n, hin, hin, 3, out32, D.DBL_F32, hout, hout, 3)
    assert max_norm_rel(host(out32), ref) <= 1e-6


def _stem_layout(r, st, pad):
    from paper_2509_26092_gb300.resnet18 import ConvSpec, StemLayout
    return StemLayout.of(ConvSpec("conv1", 64, 3, 64, r, st, pad))


@pytest.mark.parametrize("n,hin,hout,r,st,pad", [(2, 224, 160, 7, 2, 3), (3, 32, 24, 3, 1, 1), (2, 224, 224, 7, 2, 3),
                                                 (1, 20, 13, 7, 2, 3)])
def test_resize_stem_unrolls_the_resized_image(D, n, hin, hout, r, st, pad):
    lay = _stem_layout(r, st, pad)
    x = rng(hin + hout + r).standard_normal((n, hin, hin, 3)).astype(np.float32)
    ref = orc.bilinear_resize(x, hout, hout)
    P = (hout + 2 * pad - r) // st + 1
    rows = lay.rows(hout, P)
    out = torch.full((n, rows, P, 64), 7.0, dtype=torch.bfloat16, device="cuda")
    D.dbl_progressive_resize_stem(to_f32_dev(x), n, hin, hin, 3, out, hout, hout, r, st, pad, lay.rg, lay.pad_h, rows)
    xu = host(out).reshape(n, rows, P, lay.rg, 8, 8 // lay.rg)
    assert np.all(xu[..., r:, :] == 0.0)      # taps past the filter width
    assert np.all(xu[..., 3:] == 0.0)         # padded colour channels
    for q in range(P):                        # columns outside the image
        for t in range(r):
            if not 0 <= q * st + t - pad < hout:
                assert np.all(xu[:, :, q, :, t, :] == 0.0)
    for m in range(rows):                     # rows outside the image
        for e in range(lay.rg):
            if not 0 <= lay.rg * m + e - lay.pad_h < hout:
                assert np.all(xu[:, m, :, e] == 0.0)
    got = stem_fold(xu, r, st, pad, hout, lay.rg, lay.pad_h)[..., :3]
    covered = ~np.isnan(got[0, :, :, 0])
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(ref), 1e-30))) - 7)
    assert np.all(np.abs(got[:, covered] - ref[:, covered]) <= ulp[:, covered] + 1e-30)
    check_status(D)


@pytest.mark.parametrize("n,hin,hout,r,st,pad", [
    (2, 224, 160, 7, 2, 3), (2, 224, 128, 7, 2, 3), (1, 288, 160, 7, 2, 3), (2, 224, 224, 7, 2, 3),
    (3, 40, 40, 7, 2, 3),
    (3, 32, 24, 3, 1, 1), (2, 32, 32, 3, 1, 1)])           # the CIFAR stem's layout (one row per position)
def test_resize_stem_from_8bit_pixels(D, n, hin, hout, r, st, pad):
    """8-bit pixels standardized on the GPU: the same bits as the fp32 path on pixels
    standardized on the host with the same two fp32 operations, and the oracle's resize."""
    from paper_2509_26092_gb300.resnet18 import PIXEL_BIAS, PIXEL_SCALE
    lay = _stem_layout(r, st, pad)
    u8 = rng(hin + 5).integers(0, 256, size=(n, hin, hin, 3), dtype=np.uint8)
    x32 = u8.astype(np.float32) * np.asarray(PIXEL_SCALE, np.float32) + np.asarray(PIXEL_BIAS, np.float32)
    P = (hout + 2 * pad - r) // st + 1
    rows = lay.rows(hout, P)
    a = torch.empty((n, rows, P, 64), dtype=torch.bfloat16, device="cuda")
    b = torch.empty_like(a)
    D.dbl_progressive_resize_stem_u8(torch.from_numpy(u8).cuda(), n, hin, hin, 3, PIXEL_SCALE, PIXEL_BIAS, a, hout,
                                     hout, r, st, pad, lay.rg, lay.pad_h, rows)
    D.dbl_progressive_resize_stem(to_f32_dev(x32), n, hin, hin, 3, b, hout, hout, r, st, pad, lay.rg, lay.pad_h, rows)
    assert torch.equal(a, b)
    ref = orc.bilinear_resize(x32.astype(np.float64), hout, hout)
    got = stem_fold(host(a).reshape(n, rows, P, lay.rg, 8, 8 // lay.rg), r, st, pad, hout, lay.rg, lay.pad_h)[..., :3]
    covered = ~np.isnan(got[0, :, :, 0])
    # one bf16 ulp of the value, plus the fp32 rounding of interpolating O(1) inputs (values near zero)
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(ref), 1e-30))) - 7)
    assert np.all(np.abs(got[:, covered] - ref[:, covered]) <= ulp[:, covered] + 1e-6)
    check_status(D)


STEM_CASES = [  # n, h (square input), r, stride, pad
    (2, 20, 7, 2, 3),    # ImageNet stem on a small image
    (3, 10, 3, 1, 1),    # CIFAR stem
    (4, 64, 7, 2, 3),    # several tiles
    (2, 224, 7, 2, 3),   # full size: window tiles of two 112-wide rows, two-row weight-gradient K-blocks
    (1, 160, 7, 2, 3),   # tiles of three 80-wide rows
    (1, 288, 7, 2, 3),   # the paper's 288 px sub-stage: 144-wide rows
]


def _stem_inputs(n, h, r, seed, lay):
    g = rng(seed)
    x = bf16_values(g.standard_normal((n, h, h, 3)))
    wt = bf16_values(g.standard_normal((64, r, r, 3)) * np.sqrt(2.0 / (r * r * 3)))
    w_store = np.zeros((64, lay.rg * lay.taps, 8, 8 // lay.rg))
    w_store[:, :r, :r, :3] = wt
    return x, wt, w_store


@pytest.mark.parametrize("case", STEM_CASES)
def test_unrolled_stem_fwd_and_wgrad_match_oracle(D, case):
    n, h, r, st, pad = case
    lay = _stem_layout(r, st, pad)
    x, wt, w_store = _stem_inputs(n, h, r, 21, lay)
    P = (h + 2 * pad - r) // st + 1
    rows = lay.rows(h, P)
    xu = torch.empty((n, rows, P, 64), dtype=torch.bfloat16, device="cuda")
    D.dbl_progressive_resize_stem(to_f32_dev(x), n, h, h, 3, xu, h, h, r, st, pad, lay.rg, lay.pad_h,
                                  rows)  # same size: exact copy
    shape = D.conv_shape(n, rows, P, 64, 64, lay.taps, lay.conv_stride, lay.conv_pad, s=1, stride_w=1, pad_w=0)
    y = torch.full((n, P, P, 64), float("nan"), dtype=torch.bfloat16, device="cuda")
    s1, s2 = torch.empty(64, device="cuda"), torch.empty(64, device="cuda")
    wsb = max(D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_FWD), D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_WGRAD))
    D.dbl_conv_fwd(shape, xu, to_bf16_dev(w_store), y, s1, s2, ws(wsb), wsb)
    ref = orc.conv2d_fwd(x, wt, st, pad)
    assert max_norm_rel(host(y), ref) <= CONV_TOL
    dy = bf16_values(rng(22).standard_normal((n, P, P, 64)))
    dw = torch.full(w_store.shape, float("nan"), device="cuda")
    D.dbl_conv_wgrad(shape, xu, to_bf16_dev(dy), dw, False, ws(wsb), wsb)
    rows_w = lay.rg * lay.taps
    if rows_w > r:  # the padding rows of the row-grouped layout: zeroed as the worker does
        per = 8 * (8 // lay.rg)
        D.dbl_zero_f32_2d(dw[:, r:].data_ptr(), 64, (rows_w - r) * per, rows_w * per)
    got = host(dw)
    assert np.all(got[:, :, r:, :] == 0.0) and np.all(got[..., 3:] == 0.0)  # padding gets no gradient
    assert np.all(got[:, r:] == 0.0)
    rdw = orc.conv2d_wgrad(x, dy, wt.shape, st, pad)
    assert max_norm_rel(got[:, :r, :r, :3], rdw) <= WGRAD_TOL
    check_status(D)


# ----------------------------------------------------------------------------- BatchNorm
@pytest.mark.parametrize("count,C,relu,res", [(4096, 64, True, True), (1000, 128, True, False),
                                              (777, 512, False, False), (2048, 256, True, True)])
def test_bn_fwd_bwd_match_oracle(D, count, C, relu, res):
    g = rng(count + C)
    y = bf16_values(g.standard_normal((count, C)) * 2.0 + 0.5)
    r = bf16_values(g.standard_normal((count, C))) if res else None
    gamma = (1.0 + 0.2 * g.standard_normal(C)).astype(np.float32)
    beta = (0.1 * g.standard_normal(C)).astype(np.float32)
    yd = to_bf16_dev(y)
    s1 = torch.empty(C, device="cuda")
    s2 = torch.empty(C, device="cuda")
    shape = D.bn_shape(count, C, 1e-5, relu)
    D.dbl_bn_stats(shape, yd, s1, s2)
    np.testing.assert_allclose(host(s1), y.sum(0), rtol=1e-4, atol=1e-2)
    out = torch.empty((count, C), dtype=torch.bfloat16, device="cuda")
    mean = torch.empty(C, device="cuda")
    istd = torch.empty(C, device="cuda")
    D.dbl_bn_relu_fused(shape, yd, s1, s2, to_f32_dev(gamma), to_f32_dev(beta), to_bf16_dev(r) if res else None, out,
                        mean, istd)
    ro, rm, ri = orc.bn_fwd(y, gamma, beta, 1e-5, res=r, relu=relu)
    assert max_norm_rel(host(out), ro) <= CONV_TOL
    np.testing.assert_allclose(host(mean), rm, rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(host(istd), ri, rtol=1e-4)
    # backward, with a second upstream gradient
    dout = bf16_values(g.standard_normal((count, C)))
    dout2 = bf16_values(g.standard_normal((count, C)))
    out_h = host(out)
    dy = torch.empty_like(out)
    dres = torch.empty_like(out)
    dg = torch.empty(C, device="cuda")
    db = torch.empty(C, device="cuda")
    wsb = D.dbl_bn_workspace_bytes(shape)
    D.dbl_bn_relu_fused_bwd(shape, to_bf16_dev(dout), to_bf16_dev(dout2), yd, out, to_f32_dev(gamma), mean, istd, dy,
                            dres, dg, db, ws(wsb), wsb)
    rdy, rdg, rdb, rdres = orc.bn_bwd(dout, out_h, y, gamma, host(mean), host(istd), relu=relu, dout2=dout2,
                                      want_dres=True)
    assert max_norm_rel(host(dy), rdy) <= CONV_TOL
    assert max_norm_rel(host(dg), rdg) <= 1e-4
    assert max_norm_rel(host(db), rdb) <= 1e-4
    assert max_norm_rel(host(dres), rdres) <= CONV_TOL
    if relu and not res:
        # without a residual the ReLU mask can be recomputed from y instead of read from out:
        # the same decisions as the forward pass, so the same bits
        dy2, dres2 = torch.empty_like(out), torch.empty_like(out)
        dg2, db2 = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
        D.dbl_bn_relu_fused_bwd(shape, to_bf16_dev(dout), to_bf16_dev(dout2), yd, None, to_f32_dev(gamma), mean, istd,
                                dy2, dres2, dg2, db2, ws(wsb), wsb, beta=to_f32_dev(beta))
        assert torch.equal(dy2, dy) and torch.equal(dres2, dres) and torch.equal(dg2, dg) and torch.equal(db2, db)
    check_status(D)


@pytest.mark.parametrize("n,H,W,C,coarse", [(3, 20, 18, 64, False), (2, 21, 17, 64, False), (1, 112, 112, 64, False),
                                            (2, 14, 14, 128, False), (2, 30, 26, 8, True), (16, 112, 112, 64, True),
                                            (4, 48, 48, 2048, False)])
def test_bn_relu_maxpool_equals_bn_then_maxpool(D, n, H, W, C, coarse):
    """The fused stem pass equals the BatchNorm pass followed by the max pool, bit for bit.

    Odd sizes clip windows at the bottom and right; 8 channels make one channel group a
    window; 16 x 112 x 112 has more windows than the grid, so threads step on through the
    batch; coarse inputs sit on a grid of quarters, so windows hold exact positive ties."""
    g = rng(77)
    y = g.standard_normal((n, H, W, C)) * 2.0 + 0.3
    if coarse:
        y = np.round(y * 4.0) / 4.0
    y = bf16_values(y)
    gamma = (1.0 + 0.2 * g.standard_normal(C)).astype(np.float32)
    beta = (0.1 * g.standard_normal(C)).astype(np.float32)
    yd, gd, bd = to_bf16_dev(y), to_f32_dev(gamma), to_f32_dev(beta)
    shape = D.bn_shape(n * H * W, C, 1e-5, True)
    s1, s2 = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
    D.dbl_bn_stats(shape, yd, s1, s2)
    P, Q = (H - 1) // 2 + 1, (W - 1) // 2 + 1
    out = torch.empty((n, H, W, C), dtype=torch.bfloat16, device="cuda")
    m1, i1, m2, i2 = (torch.empty(C, device="cuda") for _ in range(4))
    D.dbl_bn_relu_fused(shape, yd, s1, s2, gd, bd, None, out, m1, i1)
    y1 = torch.empty((n, P, Q, C), dtype=torch.bfloat16, device="cuda")
    a1 = torch.empty((n, P, Q, C), dtype=torch.uint8, device="cuda")
    D.dbl_maxpool_fwd(n, H, W, C, out, y1, a1)
    y2, a2 = torch.empty_like(y1), torch.empty_like(a1)
    D.dbl_bn_relu_maxpool_fwd(shape, n, H, W, yd, s1, s2, gd, bd, m2, i2, y2, a2)
    assert torch.equal(y1, y2) and torch.equal(a1, a2) and torch.equal(m1, m2) and torch.equal(i1, i2)
    check_status(D)


# ----------------------------------------------------------------------------- max pool
@pytest.mark.parametrize("n,h,w,c,zeros", [(2, 9, 10, 64, False), (2, 16, 16, 64, True), (1, 112, 112, 64, True)])
def test_maxpool_matches_oracle(D, n, h, w, c, zeros):
    g = rng(h * w + c)
    x = g.standard_normal((n, h, w, c))
    if zeros:  # post-ReLU-like input: many exact ties at zero
        x = np.maximum(x, 0.0)
    x = bf16_values(x)
    ry, rarg = orc.maxpool_fwd(x, 3, 2, 1)
    P, Q = ry.shape[1], ry.shape[2]
    y = torch.empty((n, P, Q, c), dtype=torch.bfloat16, device="cuda")
    arg = torch.empty((n, P, Q, c), dtype=torch.uint8, device="cuda")
    xd = to_bf16_dev(x)
    D.dbl_maxpool_fwd(n, h, w, c, xd, y, arg)
    np.testing.assert_array_equal(host(y), ry)
    np.testing.assert_array_equal(arg.cpu().numpy().astype(np.int32), rarg)
    dy = bf16_values(g.standard_normal(ry.shape))
    dy2 = bf16_values(g.standard_normal(ry.shape))
    dx = torch.empty_like(xd)
    D.dbl_maxpool_bwd(n, h, w, c, to_bf16_dev(dy), to_bf16_dev(dy2), arg, dx)
    rdx = orc.maxpool_bwd(dy + dy2, rarg, x.shape, 3, 2, 1)
    assert max_norm_rel(host(dx), rdx) <= CONV_TOL


@pytest.mark.parametrize("n,h,w,c", [(2, 9, 10, 64), (3, 13, 16, 128), (16, 112, 112, 64)])
def test_maxpool_bwd_equals_fp32_window_order_gather(D, n, h, w, c):
    """The max-pool gradient is, bit for bit, the fp32 sum from zero of each input pixel's
    window gradients (dy + dy2 in fp32) in (p, q) window order, rounded to bf16 once; odd
    sizes clip windows, and 16 x 112 x 112 has more 2x2 blocks than the grid."""
    g = rng(n * h + c)
    x = np.maximum(g.standard_normal((n, h, w, c)), 0.0)  # ties at zero
    xd = to_bf16_dev(bf16_values(x))
    P, Q = (h - 1) // 2 + 1, (w - 1) // 2 + 1
    y = torch.empty((n, P, Q, c), dtype=torch.bfloat16, device="cuda")
    arg = torch.empty((n, P, Q, c), dtype=torch.uint8, device="cuda")
    D.dbl_maxpool_fwd(n, h, w, c, xd, y, arg)
    dy = to_bf16_dev(bf16_values(g.standard_normal((n, P, Q, c))))
    dy2 = to_bf16_dev(bf16_values(g.standard_normal((n, P, Q, c))))
    dx = torch.empty_like(xd)
    D.dbl_maxpool_bwd(n, h, w, c, dy, dy2, arg, dx)
    f = torch.nn.functional.pad(dy.float() + dy2.float(), (0, 0, 0, 1, 0, 1))
    a = torch.nn.functional.pad(arg.int(), (0, 0, 0, 1, 0, 1), value=255)
    ref = torch.empty_like(dx)
    for dh in range(2):
        for dw in range(2):
            acc = torch.zeros((n, P, Q, c), device="cuda")
            for dp in range(2):
                for dq in range(2):
                    r, s = dh - 2 * dp + 1, dw - 2 * dq + 1
                    if 0 <= r <= 2 and 0 <= s <= 2:
                        win = (slice(None), slice(dp, dp + P), slice(dq, dq + Q))
                        acc = acc + torch.where(a[win] == 3 * r + s, f[win], torch.zeros_like(acc))
            ref[:, dh::2, dw::2] = acc[:, : (h - dh + 1) // 2, : (w - dw + 1) // 2].to(torch.bfloat16)
    assert torch.equal(dx, ref)
    check_status(D)


# ----------------------------------------------------------------------------- head
@pytest.mark.parametrize("n,hw,c,classes", [(4, 16, 64, 10), (8, 49, 512, 1000), (256, 16, 512, 100),
                                            (512, 49, 512, 1000), (128, 49, 512, 1000)])  # the two worker batches
def test_head_matches_oracle(D, n, hw, c, classes):
    g = rng(n * classes)
    x = bf16_values(np.maximum(g.standard_normal((n, hw, c)), 0))
    W = (0.05 * g.standard_normal((classes, c))).astype(np.float32)
    b = (0.01 * g.standard_normal(classes)).astype(np.float32)
    lab = g.integers(0, classes, n).astype(np.int32)
    loss = torch.empty(1, device="cuda")
    dW = torch.empty((classes, c), device="cuda")
    db = torch.empty(classes, device="cuda")
    dx = torch.empty((n, hw, c), dtype=torch.bfloat16, device="cuda")
    wsb = D.dbl_head_workspace_bytes(n, c, classes)
    D.dbl_head_fwd_bwd(n, hw, c, classes, to_bf16_dev(x), to_f32_dev(W), to_f32_dev(b),
                       torch.from_numpy(lab).cuda(), loss, dW, db, dx, ws(wsb), wsb)
    x4 = x.reshape(n, 1, hw, c)
    feat = orc.avgpool_fwd(x4)
    logits = orc.fc_fwd(feat, W, b)
    rl, dl = orc.softmax_ce(logits, lab)
    rdW, rdb, rdf = orc.fc_bwd(dl, feat, W)
    rdx = orc.avgpool_bwd(rdf, x4.shape).reshape(n, hw, c)
    assert abs(loss.item() - rl) <= 1e-5 * abs(rl)
    assert max_norm_rel(host(dW), rdW) <= 1e-4
    assert max_norm_rel(host(db), rdb) <= 1e-4
    assert max_norm_rel(host(dx), rdx) <= CONV_TOL


@pytest.mark.parametrize("n,hw,c,classes,rate", [(6, 4, 64, 10, 0.3), (128, 49, 512, 1000, 0.1),
                                                 (37, 16, 512, 100, 0.2)])
def test_head_dropout_matches_oracle(D, n, hw, c, classes, rate):
    """Dropout before the FC layer: the mask bit for bit against the oracle's Philox draw,
    the head's outputs against the oracle applying that mask, the step counter advanced by
    one per call, and a second call drawing a new mask."""
    g = rng(n + classes)
    x = bf16_values(np.maximum(g.standard_normal((n, hw, c)), 0))
    W = (0.05 * g.standard_normal((classes, c))).astype(np.float32)
    b = (0.01 * g.standard_normal(classes)).astype(np.float32)
    lab = g.integers(0, classes, n).astype(np.int32)
    d = float(np.float32(rate))  # the rate as the fp32 value the library receives
    seed, step0 = 0x9E3779B97F4A7C15 ^ n, 5
    step = torch.tensor([step0], dtype=torch.int64, device="cuda")
    keep = torch.empty((n, c), dtype=torch.uint8, device="cuda")
    D.dbl_dropout_mask(n, c, rate, seed, step, keep)
    rkeep = orc.dropout_mask(n, c, d, seed, step0)
    torch.cuda.synchronize()
    assert np.array_equal(keep.cpu().numpy(), rkeep)
    loss = torch.empty(1, device="cuda")
    dW = torch.empty((classes, c), device="cuda")
    db = torch.empty(classes, device="cuda")
    dx = torch.empty((n, hw, c), dtype=torch.bfloat16, device="cuda")
    wsb = D.dbl_head_workspace_bytes(n, c, classes)
    work = ws(wsb)
    xd, Wd, bd, labd = to_bf16_dev(x), to_f32_dev(W), to_f32_dev(b), torch.from_numpy(lab).cuda()
    opts = D.head_opts(rate, seed, step)
    D.dbl_head_fwd_bwd_ex(n, hw, c, classes, xd, Wd, bd, labd, opts, loss, dW, db, dx, work, wsb)
    x4 = x.reshape(n, 1, hw, c)
    feat = orc.dropout_apply(orc.avgpool_fwd(x4), rkeep, d)
    logits = orc.fc_fwd(feat, W, b)
    rl, dl = orc.softmax_ce(logits, lab)
    rdW, rdb, rdf = orc.fc_bwd(dl, feat, W)
    rdx = orc.avgpool_bwd(orc.dropout_apply(rdf, rkeep, d), x4.shape).reshape(n, hw, c)
    assert int(step.item()) == step0 + 1
    assert abs(loss.item() - rl) <= 1e-5 * abs(rl)
    assert max_norm_rel(host(dW), rdW) <= 1e-4
    assert max_norm_rel(host(db), rdb) <= 1e-4
    assert max_norm_rel(host(dx), rdx) <= CONV_TOL
    dropped = np.broadcast_to((rkeep == 0)[:, None, :], (n, hw, c))
    assert np.all(host(dx)[dropped] == 0.0)  # a dropped feature passes no gradient back
    # the next call draws the mask of step 6
    D.dbl_head_fwd_bwd_ex(n, hw, c, classes, xd, Wd, bd, labd, opts, loss, dW, db, dx, work, wsb)
    rkeep6 = orc.dropout_mask(n, c, d, seed, step0 + 1)
    feat6 = orc.dropout_apply(orc.avgpool_fwd(x4), rkeep6, d)
    rl6, _ = orc.softmax_ce(orc.fc_fwd(feat6, W, b), lab)
    assert int(step.item()) == step0 + 2 and not np.array_equal(rkeep6, rkeep)
    assert abs(loss.item() - rl6) <= 1e-5 * abs(rl6)


def test_head_dropout_rate_zero_is_the_plain_head(D):
    n, hw, c, classes = 9, 16, 64, 10
    g = rng(3)
    x = to_bf16_dev(bf16_values(np.maximum(g.standard_normal((n, hw, c)), 0)))
    W, b = to_f32_dev(0.05 * g.standard_normal((classes, c))), to_f32_dev(0.01 * g.standard_normal(classes))
    lab = torch.from_numpy(g.integers(0, classes, n).astype(np.int32)).cuda()
    wsb = D.dbl_head_workspace_bytes(n, c, classes)
    outs = []
    for drop in (False, True):
        o = (torch.empty(1, device="cuda"), torch.empty((classes, c), device="cuda"), torch.empty(classes, device="cuda"),
             torch.empty((n, hw, c), dtype=torch.bfloat16, device="cuda"))
        if drop:
            D.dbl_head_fwd_bwd_ex(n, hw, c, classes, x, W, b, lab, D.head_opts(0.0, 1), *o, ws(wsb), wsb)
        else:
            D.dbl_head_fwd_bwd(n, hw, c, classes, x, W, b, lab, *o, ws(wsb), wsb)
        outs.append(o)
    torch.cuda.synchronize()
    for a, b_ in zip(*outs):
        assert torch.equal(a, b_)
    with pytest.raises(D.DblError):
        D.dbl_head_fwd_bwd_ex(n, hw, c, classes, x, W, b, lab, D.head_opts(1.0, 1), *outs[0], ws(wsb), wsb)


# ----------------------------------------------------------------------------- convolutions
FWD_CASES = [  # n, h, w, c, k, r, stride, pad
    (2, 8, 8, 64, 64, 3, 1, 1),      # exactly one 128-row tile
    (3, 7, 9, 64, 128, 3, 1, 1),     # ragged last tile, BN = 128
    (2, 8, 8, 128, 64, 3, 2, 1),     # stride 2, two channel blocks
    (2, 8, 8, 64, 128, 1, 2, 0),     # 1x1 stride-2 projection
    (8, 16, 16, 64, 64, 3, 1, 1),    # the single-block workload (batch 8, 16x16)
    (2, 6, 6, 8, 64, 3, 1, 1),       # CIFAR stem, 8 padded channels
    (2, 20, 20, 8, 64, 7, 2, 3),     # ImageNet stem, 8 padded channels
    (1, 4, 4, 256, 256, 3, 1, 1),    # deep layer, small image, 256-wide tile
    (4, 14, 14, 256, 512, 3, 2, 1),  # two 256-wide column tiles, stride 2
    (32, 56, 56, 64, 64, 3, 1, 1),   # 784 tiles: every persistent CTA loops over several
    # 256-wide tiles on CTA pairs (M = 256 across two SMs, half of B in each)
    (32, 14, 14, 256, 256, 3, 1, 1),  # 24.5 pair tiles: the second CTA of the last pair has no rows
    (64, 14, 14, 256, 512, 3, 2, 1),  # stride 2, two column tiles, several tiles per pair
    # 3x3 stride-1 window kernel: strips of zero-padded rows, taps as shifted descriptors
    (4, 28, 28, 128, 128, 3, 1, 1),  # streamed 128-wide weight tiles, two channel blocks
    (5, 5, 13, 128, 64, 3, 1, 1),    # streamed 64-wide tiles; a tile spans several small images
    (1, 3, 254, 64, 64, 3, 1, 1),    # widest padded row a copy can carry (256 pixels)
]


def _conv_inputs(case, seed):
    n, h, w, c, k, r, st, pad = case
    g = rng(seed)
    x = g.standard_normal((n, h, w, c))
    if c == 8:
        x[..., 3:] = 0.0  # 3 colour channels padded to 8
    wt = g.standard_normal((k, r, r, c)) * np.sqrt(2.0 / (r * r * c))
    return bf16_values(x), bf16_values(wt)


@pytest.mark.parametrize("case", FWD_CASES)
def test_conv_fwd_matches_oracle(D, case):
    n, h, w, c, k, r, st, pad = case
    x, wt = _conv_inputs(case, 11)
    ref = orc.conv2d_fwd(x, wt, st, pad)
    P, Q = ref.shape[1], ref.shape[2]
    shape = D.conv_shape(n, h, w, c, k, r, st, pad)
    y = torch.full((n, P, Q, k), float("nan"), dtype=torch.bfloat16, device="cuda")
    s1 = torch.empty(k, device="cuda")
    s2 = torch.empty(k, device="cuda")
    wsb = D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_FWD)
    D.dbl_conv_fwd(shape, to_bf16_dev(x), to_bf16_dev(wt), y, s1, s2, ws(wsb), wsb)
    got = host(y)
    assert np.all(np.isfinite(got))
    assert max_norm_rel(got, ref) <= CONV_TOL
    # channel statistics are those of the stored outputs
    flat = got.reshape(-1, k)
    np.testing.assert_allclose(host(s1), flat.sum(0), rtol=1e-4, atol=1e-3 * np.abs(flat).max())
    np.testing.assert_allclose(host(s2), (flat ** 2).sum(0), rtol=1e-4, atol=1e-3)
    check_status(D)


_PAIR64_IN_CHILD = r"""
import sys, torch, numpy as np
sys.path.insert(0, sys.argv[1])
from paper_2509_26092_gb300 import build_lib
build_lib.build()
from paper_2509_26092_gb300 import dbl as D
cases = [(32, 56, 56), (3, 7, 9), (2, 8, 8)]
out = []
for i, (n, h, w) in enumerate(cases):
    shape = D.conv_shape(n, h, w, 64, 64, 3, 1, 1)
    assert D.dbl_conv_plan(shape, D.DBL_PASS_FWD).ctas_per_mma == int(sys.argv[3])
    g = np.random.default_rng(100 + i)
    x = torch.from_numpy(g.standard_normal((n, h, w, 64)).astype(np.float32)).cuda().to(torch.bfloat16)
    wt = torch.from_numpy((0.05 * g.standard_normal((64, 3, 3, 64))).astype(np.float32)).cuda().to(torch.bfloat16)
    y = torch.full((n, h, w, 64), float("nan"), dtype=torch.bfloat16, device="cuda")
    s1, s2 = torch.empty(64, device="cuda"), torch.empty(64, device="cuda")
    wsb = D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_FWD)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    D.dbl_conv_fwd(shape, x, wt, y, s1, s2, ws, wsb)
    out.append((y.cpu(), s1.cpu(), s2.cpu()))
torch.cuda.synchronize()
assert D.dbl_device_status() == D.DBL_OK
torch.save(out, sys.argv[2])
"""


def test_window_pairs_of_64_columns_give_the_same_outputs(tmp_path):
    """The 64-column window forward pass on CTA pairs (DBL_CONV_CTA_PAIRS=2, read once per process,
    hence child processes; M = 256 MMAs across two SMs, half of the resident weights in each) stores
    the same bits and channel sums as on single CTAs, on tiles that fill pairs, leave the second
    CTA of the last pair without a tile, and span several small images."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    got = {}
    for level, cg in (("1", "1"), ("2", "2")):
        path = str(tmp_path / f"y{level}.pt")
        r = subprocess.run([sys.executable, "-c", _PAIR64_IN_CHILD, root, path, cg], capture_output=True, text=True,
                           timeout=600, env=dict(os.environ, DBL_CONV_CTA_PAIRS=level))
        assert r.returncode == 0, r.stderr[-2000:]
        got[level] = torch.load(path)
    for a, b in zip(got["1"], got["2"]):
        assert torch.isfinite(a[0].float()).all()
        for t1, t2 in zip(a, b):
            assert torch.equal(t1, t2)


@pytest.mark.parametrize("case", [(2, 8, 8, 64, 64, 3, 1, 1), (4, 14, 14, 256, 512, 3, 2, 1), (32, 14, 14, 256, 256, 3, 1, 1),
                                  (8, 16, 16, 64, 128, 3, 1, 1), (2, 8, 8, 64, 128, 1, 2, 0)])
def test_conv_fwd_parts_then_bn_matches_two_step_path(D, case):
    """Statistics left as per-CTA partials and reduced in the BatchNorm finalize give
    the same bits as dbl_conv_fwd's own reduction followed by dbl_bn_relu_fused."""
    n, h, w, c, k, r, st, pad = case
    x, wt = _conv_inputs(case, 21)
    shape = D.conv_shape(n, h, w, c, k, r, st, pad)
    P, Q = orc.out_dim(h, r, st, pad), orc.out_dim(w, r, st, pad)
    xd, wd = to_bf16_dev(x), to_bf16_dev(wt)
    y1 = torch.empty((n, P, Q, k), dtype=torch.bfloat16, device="cuda")
    y2 = torch.empty_like(y1)
    s1, s2 = torch.empty(k, device="cuda"), torch.empty(k, device="cuda")
    wsb = D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_FWD)
    D.dbl_conv_fwd(shape, xd, wd, y1, s1, s2, ws(wsb), wsb)
    pb = D.dbl_conv_stats_parts_bytes(shape)
    parts = torch.empty(pb // 4, device="cuda")
    nparts = D.dbl_conv_fwd_parts(shape, xd, wd, y2, parts, pb)
    assert nparts >= 1 and torch.equal(y1, y2)
    g = rng(22)
    gamma = to_f32_dev(g.uniform(0.5, 1.5, k).astype(np.float32))
    beta = to_f32_dev((0.1 * g.standard_normal(k)).astype(np.float32))
    res = to_bf16_dev(bf16_values(g.standard_normal((n, P, Q, k))))
    bs = D.bn_shape(n * P * Q, k, 1e-5, True)
    outs = []
    for use_parts in (False, True):
        out = torch.empty_like(y1)
        mean, istd = torch.empty(k, device="cuda"), torch.empty(k, device="cuda")
        if use_parts:
            D.dbl_bn_relu_fused_parts(bs, y2, parts, nparts, gamma, beta, res, out, mean, istd)
        else:
            D.dbl_bn_relu_fused(bs, y1, s1, s2, gamma, beta, res, out, mean, istd)
        outs.append((out, mean, istd))
    for a, b in zip(outs[0], outs[1]):
        assert torch.equal(a, b)
    # and both are the oracle's BatchNorm of the stored y
    ref, _, _ = orc.bn_fwd(host(y1), host(gamma), host(beta), 1e-5, res=host(res))
    assert max_norm_rel(host(outs[1][0]), ref) <= CONV_TOL
    check_status(D)


DGRAD_CASES = [
    (2, 8, 8, 64, 64, 3, 1, 1),
    (3, 6, 10, 64, 64, 3, 1, 1),     # ragged
    (2, 8, 8, 128, 64, 3, 2, 1),     # stride-2 phases, BN = 128
    (2, 8, 8, 64, 128, 1, 2, 0),     # 1x1 stride 2: three phases are all zero
    (2, 16, 16, 64, 128, 3, 2, 1),
    (1, 4, 4, 256, 256, 3, 1, 1),
    (2, 8, 8, 512, 512, 3, 1, 1),    # 256-wide tiles, 8 channel blocks of dy
    (16, 28, 28, 128, 128, 3, 1, 1), # many tiles per CTA
    (24, 14, 14, 256, 256, 3, 1, 1), # CTA pairs, ragged last pair tile
    (6, 28, 28, 256, 512, 3, 2, 1),  # CTA pairs over stride-2 phases (4, 2, 2, 1 taps)
    (8, 28, 28, 128, 256, 3, 2, 1),  # 128-wide tiles over stride-2 phases
    (5, 5, 13, 64, 128, 3, 1, 1),    # window kernel, 64-wide streamed tiles over two dy channel blocks
    (2, 9, 30, 64, 64, 3, 1, 1),     # window kernel, resident flipped weights, non-square image
]


@pytest.mark.parametrize("case", DGRAD_CASES)
def test_conv_dgrad_matches_oracle(D, case):
    n, h, w, c, k, r, st, pad = case
    x, wt = _conv_inputs(case, 12)
    P, Q = orc.out_dim(h, r, st, pad), orc.out_dim(w, r, st, pad)
    dy = bf16_values(rng(13).standard_normal((n, P, Q, k)))
    ref = orc.conv2d_dgrad(dy, wt, x.shape, st, pad)
    shape = D.conv_shape(n, h, w, c, k, r, st, pad)
    dx = torch.full((n, h, w, c), float("nan"), dtype=torch.bfloat16, device="cuda")
    D.dbl_conv_dgrad(shape, to_bf16_dev(dy), to_bf16_dev(wt), dx)
    got = host(dx)
    assert np.all(np.isfinite(got))
    assert max_norm_rel(got, ref) <= CONV_TOL
    check_status(D)


@pytest.mark.parametrize("n,h,c,k,k2", [(2, 8, 64, 128, 128), (3, 14, 128, 256, 256), (4, 14, 256, 512, 512),
                                        (2, 10, 64, 128, 64)])
def test_conv_dgrad_with_projection_matches_oracle(D, n, h, c, k, k2):
    """Block-input gradient of a downsampling block: the 3x3 stride-2 convolution's data
    gradient plus that of the 1x1 stride-2 projection shortcut, in one pass."""
    g = rng(n * 1000 + c)
    x = bf16_values(g.standard_normal((n, h, h, c)))
    wt = bf16_values(g.standard_normal((k, 3, 3, c)) * np.sqrt(2.0 / (9 * c)))
    w2 = bf16_values(g.standard_normal((k2, 1, 1, c)) * np.sqrt(2.0 / c))
    P = h // 2
    dy = bf16_values(g.standard_normal((n, P, P, k)))
    dy2 = bf16_values(g.standard_normal((n, P, P, k2)))
    ref = orc.conv2d_dgrad(dy, wt, x.shape, 2, 1) + orc.conv2d_dgrad(dy2, w2, x.shape, 2, 0)
    shape = D.conv_shape(n, h, h, c, k, 3, 2, 1)
    dx = torch.full((n, h, h, c), float("nan"), dtype=torch.bfloat16, device="cuda")
    D.dbl_conv_dgrad_proj(shape, to_bf16_dev(dy), to_bf16_dev(wt), k2, to_bf16_dev(dy2), to_bf16_dev(w2), dx)
    got = host(dx)
    assert np.all(np.isfinite(got))
    assert max_norm_rel(got, ref) <= CONV_TOL
    # the odd rows and columns carry the main term only
    ref_main = orc.conv2d_dgrad(dy, wt, x.shape, 2, 1)
    assert max_norm_rel(got[:, 1::2, :, :], ref_main[:, 1::2, :, :]) <= CONV_TOL
    check_status(D)


WGRAD_CASES = [
    (2, 8, 8, 64, 64, 3, 1, 1),
    (5, 7, 7, 64, 64, 3, 1, 1),      # ragged pixel count
    (2, 8, 8, 128, 64, 3, 2, 1),
    (2, 8, 8, 64, 128, 1, 2, 0),
    (2, 6, 6, 8, 64, 3, 1, 1),       # CIFAR stem
    (2, 20, 20, 8, 64, 7, 2, 3),     # ImageNet stem
    (1, 4, 4, 256, 256, 3, 1, 1),
    (8, 16, 16, 64, 64, 3, 1, 1),
    (2, 8, 8, 256, 512, 3, 2, 1),    # 256-wide tiles
    (16, 28, 28, 128, 128, 3, 1, 1), # split-K slices reduced in order
    (16, 14, 14, 256, 256, 3, 1, 1), # CTA pairs: 9 pair tiles of 256 (tap, c) rows, split-K
    (8, 7, 7, 512, 512, 3, 1, 1),    # CTA pairs, two column tiles
    (1, 3, 3, 64, 64, 3, 1, 1),      # a single slice, written straight into dw
    # window weight gradient (64 -> 64, 3x3 stride 1): x and dy strips, five tap-pair accumulators
    (32, 56, 56, 64, 64, 3, 1, 1),   # the layer1 shape at batch 32: one K-range per CTA
    (3, 5, 30, 64, 64, 3, 1, 1),     # K-blocks spanning several small non-square images
]


@pytest.mark.parametrize("case", WGRAD_CASES)
def test_conv_wgrad_matches_oracle(D, case):
    n, h, w, c, k, r, st, pad = case
    x, wt = _conv_inputs(case, 14)
    P, Q = orc.out_dim(h, r, st, pad), orc.out_dim(w, r, st, pad)
    dy = bf16_values(rng(15).standard_normal((n, P, Q, k)))
    ref = orc.conv2d_wgrad(x, dy, wt.shape, st, pad)
    shape = D.conv_shape(n, h, w, c, k, r, st, pad)
    wsb = D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_WGRAD)
    dw = torch.full((k, r, r, c), float("nan"), dtype=torch.float32, device="cuda")
    xd, dyd = to_bf16_dev(x), to_bf16_dev(dy)
    D.dbl_conv_wgrad(shape, xd, dyd, dw, False, ws(wsb), wsb)
    got = host(dw)
    assert np.all(np.isfinite(got))
    assert max_norm_rel(got, ref) <= WGRAD_TOL
    # accumulate mode adds onto what is there
    D.dbl_conv_wgrad(shape, xd, dyd, dw, True, ws(wsb), wsb)
    assert max_norm_rel(host(dw), 2 * ref) <= WGRAD_TOL
    check_status(D)
