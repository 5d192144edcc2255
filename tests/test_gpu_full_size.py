"""The step's kernels at the full sizes the bench times: the 224 px layers of the
ImageNet-shaped ResNet-18 at the large worker's batch of 512, and the 288 px layers
of the paper's last ImageNet sub-stage at its batch of 740, through the same
library calls and launch configurations as the training step.

Convolutions (window kernels, the 128-column window tiles and the 256-column tiles
on CTA pairs, phase-split stride-2 data gradients, split-K weight gradients): the
oracle computes sampled outputs one by one in fp64 from the same inputs, the corners
of every output tensor always among them; tolerance max-norm relative 1e-2 over the
samples.  A layer1 BatchNorm: the oracle over the whole tensor.  The stem's pool at
batch 512: the fused forward equals the two-step path and the gradient equals the
fp32 window-order gather, bit for bit."""
import numpy as np
import pytest
import torch

import oracle as orc
from gpu_common import check_status, load_dbl, rng, ws

pytestmark = pytest.mark.gpu

TOL = 1e-2
SAMPLES = 40

SHAPES = [  # n, h, w, c, k, r, stride, pad
    (512, 56, 56, 64, 64, 3, 1, 1),    # layer1: window kernels, window weight gradient
    (512, 56, 56, 64, 128, 3, 2, 1),   # layer2.0.conv1: stride 2, phase-split data gradient
    (512, 28, 28, 128, 128, 3, 1, 1),  # layer2: 128-column window tiles on CTA pairs
    (512, 14, 14, 256, 256, 3, 1, 1),  # layer3: 256-column tiles on CTA pairs
    (512, 7, 7, 512, 512, 3, 1, 1),    # layer4: two 256-column tiles
    (512, 56, 56, 64, 128, 1, 2, 0),   # layer2.0.down: 1x1 stride-2 projection
    # the paper's 288 px ImageNet sub-stage (Table 9) at its large-batch worker's batch of 740
    (740, 72, 72, 64, 64, 3, 1, 1),    # layer1
    (740, 72, 72, 64, 128, 3, 2, 1),   # layer2.0.conv1
    (740, 36, 36, 128, 128, 3, 1, 1),  # layer2
    (740, 18, 18, 256, 256, 3, 1, 1),  # layer3
    (740, 9, 9, 512, 512, 3, 1, 1),    # layer4: 59,940 rows, a ragged last tile
    (740, 18, 18, 256, 512, 1, 2, 0),  # layer4.0.down
]


def _bf16(shape, g, scale=1.0):
    """Seeded normal values on the bf16 grid: (fp64 host array, bf16 device tensor)."""
    a = torch.from_numpy(g.standard_normal(shape, dtype=np.float32) * np.float32(scale)).to(torch.bfloat16)
    return a.double().numpy(), a.cuda()


def _indices(shape, g):
    """SAMPLES index tuples into shape: the two extreme corners, then uniform draws."""
    idx = [tuple(0 for _ in shape), tuple(d - 1 for d in shape)]
    while len(idx) < SAMPLES:
        idx.append(tuple(int(g.integers(0, d)) for d in shape))
    return idx


def _check(got, ref, what, tol=TOL):
    got, ref = np.asarray(got, dtype=np.float64), np.asarray(ref, dtype=np.float64)
    err = float(np.max(np.abs(got - ref))) / max(float(np.max(np.abs(ref))), 1e-30)
    assert err <= tol, f"{what}: sampled max-norm relative error {err:.3e}"


@pytest.mark.parametrize("case", SHAPES)
def test_conv_passes_at_full_size(case):
    D = load_dbl()
    n, h, w, c, k, r, st, pad = case
    P, Q = orc.out_dim(h, r, st, pad), orc.out_dim(w, r, st, pad)
    g = rng(1000 + c + k + r)
    x64, xd = _bf16((n, h, w, c), g)
    w64, wd = _bf16((k, r, r, c), g, scale=(2.0 / (r * r * c)) ** 0.5)
    dy64, dyd = _bf16((n, P, Q, k), g)
    shape = D.conv_shape(n, h, w, c, k, r, st, pad)
    s = torch.cuda.current_stream()
    # forward, with the BatchNorm channel sums as in the step
    y = torch.empty((n, P, Q, k), dtype=torch.bfloat16, device="cuda")
    s1, s2 = torch.empty(k, device="cuda"), torch.empty(k, device="cuda")
    wsb = D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_FWD)
    D.dbl_conv_fwd(shape, xd, wd, y, s1, s2, ws(wsb), wsb, s)
    # data gradient
    dx = torch.empty_like(xd)
    wsb = D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_DGRAD)
    D.dbl_conv_dgrad(shape, dyd, wd, dx, ws(wsb), wsb, s)
    # weight gradient (split-K slices reduced in a fixed order)
    dw = torch.empty((k, r, r, c), dtype=torch.float32, device="cuda")
    wsb = D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_WGRAD)
    D.dbl_conv_wgrad(shape, xd, dyd, dw, False, ws(wsb), wsb, s)
    torch.cuda.synchronize()
    check_status(D)
    yh, dxh, dwh = y.float().cpu().numpy(), dx.float().cpu().numpy(), dw.cpu().numpy()
    fwd = _indices((n, P, Q, k), g)
    _check([yh[i] for i in fwd], [orc.conv2d_fwd_at(x64, w64, st, pad, *i) for i in fwd], f"{case} fwd")
    dg = _indices((n, h, w, c), g)
    _check([dxh[i] for i in dg], [orc.conv2d_dgrad_at(dy64, w64, x64.shape, st, pad, *i) for i in dg], f"{case} dgrad")
    wg = _indices((k, r, r, c), g)
    # fp32 weight gradient: exact bf16 products, fp32 sums of up to 3.6 M terms
    _check([dwh[i] for i in wg], [orc.conv2d_wgrad_at(x64, dy64, w64.shape, st, pad, *i) for i in wg], f"{case} wgrad",
           1e-3)


def test_batchnorm_at_full_size():
    """A layer1 BatchNorm with residual and ReLU at batch 512 (1.6 M rows x 64 channels), forward
    and backward with two upstream gradients, against the oracle over the whole tensor."""
    from conftest import max_norm_rel
    D = load_dbl()
    count, C = 512 * 56 * 56, 64
    g = rng(2024)
    y64, yd = _bf16((count, C), g, scale=2.0)
    r64, rd = _bf16((count, C), g)
    gamma = (1.0 + 0.2 * g.standard_normal(C)).astype(np.float32)
    beta = (0.1 * g.standard_normal(C)).astype(np.float32)
    gd, bd = torch.from_numpy(gamma).cuda(), torch.from_numpy(beta).cuda()
    shape = D.bn_shape(count, C, 1e-5, True)
    s1, s2 = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
    D.dbl_bn_stats(shape, yd, s1, s2)
    out = torch.empty_like(yd)
    mean, istd = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
    D.dbl_bn_relu_fused(shape, yd, s1, s2, gd, bd, rd, out, mean, istd)
    do64, dod = _bf16((count, C), g)
    do264, do2d = _bf16((count, C), g)
    dy, dres = torch.empty_like(yd), torch.empty_like(yd)
    dg, db = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
    wsb = D.dbl_bn_workspace_bytes(shape)
    D.dbl_bn_relu_fused_bwd(shape, dod, do2d, yd, out, gd, mean, istd, dy, dres, dg, db, ws(wsb), wsb)
    torch.cuda.synchronize()
    check_status(D)
    ro, rm, ri = orc.bn_fwd(y64, gamma, beta, 1e-5, res=r64, relu=True)
    assert max_norm_rel(out.double().cpu().numpy(), ro) <= TOL
    np.testing.assert_allclose(mean.cpu().numpy(), rm, rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(istd.cpu().numpy(), ri, rtol=1e-4)
    rdy, rdg, rdb, rdres = orc.bn_bwd(do64, out.double().cpu().numpy(), y64, gamma, mean.double().cpu().numpy(),
                                      istd.double().cpu().numpy(), relu=True, dout2=do264, want_dres=True)
    assert max_norm_rel(dy.double().cpu().numpy(), rdy) <= TOL
    assert max_norm_rel(dres.double().cpu().numpy(), rdres) <= TOL
    assert max_norm_rel(dg.double().cpu().numpy(), rdg) <= 1e-4
    assert max_norm_rel(db.double().cpu().numpy(), rdb) <= 1e-4


def test_stem_pool_at_full_size():
    """The stem's fused BatchNorm + ReLU + max pool at batch 512 (112 x 112 x 64) equals the
    BatchNorm pass followed by the max pool bit for bit, and the pool gradient equals the fp32
    window-order gather of the two upstream gradients."""
    D = load_dbl()
    n, H, C = 512, 112, 64
    P = (H - 1) // 2 + 1
    gen = torch.Generator(device="cuda").manual_seed(7)
    x = (torch.randn((n, H, H, C), device="cuda", generator=gen) * 2.0 + 0.3).to(torch.bfloat16)
    shape = D.bn_shape(n * H * H, C, 1e-5, True)
    s1, s2 = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
    D.dbl_bn_stats(shape, x, s1, s2)
    gd = (1.0 + 0.2 * torch.randn(C, device="cuda", generator=gen)).float()
    bd = (0.1 * torch.randn(C, device="cuda", generator=gen)).float()
    m1, i1, m2, i2 = (torch.empty(C, device="cuda") for _ in range(4))
    a = torch.empty_like(x)
    D.dbl_bn_relu_fused(shape, x, s1, s2, gd, bd, None, a, m1, i1)
    y1 = torch.empty((n, P, P, C), dtype=torch.bfloat16, device="cuda")
    a1 = torch.empty((n, P, P, C), dtype=torch.uint8, device="cuda")
    D.dbl_maxpool_fwd(n, H, H, C, a, y1, a1)
    del a
    y2, a2 = torch.empty_like(y1), torch.empty_like(a1)
    D.dbl_bn_relu_maxpool_fwd(shape, n, H, H, x, s1, s2, gd, bd, m2, i2, y2, a2)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2) and torch.equal(a1, a2) and torch.equal(m1, m2) and torch.equal(i1, i2)
    dp = torch.randn((n, P, P, C), device="cuda", generator=gen).to(torch.bfloat16)
    dp2 = torch.randn((n, P, P, C), device="cuda", generator=gen).to(torch.bfloat16)
    dx = torch.empty_like(x)
    D.dbl_maxpool_bwd(n, H, H, C, dp, dp2, a2, dx)
    torch.cuda.synchronize()
    check_status(D)
    f = torch.nn.functional.pad(dp.float() + dp2.float(), (0, 0, 0, 1, 0, 1))
    am = torch.nn.functional.pad(a2.int(), (0, 0, 0, 1, 0, 1), value=255)
    for dh in range(2):
        for dw in range(2):
            acc = torch.zeros((n, P, P, C), device="cuda")
            for dpp in range(2):
                for dq in range(2):
                    r, s = dh - 2 * dpp + 1, dw - 2 * dq + 1
                    if 0 <= r <= 2 and 0 <= s <= 2:
                        win = (slice(None), slice(dpp, dpp + P), slice(dq, dq + P))
                        acc = acc + torch.where(am[win] == 3 * r + s, f[win], torch.zeros_like(acc))
            assert torch.equal(dx[:, dh::2, dw::2], acc.to(torch.bfloat16)), (dh, dw)


@pytest.mark.parametrize("case", [(740, 72, 72, 64, 64, 3, 1, 1), (740, 18, 18, 256, 256, 3, 1, 1),
                                  (512, 56, 56, 64, 128, 3, 2, 1)])
def test_conv_passes_at_full_size_in_fp16(case):
    """The same passes from the binary16-storage build (the paper's mixed precision) at full size:
    the 288 px sub-stage's layer1 and layer3 at batch 740 and layer2.0.conv1 at batch 512."""
    D = load_dbl()
    n, h, w, c, k, r, st, pad = case
    P, Q = orc.out_dim(h, r, st, pad), orc.out_dim(w, r, st, pad)
    g = rng(2000 + c + k + r)

    def f16(shape, scale=1.0):
        a = torch.from_numpy(g.standard_normal(shape, dtype=np.float32) * np.float32(scale)).to(torch.float16)
        return a.double().numpy(), a.cuda()

    x64, xd = f16((n, h, w, c))
    w64, wd = f16((k, r, r, c), (2.0 / (r * r * c)) ** 0.5)
    dy64, dyd = f16((n, P, Q, k))
    shape = D.conv_shape(n, h, w, c, k, r, st, pad)
    with D.precision("f16"):
        y = torch.empty((n, P, Q, k), dtype=torch.float16, device="cuda")
        s1, s2 = torch.empty(k, device="cuda"), torch.empty(k, device="cuda")
        wsb = max(D.dbl_conv_workspace_bytes(shape, p) for p in (D.DBL_PASS_FWD, D.DBL_PASS_WGRAD))
        work = ws(wsb)
        D.dbl_conv_fwd(shape, xd, wd, y, s1, s2, work, wsb)
        dx = torch.empty_like(xd)
        D.dbl_conv_dgrad(shape, dyd, wd, dx, None, 0)
        dw = torch.empty((k, r, r, c), dtype=torch.float32, device="cuda")
        D.dbl_conv_wgrad(shape, xd, dyd, dw, False, work, wsb)
        torch.cuda.synchronize()
        check_status(D)
    yh, dxh, dwh = y.double().cpu().numpy(), dx.double().cpu().numpy(), dw.double().cpu().numpy()
    fwd = _indices((n, P, Q, k), g)
    _check([yh[i] for i in fwd], [orc.conv2d_fwd_at(x64, w64, st, pad, *i) for i in fwd], f"{case} fwd", 2e-3)
    dg = _indices((n, h, w, c), g)
    _check([dxh[i] for i in dg], [orc.conv2d_dgrad_at(dy64, w64, x64.shape, st, pad, *i) for i in dg], f"{case} dgrad",
           2e-3)
    wg = _indices((k, r, r, c), g)
    _check([dwh[i] for i in wg], [orc.conv2d_wgrad_at(x64, dy64, w64.shape, st, pad, *i) for i in wg], f"{case} wgrad",
           1e-3)

