"""fp16 mixed precision with loss scaling (the paper's ImageNet runs, Sec. 5.2.3) on the GPU:
the library built with IEEE binary16 storage (libdbl_f16.so), checked against the fp64 oracle
on inputs rounded to binary16, and the loss-scaling pieces (the scaled head, the finiteness
check, the scaled merge with its skip rule, the dynamic scale) against the oracle's rules.

Tolerances: convolutions and BatchNorm outputs stored in binary16 (11-bit significand, a
relative rounding step of 2^-11) are held to max-norm relative 2e-3, five times tighter than
the bf16 tests' 1e-2; fp32 statistics and sums to 1e-4; the merge to 1e-6.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from conftest import max_norm_rel
from gpu_common import load_dbl, rng, ws

pytestmark = pytest.mark.gpu

F16_TOL = 2e-3


@pytest.fixture(scope="module")
def D():
    return load_dbl()


def f16_values(a):
    """The float64 values of a after rounding to binary16 (what both sides see)."""
    return np.asarray(a, dtype=np.float64).astype(np.float16).astype(np.float64)


def dev16(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64).astype(np.float16)).cuda()


def dev32(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def host(t):
    return t.detach().double().cpu().numpy()


CONV_CASES = [  # n, h, w, c, k, r, stride, pad: one of each kernel family the step uses
    (2, 20, 20, 64, 64, 3, 1, 1),     # window kernel, 64 columns, resident weights
    (4, 28, 28, 128, 128, 3, 1, 1),   # window kernel, 128 columns on CTA pairs
    (4, 14, 14, 256, 512, 3, 2, 1),   # implicit GEMM, 256 columns on CTA pairs, stride 2 (phase-split dgrad)
    (2, 8, 8, 64, 128, 1, 2, 0),      # 1x1 stride-2 projection
    (32, 14, 14, 256, 256, 3, 1, 1),  # several pair tiles per CTA pair
]


@pytest.mark.parametrize("case", CONV_CASES)
def test_conv_passes_in_fp16_match_oracle(D, case):
    n, h, w, c, k, r, st, pad = case
    g = rng(500 + c + k)
    x = f16_values(g.standard_normal((n, h, w, c)))
    wt = f16_values(g.standard_normal((k, r, r, c)) * np.sqrt(2.0 / (r * r * c)))
    P, Q = orc.out_dim(h, r, st, pad), orc.out_dim(w, r, st, pad)
    dy = f16_values(g.standard_normal((n, P, Q, k)))
    shape = D.conv_shape(n, h, w, c, k, r, st, pad)
    with D.precision("f16"):
        xd, wd, dyd = dev16(x), dev16(wt), dev16(dy)
        y = torch.full((n, P, Q, k), float("nan"), dtype=torch.float16, device="cuda")
        s1, s2 = torch.empty(k, device="cuda"), torch.empty(k, device="cuda")
        wsb = max(D.dbl_conv_workspace_bytes(shape, p) for p in (D.DBL_PASS_FWD, D.DBL_PASS_WGRAD))
        work = ws(wsb)
        D.dbl_conv_fwd(shape, xd, wd, y, s1, s2, work, wsb)
        dx = torch.full_like(xd, float("nan"))
        D.dbl_conv_dgrad(shape, dyd, wd, dx, None, 0)
        dw = torch.empty((k, r, r, c), device="cuda")
        D.dbl_conv_wgrad(shape, xd, dyd, dw, False, work, wsb)
        torch.cuda.synchronize()
        assert D.dbl_device_status() == D.DBL_OK
    assert max_norm_rel(host(y), orc.conv2d_fwd(x, wt, st, pad)) <= F16_TOL
    flat = host(y).reshape(-1, k)  # BatchNorm sums are those of the stored fp16 outputs
    np.testing.assert_allclose(host(s1), flat.sum(0), rtol=1e-4, atol=1e-3 * np.abs(flat).max())
    assert max_norm_rel(host(dx), orc.conv2d_dgrad(dy, wt, x.shape, st, pad)) <= F16_TOL
    assert max_norm_rel(host(dw), orc.conv2d_wgrad(x, dy, wt.shape, st, pad)) <= 1e-4


def test_batchnorm_in_fp16_matches_oracle(D):
    count, C = 3001, 128
    g = rng(77)
    y = f16_values(g.standard_normal((count, C)) * 2.0 + 0.5)
    r = f16_values(g.standard_normal((count, C)))
    gamma = (1.0 + 0.2 * g.standard_normal(C)).astype(np.float32)
    beta = (0.1 * g.standard_normal(C)).astype(np.float32)
    shape = D.bn_shape(count, C, 1e-5, True)
    with D.precision("f16"):
        yd = dev16(y)
        s1, s2 = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
        D.dbl_bn_stats(shape, yd, s1, s2)
        out = torch.empty((count, C), dtype=torch.float16, device="cuda")
        mean, istd = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
        D.dbl_bn_relu_fused(shape, yd, s1, s2, dev32(gamma), dev32(beta), dev16(r), out, mean, istd)
        dout = f16_values(g.standard_normal((count, C)))
        dy, dres = torch.empty_like(out), torch.empty_like(out)
        dg, db = torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
        wsb = D.dbl_bn_workspace_bytes(shape)
        D.dbl_bn_relu_fused_bwd(shape, dev16(dout), None, yd, out, dev32(gamma), mean, istd, dy, dres, dg, db, ws(wsb),
                                wsb)
        torch.cuda.synchronize()
    ro, rm, ri = orc.bn_fwd(y, gamma, beta, 1e-5, res=r, relu=True)
    assert max_norm_rel(host(out), ro) <= F16_TOL
    np.testing.assert_allclose(host(mean), rm, rtol=1e-5, atol=1e-5)
    rdy, rdg, rdb, rdres = orc.bn_bwd(dout, host(out), y, gamma, host(mean), host(istd), relu=True, want_dres=True)
    assert max_norm_rel(host(dy), rdy) <= F16_TOL
    assert max_norm_rel(host(dres), rdres) <= F16_TOL
    assert max_norm_rel(host(dg), rdg) <= 1e-4 and max_norm_rel(host(db), rdb) <= 1e-4


def test_max_pool_in_fp16_is_exact(D):
    n, H, C = 3, 17, 64
    g = rng(5)
    x = f16_values(np.maximum(g.standard_normal((n, H, H, C)), 0.0))  # post-ReLU: many ties at zero
    with D.precision("f16"):
        P = (H - 1) // 2 + 1
        y = torch.empty((n, P, P, C), dtype=torch.float16, device="cuda")
        arg = torch.empty((n, P, P, C), dtype=torch.uint8, device="cuda")
        D.dbl_maxpool_fwd(n, H, H, C, dev16(x), y, arg)
        torch.cuda.synchronize()
    ry, rarg = orc.maxpool_fwd(x, 3, 2, 1)
    assert np.array_equal(host(y), ry) and np.array_equal(arg.cpu().numpy().astype(np.int32), rarg)


def test_scaled_head_is_the_scale_times_the_head(D):
    """Loss scaling by a power of two multiplies the head's fp32 gradients exactly."""
    n, hw, c, classes = 64, 16, 512, 100
    g = rng(9)
    x = dev16(f16_values(np.maximum(g.standard_normal((n, hw, c)), 0)))
    W, b = dev32(0.05 * g.standard_normal((classes, c))), dev32(0.01 * g.standard_normal(classes))
    lab = torch.from_numpy(g.integers(0, classes, n).astype(np.int32)).cuda()
    S = torch.tensor([2.0 ** 15], device="cuda")
    wsb = D.dbl_head_workspace_bytes(n, c, classes)
    outs = []
    with D.precision("f16"):
        for scale in (None, S):
            o = (torch.empty(1, device="cuda"), torch.empty((classes, c), device="cuda"),
                 torch.empty(classes, device="cuda"), torch.empty((n, hw, c), dtype=torch.float16, device="cuda"))
            D.dbl_head_fwd_bwd_ex(n, hw, c, classes, x, W, b, lab, D.head_opts(0.0, 0, None, scale), *o, ws(wsb), wsb)
            outs.append(o)
        torch.cuda.synchronize()
    (l1, w1, b1, _), (l2, w2, b2, dx2) = outs
    assert torch.equal(l1, l2)  # the loss is reported unscaled
    assert torch.equal(w2, w1 * 2.0 ** 15) and torch.equal(b2, b1 * 2.0 ** 15)
    assert torch.isfinite(dx2.float()).all()


@pytest.mark.parametrize("order", [0, 2])
def test_scaled_merge_matches_oracle_and_skips_overflow(D, order):
    n = 100_003
    g = rng(order + 40)
    w0, u0 = g.standard_normal(n).astype(np.float32), (0.01 * g.standard_normal(n)).astype(np.float32)
    SL, SS = 2.0 ** 15, 2.0 ** 13
    gl = (g.standard_normal(n) * 0.1 * SL).astype(np.float32)
    gs = (g.standard_normal(n) * 0.1 * SS).astype(np.float32)
    with D.precision("f16"):
        w, u = dev32(w0), dev32(u0)
        w16 = torch.empty(n, dtype=torch.float16, device="cuda")
        sl, ss = torch.tensor([SL], device="cuda"), torch.tensor([SS], device="cuda")
        fi = torch.zeros(1, dtype=torch.int32, device="cuda")
        D.dbl_grads_finite(dev32(gl), n, fi)
        D.dbl_grads_finite(dev32(gs), n, fi)
        D.dbl_ps_dual_batch_merge_scaled(w, u, w16, dev32(gl), dev32(gs), n, 0.2, 0.9, 1.0, 19 / 21, order, sl, ss, fi)
        torch.cuda.synchronize()
        assert int(fi.item()) == 0
        rw, ru, ok = orc.ps_merge_scaled(w0, u0, gl, gs, 0.2, 0.9, 1.0, 19 / 21, order, SL, SS)
        assert ok and max_norm_rel(host(w), rw) <= 1e-6 and max_norm_rel(host(u), ru) <= 1e-6
        assert torch.equal(w16, w.to(torch.float16))
        # one infinite value in the small push: nothing is written
        gs_bad = gs.copy()
        gs_bad[n // 2] = np.inf
        w1, u1, w161 = w.clone(), u.clone(), w16.clone()
        D.dbl_grads_finite(dev32(gl), n, fi)
        D.dbl_grads_finite(dev32(gs_bad), n, fi)
        D.dbl_ps_dual_batch_merge_scaled(w, u, w16, dev32(gl), dev32(gs_bad), n, 0.2, 0.9, 1.0, 19 / 21, order, sl, ss,
                                         fi)
        torch.cuda.synchronize()
    assert int(fi.item()) == 1
    assert torch.equal(w, w1) and torch.equal(u, u1) and torch.equal(w16, w161)


def test_loss_scale_update_follows_the_oracle(D):
    st = torch.zeros(4, dtype=torch.int32, device="cuda")
    st[0:1].view(torch.float32).fill_(2.0 ** 15)
    s, good = 2.0 ** 15, 0
    with D.precision("f16"):
        for found_inf in (0, 0, 1, 0, 0, 0, 1, 1, 0):
            st[2] = found_inf
            D.dbl_loss_scale_update(st, 3)
            s, good = orc.loss_scale_update(s, good, found_inf, 3)
            h = st.cpu()
            assert (float(h[0:1].view(torch.float32)), int(h[1]), int(h[2])) == (s, good, 0)
    assert int(st[3]) == 3  # skipped updates
