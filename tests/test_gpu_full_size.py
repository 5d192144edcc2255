"""Convolution passes at the full sizes the bench times: the 224 px layers of the
ImageNet-shaped ResNet-18 at the large worker's batch of 512, through the same
library calls and launch configurations as the training step (window kernels,
the 128-column window tiles and the 256-column tiles on CTA pairs, phase-split
stride-2 data gradients, split-K weight gradients).  The oracle computes sampled
outputs one by one in fp64 from the same inputs; the corners of every output
tensor are always among the samples.  Tolerance: max-norm relative 1e-2 over the
samples."""
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


def _check(got, ref, what):
    got, ref = np.asarray(got, dtype=np.float64), np.asarray(ref, dtype=np.float64)
    err = float(np.max(np.abs(got - ref))) / max(float(np.max(np.abs(ref))), 1e-30)
    assert err <= TOL, f"{what}: sampled max-norm relative error {err:.3e}"


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
    _check([dwh[i] for i in wg], [orc.conv2d_wgrad_at(x64, dy64, w64.shape, st, pad, *i) for i in wg], f"{case} wgrad")
