"""The convolution kernels' bounded waits: every mbarrier wait has a time and a poll limit, after
which the block records DBL_ERR_TIMEOUT in the device status and each of its roles winds down
through its own bounded waits.  A wait made to run out on purpose (dbl_conv_test_stall_next:
block 0 never loads its first K-block, so its MMA issuer waits on a stage that never fills) is
reported through the status, without a fault, and the context stays usable."""
import time

import numpy as np
import pytest
import torch

import oracle as orc
from conftest import max_norm_rel
from gpu_common import bf16_values, host, load_dbl, rng, to_bf16_dev, ws

pytestmark = pytest.mark.gpu


def test_a_conv_wait_that_runs_out_is_reported_and_the_context_survives():
    D = load_dbl()
    n, h, c, k = 4, 16, 64, 64
    shape = D.conv_shape(n, h, h, c, k, 1, 2, 0)  # 1x1 stride 2: one implicit-GEMM tile, one block
    info = D.dbl_conv_plan(shape, D.DBL_PASS_FWD)
    assert info.kernel == D.DBL_KERNEL_IGEMM and info.ctas_per_mma == 1 and info.grid == 1
    g = rng(77)
    x = bf16_values(g.standard_normal((n, h, h, c)))
    wt = bf16_values(g.standard_normal((k, 1, 1, c)) * 0.1)
    xd, wd = to_bf16_dev(x), to_bf16_dev(wt)
    y = torch.empty((n, h // 2, h // 2, k), dtype=torch.bfloat16, device="cuda")
    s1, s2 = torch.empty(k, device="cuda"), torch.empty(k, device="cuda")
    wsb = D.dbl_conv_workspace_bytes(shape, D.DBL_PASS_FWD)
    buf = ws(wsb)
    assert D.dbl_device_status() == D.DBL_OK
    D.dbl_conv_test_stall_next()
    t0 = time.monotonic()
    D.dbl_conv_fwd(shape, xd, wd, y, s1, s2, buf, wsb)
    status = D.dbl_device_status()  # synchronizes, then clears the status word
    waited = time.monotonic() - t0
    assert status == D.DBL_ERR_TIMEOUT
    assert 1.0 < waited < 60.0  # the wait's limit is about two seconds
    # the hook disarmed itself: the same call again completes and is right
    D.dbl_conv_fwd(shape, xd, wd, y, s1, s2, buf, wsb)
    assert D.dbl_device_status() == D.DBL_OK
    assert max_norm_rel(host(y), orc.conv2d_fwd(x, wt, 2, 0)) <= 1e-2
    np.testing.assert_allclose(host(s1), host(y).reshape(-1, k).sum(0), rtol=1e-4, atol=1e-2)
