"""The workspace-free BatchNorm backward entry point, called through the C ABI.

Some callers cannot allocate device memory on demand.  For example, a host
framework may own every device allocation, or a service may have to keep its
device-memory footprint fixed after start-up.  For them the library offers
dbl_bn_relu_fused_bwd_noalloc, which keeps its scratch in a fixed array
inside libdbl.so instead of taking a workspace.  This test checks that it
gives the same results as the workspace version, dbl_bn_relu_fused_bwd, on
two calls in a row with different shapes, so a stale array from the first call
cannot go unnoticed.  It also checks that oversized shapes are refused.

The file is named to be collected last, so a run that stops at the first
failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from conftest import max_norm_rel
from gpu_common import bf16_values, host, load_dbl, rng, to_bf16_dev, to_f32_dev, ws

pytestmark = pytest.mark.gpu

BF16_TOL = 1e-2   # bf16 outputs, as in the other BatchNorm parity tests
F32_TOL = 1e-4    # fp32 channel sums


def _case(seed, count, C):
    g = rng(seed)
    y = bf16_values(g.standard_normal((count, C)) * 1.5 + 0.3)
    out = bf16_values(np.maximum(g.standard_normal((count, C)), 0.0))
    dout = bf16_values(g.standard_normal((count, C)))
    dout2 = bf16_values(g.standard_normal((count, C)))
    gamma = (1.0 + 0.2 * g.standard_normal(C)).astype(np.float32)
    mean = y.mean(0).astype(np.float32)
    istd = (1.0 / np.sqrt(y.var(0) + 1e-5)).astype(np.float32)
    return [to_bf16_dev(a) for a in (dout, dout2, y, out)] + [to_f32_dev(a) for a in (gamma, mean, istd)]


def _outputs(count, C):
    bf = dict(dtype=torch.bfloat16, device="cuda")
    return (torch.full((count, C), float("nan"), **bf), torch.full((count, C), float("nan"), **bf),
            torch.full((C,), float("nan"), device="cuda"), torch.full((C,), float("nan"), device="cuda"))


def test_noalloc_matches_workspace_version_twice():
    D = load_dbl()
    L = D.lib()
    for seed, (count, C) in enumerate([(4096, 512), (1000, 64)]):
        dout, dout2, y, out, gamma, mean, istd = _case(100 + seed, count, C)
        shape = D.bn_shape(count, C, 1e-5, True)
        ref = _outputs(count, C)
        nbytes = D.dbl_bn_workspace_bytes(shape)
        D.dbl_bn_relu_fused_bwd(shape, dout, dout2, y, out, gamma, mean, istd, *ref[:2], *ref[2:], ws(nbytes), nbytes)
        got = _outputs(count, C)
        stream = torch.cuda.current_stream().cuda_stream
        rc = L.dbl_bn_relu_fused_bwd_noalloc(ctypes.byref(shape), dout.data_ptr(), dout2.data_ptr(), y.data_ptr(),
                                             out.data_ptr(), gamma.data_ptr(), None, mean.data_ptr(), istd.data_ptr(),
                                             got[0].data_ptr(), got[1].data_ptr(), got[2].data_ptr(),
                                             got[3].data_ptr(), stream)
        assert rc == D.DBL_OK, D.dbl_last_error()
        torch.cuda.synchronize()
        for r, g_, tol in zip(ref, got, (BF16_TOL, BF16_TOL, F32_TOL, F32_TOL)):
            assert torch.isfinite(g_).all()
            assert max_norm_rel(host(g_), host(r)) <= tol
    assert D.dbl_device_status() == D.DBL_OK


def test_noalloc_refuses_shapes_beyond_its_scratch():
    D = load_dbl()
    shape = D.bn_shape(256, 1024, 1e-5, True)
    t = torch.zeros((256, 1024), dtype=torch.bfloat16, device="cuda")
    v = torch.zeros(1024, device="cuda")
    with pytest.raises(D.DblError) as e:
        D.dbl_bn_relu_fused_bwd_noalloc(shape, t, None, t, t, v, v, v, t, None, v, v)
    assert e.value.code == D.DBL_ERR_UNSUPPORTED
    assert "512" in str(e.value)
