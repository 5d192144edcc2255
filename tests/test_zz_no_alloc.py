"""The workspace-free BatchNorm backward entry point, called through the C ABI.

Some callers cannot allocate device memory on demand.  For example, a host
framework may own every device allocation, or a service may have to keep its
device-memory footprint fixed after start-up.  For them the library offers
dbl_bn_relu_fused_bwd_noalloc, which keeps its scratch in a fixed array
inside libdbl.so instead of taking a workspace.

Both entry points run the same kernels with the same partial counts, so their
outputs must agree bit for bit.  The test compares them on calls in a row with
different shapes, covering the branches that read the scratch differently (a
second incoming gradient, the residual-branch gradient whose apply pass reads
the coefficients back, and the ReLU mask recomputed from y), so a stale array
from an earlier call cannot go unnoticed.  It also checks that oversized
shapes are refused, and that a first call made inside a stream capture is
refused with a clear error (a fresh process, so the array's address is not
yet known).

The file is named to be collected last, so a run that stops at the first
failure has already run every other test.
"""
import ctypes
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from gpu_common import bf16_values, load_dbl, rng, to_bf16_dev, to_f32_dev, ws

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _case(seed, count, C):
    g = rng(seed)
    y = bf16_values(g.standard_normal((count, C)) * 1.5 + 0.3)
    out = bf16_values(np.maximum(g.standard_normal((count, C)), 0.0))
    dout = bf16_values(g.standard_normal((count, C)))
    dout2 = bf16_values(g.standard_normal((count, C)))
    gamma = (1.0 + 0.2 * g.standard_normal(C)).astype(np.float32)
    beta = (0.1 * g.standard_normal(C)).astype(np.float32)
    mean = y.mean(0).astype(np.float32)
    istd = (1.0 / np.sqrt(y.var(0) + 1e-5)).astype(np.float32)
    return ([to_bf16_dev(a) for a in (dout, dout2, y, out)] + [to_f32_dev(a) for a in (gamma, beta, mean, istd)])


def _outputs(count, C):
    bf = dict(dtype=torch.bfloat16, device="cuda")
    return (torch.full((count, C), float("nan"), **bf), torch.full((count, C), float("nan"), **bf),
            torch.full((C,), float("nan"), device="cuda"), torch.full((C,), float("nan"), device="cuda"))


# (count, channels, second incoming gradient, residual-branch gradient, stored ReLU output)
CASES = [(4096, 512, True, False, True), (1000, 64, False, True, True), (777, 128, True, False, False),
         (3001, 256, False, True, True)]


def test_noalloc_matches_workspace_version_bit_for_bit():
    D = load_dbl()
    L = D.lib()
    ptr = lambda t: None if t is None else t.data_ptr()
    for seed, (count, C, two, dres, stored) in enumerate(CASES):
        dout, dout2, y, out, gamma, beta, mean, istd = _case(100 + seed, count, C)
        dout2 = dout2 if two else None
        out = out if stored else None
        shape = D.bn_shape(count, C, 1e-5, True)
        ref = _outputs(count, C)
        nbytes = D.dbl_bn_workspace_bytes(shape)
        D.dbl_bn_relu_fused_bwd(shape, dout, dout2, y, out, gamma, mean, istd, ref[0], ref[1] if dres else None,
                                ref[2], ref[3], ws(nbytes), nbytes, beta=beta)
        got = _outputs(count, C)
        stream = torch.cuda.current_stream().cuda_stream
        rc = L.dbl_bn_relu_fused_bwd_noalloc(ctypes.byref(shape), ptr(dout), ptr(dout2), ptr(y), ptr(out), ptr(gamma),
                                             ptr(beta), ptr(mean), ptr(istd), ptr(got[0]), ptr(got[1]) if dres else None,
                                             ptr(got[2]), ptr(got[3]), stream)
        assert rc == D.DBL_OK, D.dbl_last_error()
        torch.cuda.synchronize()
        names = ("dy", "dresidual", "dgamma", "dbeta")
        for name, r, g_ in zip(names, ref, got):
            if name == "dresidual" and not dres:
                assert torch.isnan(g_.float()).all()  # not asked for: left untouched
                continue
            assert torch.isfinite(r.float()).all(), (count, C, name)
            assert torch.equal(g_, r), (count, C, name)
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


_FIRST_CALL_IN_CAPTURE = r"""
import sys, torch
sys.path.insert(0, sys.argv[1])
from paper_2509_26092_gb300 import build_lib
build_lib.build()
from paper_2509_26092_gb300 import dbl as D
torch.cuda.set_device(0)
C, n = 64, 512
g = torch.Generator(device="cuda").manual_seed(0)
t = lambda: torch.randn(n, C, device="cuda", generator=g).to(torch.bfloat16)
dout, y, out = t(), t(), torch.relu(t())
gamma, mean, istd = torch.ones(C, device="cuda"), y.float().mean(0), torch.ones(C, device="cuda")
dy, dg, db = torch.empty_like(y), torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
shape = D.bn_shape(n, C, 1e-5, True)
torch.cuda.synchronize()
graph, code = torch.cuda.CUDAGraph(), None
with torch.cuda.graph(graph):
    try:
        D.dbl_bn_relu_fused_bwd_noalloc(shape, dout, None, y, out, gamma, mean, istd, dy, None, dg, db)
    except D.DblError as e:
        code, msg = e.code, str(e)
assert code == D.DBL_ERR_INVALID and "capture" in msg, (code, msg)
# outside capture the same call runs, and matches the workspace version bit for bit
D.dbl_bn_relu_fused_bwd_noalloc(shape, dout, None, y, out, gamma, mean, istd, dy, None, dg, db)
rdy, rdg, rdb = torch.empty_like(y), torch.empty(C, device="cuda"), torch.empty(C, device="cuda")
nb = D.dbl_bn_workspace_bytes(shape)
D.dbl_bn_relu_fused_bwd(shape, dout, None, y, out, gamma, mean, istd, rdy, None, rdg, rdb,
                        torch.empty(nb, dtype=torch.uint8, device="cuda"), nb)
torch.cuda.synchronize()
assert torch.equal(dy, rdy) and torch.equal(dg, rdg) and torch.equal(db, rdb)
print("ok")
"""


def test_noalloc_first_call_inside_capture_is_refused():
    load_dbl()
    r = subprocess.run([sys.executable, "-c", _FIRST_CALL_IN_CAPTURE, ROOT], capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout[-2000:] + r.stderr[-2000:]
