"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every entry point include/dbl.h declares, its host helpers agree with the
oracle, and malformed arguments are rejected before any launch."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle as orc
from oracle import planner
from paper_2509_26092_gb300 import build_lib

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def D():
    build_lib.build()
    from paper_2509_26092_gb300 import dbl
    return dbl


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "dbl.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dbl_[a-z0-9_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(D):
    L = D.lib()
    names = declared_symbols()
    assert len(names) >= 20
    for name in names:
        assert hasattr(L, name), name


def test_version(D):
    assert D.dbl_version() >= 100


@pytest.mark.parametrize("n_in,n_out", [(32, 16), (32, 24), (224, 128), (224, 160), (224, 224), (17, 5)])
def test_resize_taps_match_oracle(D, n_in, n_out):
    i0, i1, lam = D.dbl_resize_taps(n_in, n_out)
    r0, r1, rl = orc.resize_taps(n_in, n_out)
    np.testing.assert_array_equal(i0, r0)
    np.testing.assert_array_equal(i1, r1)
    np.testing.assert_allclose(lam, rl, rtol=0, atol=2 ** -24)


def test_resize_upsampling_rejected(D):
    with pytest.raises(D.DblError) as e:
        D.dbl_resize_taps(16, 32)
    assert e.value.code == D.DBL_ERR_UNSUPPORTED


def test_update_factor_and_plan_match_oracle(D):
    assert D.dbl_update_factor(10625, 13125) == planner.update_factor(10625, 13125)
    assert D.dbl_update_factor(8750, 13750, True) == planner.update_factor(8750, 13750, True)
    dL, dS, BS, fS = D.dbl_plan(1.05, 50000, 1, 3, 1.0, 24.8, 500, False)
    assert abs(dL - planner.data_large(1.05, 50000, 4)) < 1e-9
    assert abs(dS - planner.data_small(50000, 3, 1, dL)) < 1e-9
    assert abs(BS - planner.small_batch(1.0, 24.8, 500, dL, dS)) < 1e-9
    assert int(BS) == 83
    assert abs(fS - dS / dL) < 1e-15
    with pytest.raises(D.DblError):
        D.dbl_plan(1.05, 50000, 0, 4, 1.0, 24.8, 500, False)


def test_workspace_sizes_are_host_computable(D):
    s = D.conv_shape(8, 16, 16, 64, 64, 3, 1, 1)
    assert D.dbl_conv_workspace_bytes(s, D.DBL_PASS_FWD) > 0
    assert D.dbl_conv_workspace_bytes(s, D.DBL_PASS_WGRAD) >= 0
    assert D.dbl_conv_workspace_bytes(D.conv_shape(8, 16, 16, 64, 60, 3, 1, 1), D.DBL_PASS_FWD) == 0  # unsupported
    assert D.dbl_bn_workspace_bytes(D.bn_shape(1000, 64)) > 0
    assert D.dbl_head_workspace_bytes(4, 512, 100) > 0


def test_invalid_arguments_rejected_before_launch(D):
    L = D.lib()
    p = D.MergeParams(0.2, 0.9, 1.0, 0.9, 0)
    # both pushes missing
    assert L.dbl_ps_dual_batch_merge(16, 32, None, None, None, 8, ctypes.byref(p), None) == D.DBL_ERR_INVALID
    # misaligned master weights
    assert L.dbl_ps_dual_batch_merge(18, 32, None, 48, None, 8, ctypes.byref(p), None) == D.DBL_ERR_INVALID
    bad = D.MergeParams(0.2, 0.9, 1.0, 0.9, 7)
    assert L.dbl_ps_dual_batch_merge(16, 32, None, 48, None, 8, ctypes.byref(bad), None) == D.DBL_ERR_INVALID
    # conv: unsupported channel counts, non-square filters, bad workspace
    s = D.ConvShape(2, 8, 8, 60, 64, 3, 3, 1, 1)
    assert L.dbl_conv_fwd(ctypes.byref(s), 16, 16, 16, None, None, None, 0, None) == D.DBL_ERR_INVALID
    s = D.ConvShape(2, 8, 8, 64, 64, 3, 1, 1, 1)  # non-square: fine forward, not for the data gradient
    assert L.dbl_conv_dgrad(ctypes.byref(s), 16, 16, 16, None, 0, None) == D.DBL_ERR_UNSUPPORTED
    s = D.ConvShape(2, 8, 8, 64, 64, 3, 3, 3, 1)  # stride 3
    assert L.dbl_conv_fwd(ctypes.byref(s), 16, 16, 16, None, None, None, 0, None) == D.DBL_ERR_UNSUPPORTED
    s = D.ConvShape(8, 32, 32, 64, 64, 3, 3, 1, 1)  # 8192 pixels: the reduction is split, needing a workspace
    assert D.dbl_conv_workspace_bytes(s, D.DBL_PASS_WGRAD) > 0
    assert L.dbl_conv_wgrad(ctypes.byref(s), 16, 16, 16, 0, None, 0, None) == D.DBL_ERR_WORKSPACE
    s = D.ConvShape(2, 8, 8, 8, 64, 7, 7, 2, 3)
    assert L.dbl_conv_dgrad(ctypes.byref(s), 16, 16, 16, None, 0, None) == D.DBL_ERR_UNSUPPORTED
    # fused projection data gradient: stride 2 only, 64-multiple projection channels, both tensors given
    s = D.ConvShape(2, 8, 8, 64, 128, 3, 3, 1, 1)
    assert L.dbl_conv_dgrad_proj(ctypes.byref(s), 16, 16, 128, 16, 16, 16, None, 0, None) == D.DBL_ERR_UNSUPPORTED
    s = D.ConvShape(2, 8, 8, 64, 128, 3, 3, 2, 1)
    assert L.dbl_conv_dgrad_proj(ctypes.byref(s), 16, 16, 96, 16, 16, 16, None, 0, None) == D.DBL_ERR_UNSUPPORTED
    assert L.dbl_conv_dgrad_proj(ctypes.byref(s), 16, 16, 128, None, 16, 16, None, 0, None) == D.DBL_ERR_INVALID
    assert L.dbl_conv_dgrad_proj(ctypes.byref(s), 16, 16, 128, 24, 16, 16, None, 0, None) == D.DBL_ERR_INVALID
    # resize: upsampling
    assert L.dbl_progressive_resize(16, 0, 1, 8, 8, 3, 16, 1, 16, 16, 8, None) == D.DBL_ERR_UNSUPPORTED
    assert L.dbl_progressive_resize_stem(16, 1, 8, 8, 3, 16, 16, 16, 7, 2, 3, 1, 0, 16, None) == D.DBL_ERR_UNSUPPORTED
    assert L.dbl_progressive_resize_stem(16, 1, 16, 16, 3, 16, 16, 16, 9, 2, 3, 1, 0, 16, None) == D.DBL_ERR_UNSUPPORTED
    assert L.dbl_progressive_resize_stem(16, 1, 16, 16, 3, 16, 16, 16, 7, 2, 3, 3, 3, 11, None) == D.DBL_ERR_UNSUPPORTED
    assert L.dbl_progressive_resize_stem(16, 1, 16, 16, 5, 16, 16, 16, 7, 2, 3, 2, 3, 11, None) == D.DBL_ERR_UNSUPPORTED
    assert L.dbl_progressive_resize_stem(16, 1, 16, 16, 3, 16, 16, 16, 7, 2, 3, 2, 3, 0, None) == D.DBL_ERR_INVALID
    assert L.dbl_zero_f32_2d(16, 4, 8, 4, None) == D.DBL_ERR_INVALID
    # BN: channel count that is not a multiple of 8
    b = D.BnShape(100, 12, 1e-5, 1)
    assert L.dbl_bn_relu_fused(ctypes.byref(b), 16, 16, 16, 16, 16, None, 16, 16, 16, None) == D.DBL_ERR_UNSUPPORTED
    assert "channel" in D.dbl_last_error()
