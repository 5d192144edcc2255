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


@pytest.mark.parametrize("precision", ["bf16", "f16"])
def test_every_declared_symbol_is_exported(D, precision):
    """Both builds (bfloat16 and binary16 storage) export every entry point dbl.h declares."""
    L = D.lib(precision)
    names = declared_symbols()
    assert len(names) >= 20
    for name in names:
        assert hasattr(L, name), name


def test_calls_go_to_the_library_of_the_current_precision(D):
    assert D.current_precision() == "bf16" and D.lib_path().endswith("libdbl.so")
    with D.precision("f16"):
        assert D.current_precision() == "f16" and D.lib_path().endswith("libdbl_f16.so")
        assert D.lib() is D.lib("f16") and D.lib("f16") is not D.lib("bf16")
    assert D.current_precision() == "bf16"
    with pytest.raises(ValueError):
        with D.precision("fp8"):
            pass


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


def _resnet18_convs(variant, batch, res):
    """(n, h, w, c, k, r, stride, pad) of every non-stem convolution of ResNet-18."""
    h = res // 4 if variant == "imagenet" else res  # after the ImageNet stem's stride 2 and max pool
    out, cin = [], 64
    for cout, st in ((64, 1), (128, 2), (256, 2), (512, 2)):
        for b in range(2):
            s = st if b == 0 else 1
            ho = (h + 2 - 3) // s + 1
            out.append((batch, h, h, cin, cout, 3, s, 1))
            out.append((batch, ho, ho, cout, cout, 3, 1, 1))
            if b == 0 and (s != 1 or cin != cout):
                out.append((batch, h, h, cin, cout, 1, s, 0))
            h, cin = ho, cout
    return out


def test_conv_plans_of_the_resnet18_layers(D):
    """The host-side plan (dbl_conv_plan): which kernel each layer of the step uses, and the
    invariants every plan keeps (grid within the workspace bound, even grids for CTA pairs,
    window kernels within shared memory).  Without a GPU the grid and tile counts come from a
    nominal SM count (never cached), so on a CPU host this pins only the choices that do not
    depend on the device: kernel, tile width, CTAs per MMA and phase count; the invariants hold
    for any SM count."""
    plan = lambda shp, p: D.dbl_conv_plan(D.conv_shape(*shp), p)
    FWD, DG, WG = D.DBL_PASS_FWD, D.DBL_PASS_DGRAD, D.DBL_PASS_WGRAD
    l1, l2, l3 = (512, 56, 56, 64, 64, 3, 1, 1), (512, 28, 28, 128, 128, 3, 1, 1), (512, 14, 14, 256, 256, 3, 1, 1)
    for p in (FWD, DG):
        i = plan(l1, p)
        assert (i.kernel, i.tile_cols, i.ctas_per_mma) == (D.DBL_KERNEL_WINDOW, 64, 1)
        i = plan(l2, p)
        assert (i.kernel, i.tile_cols, i.ctas_per_mma) == (D.DBL_KERNEL_WINDOW, 128, 2)
        i = plan(l3, p)
        assert (i.kernel, i.tile_cols, i.ctas_per_mma) == (D.DBL_KERNEL_IGEMM, 256, 2)
    assert plan(l1, WG).kernel == D.DBL_KERNEL_WINDOW_WGRAD
    assert plan((512, 56, 56, 64, 128, 3, 2, 1), DG).zdim == 4  # stride-2 data gradient: four phases
    for variant, batch, res in (("imagenet", 512, 224), ("imagenet", 128, 224), ("imagenet", 512, 160),
                                ("imagenet", 512, 128), ("cifar", 256, 32), ("cifar", 1024, 16)):
        for shp in _resnet18_convs(variant, batch, res):
            for p in (FWD, DG, WG):
                i = plan(shp, p)
                assert 1 <= i.grid <= 256 and i.tiles >= 1 and i.zdim >= 1, (shp, p)
                assert i.ctas_per_mma in (1, 2) and (i.ctas_per_mma == 1 or i.grid % 2 == 0), (shp, p)
                if i.kernel == D.DBL_KERNEL_IGEMM:
                    assert i.smem_bytes == 0
                else:
                    assert 0 < i.smem_bytes <= 232448 - 2048, (shp, p, i.smem_bytes)
    with pytest.raises(Exception):
        D.dbl_conv_plan(D.conv_shape(2, 8, 8, 24, 64, 3, 1, 1), FWD)  # 24 input channels: unsupported


def test_cta_pairs_can_be_switched_off():
    """DBL_CONV_CTA_PAIRS=0 plans every pass on single CTAs (read once per process)."""
    import subprocess
    import sys
    code = ("from paper_2509_26092_gb300 import build_lib\nbuild_lib.build()\n"
            "from paper_2509_26092_gb300 import dbl as D\n"
            "for shp in ((512, 28, 28, 128, 128, 3, 1, 1), (512, 14, 14, 256, 256, 3, 1, 1)):\n"
            "    for p in (0, 1, 2):\n"
            "        assert D.dbl_conv_plan(D.conv_shape(*shp), p).ctas_per_mma == 1\n")
    env = dict(os.environ, DBL_CONV_CTA_PAIRS="0")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]


def test_window_pairs_of_64_columns_only_for_comparison():
    """The 64-column window forward pass with resident weights runs on CTA pairs only with
    DBL_CONV_CTA_PAIRS=2 (measured no faster); its data gradient never does."""
    import subprocess
    import sys
    code = ("from paper_2509_26092_gb300 import build_lib\nbuild_lib.build()\n"
            "from paper_2509_26092_gb300 import dbl as D\nimport sys\n"
            "i = D.dbl_conv_plan(D.conv_shape(512, 56, 56, 64, 64, 3, 1, 1), 0)\n"
            "d = D.dbl_conv_plan(D.conv_shape(512, 56, 56, 64, 64, 3, 1, 1), 1)\n"
            "assert i.kernel == D.DBL_KERNEL_WINDOW and d.ctas_per_mma == 1\n"
            "print(i.ctas_per_mma)\n")
    got = {}
    for level in ("1", "2"):
        r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=dict(os.environ, DBL_CONV_CTA_PAIRS=level),
                           capture_output=True, text=True, timeout=300)
        assert r.returncode == 0, r.stderr[-2000:]
        got[level] = int(r.stdout.split()[-1])
    assert got == {"1": 1, "2": 2}


def test_conv_pdl_setter_validates_its_mode(D):
    """dbl_set_conv_pdl (host): 1, 0 and -1 are accepted by both libraries, anything else refused."""
    for mode in (1, 0, -1):
        D.dbl_set_conv_pdl(mode)
    for p in D.PRECISIONS:
        assert D.lib(p).dbl_set_conv_pdl(2) == D.DBL_ERR_INVALID
