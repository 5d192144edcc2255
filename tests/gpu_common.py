"""Helpers shared by the GPU parity tests (no arithmetic of the method here)."""
import numpy as np
import pytest
import torch

from paper_2509_26092_gb300 import build_lib


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def load_dbl():
    need_gpu()
    build_lib.build()
    from paper_2509_26092_gb300 import dbl
    return dbl


def to_bf16_dev(a):
    """numpy float -> bf16 CUDA tensor (round to nearest even)."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).cuda()


def to_f32_dev(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def host(t):
    """CUDA tensor -> float64 numpy."""
    return t.detach().float().cpu().numpy().astype(np.float64)


def bf16_values(a):
    """The float64 values of a after rounding to bf16 (the inputs both sides see)."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).double().numpy()


def ws(nbytes):
    return torch.empty(max(int(nbytes), 16), dtype=torch.uint8, device="cuda")


def rng(seed):
    return np.random.default_rng(seed)


def check_status(D):
    assert D.dbl_device_status() == D.DBL_OK


def stem_fold(x_u, r, stride, pad, width, rg=1, pad_h=0, height=None):
    """Logical NHWC stem input [n, height, width, 8/rg] from the unrolled tensor
    [n, rows, P, rg rows, 8 taps, 8/rg channels]: x_u[:, m, q, e, t, :] is the pixel at
    row rg*m + e - pad_h, column q*stride + t - pad.  Pixels no position covers stay NaN.
    Checks that every copy of a pixel holds the same values."""
    height = width if height is None else height
    n, rows, P = x_u.shape[0], x_u.shape[1], x_u.shape[2]
    cu = 8 // rg
    x_u = x_u.reshape(n, rows, P, rg, 8, cu)
    out = np.full((n, height, width, cu), np.nan)
    for m in range(rows):
        for e in range(rg):
            y = rg * m + e - pad_h
            if not 0 <= y < height:
                continue
            for q in range(P):
                for t in range(r):
                    x = q * stride + t - pad
                    if 0 <= x < width:
                        v = x_u[:, m, q, e, t, :]
                        if not np.all(np.isnan(out[:, y, x, :])):
                            assert np.array_equal(out[:, y, x, :], v), "unrolled copies disagree"
                        out[:, y, x, :] = v
    return out
