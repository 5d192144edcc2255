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


def stem_fold(x_u, r, stride, pad, width):
    """Logical NHWC stem input [n, h, width, 8] from the W-unrolled tensor
    [n, h, P, 8 taps, 8 channels] (x_u[..., q, t, :] is column q*stride + t - pad).
    Checks that every copy of a column holds the same values."""
    n, h, P = x_u.shape[0], x_u.shape[1], x_u.shape[2]
    x_u = x_u.reshape(n, h, P, 8, 8)
    out = np.full((n, h, width, 8), np.nan)
    for q in range(P):
        for t in range(r):
            w = q * stride + t - pad
            if 0 <= w < width:
                if not np.all(np.isnan(out[:, :, w, :])):
                    assert np.array_equal(out[:, :, w, :], x_u[:, :, q, t, :]), "unrolled copies disagree"
                out[:, :, w, :] = x_u[:, :, q, t, :]
    return out
