"""Helpers shared by the GPU parity tests: device upload and tolerance checks."""
import numpy as np

# Parity bar (fp64 oracle vs the CUDA path on identical bf16 inputs)
TOL_MAX_ABS = 2e-2
TOL_MEAN_ABS = 2e-3
TOL_LSE = 1e-3


def to_dev(bits, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


def o_to_f64(o):
    return o.float().cpu().numpy().astype(np.float64)


def assert_parity(o_gpu, o_ref, lse_gpu=None, lse_ref=None, what=""):
    o_gpu = np.asarray(o_gpu, np.float64).reshape(o_ref.shape)
    assert np.all(np.isfinite(o_gpu)), f"{what}: non-finite output"
    err = np.abs(o_gpu - o_ref)
    msg = f"{what}: max_abs={err.max():.3e} mean_abs={err.mean():.3e}"
    if lse_gpu is not None:
        lse_gpu = np.asarray(lse_gpu, np.float64).reshape(lse_ref.shape)
        fin = np.isfinite(lse_ref)
        assert np.array_equal(np.isneginf(lse_gpu), np.isneginf(lse_ref)), f"{what}: -inf pattern of LSE differs"
        lerr = np.abs(lse_gpu[fin] - lse_ref[fin])
        msg += f" lse={lerr.max() if lerr.size else 0:.3e}"
        assert lerr.size == 0 or lerr.max() <= TOL_LSE, msg
    assert err.max() <= TOL_MAX_ABS, msg
    assert err.mean() <= TOL_MEAN_ABS, msg
    return msg
