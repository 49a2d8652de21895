"""loom_attn_decode_noalloc: the decode entry point for callers that cannot allocate.

Callers such as serving engines that reserve all device memory up front (cudaMalloc on
the request path would synchronise the device and may fail) or plug-in hosts that hand
over only the call's tensors cannot supply a decode workspace.  This test calls the
no-allocation entry point directly through the C ABI, twice in a row with different
inputs, and checks each result against loom_attn_decode with a caller-provided
workspace, within the parity tolerances of the other tests.  It runs last (file name)
and also passes alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest

import synth
from tests.gpu_util import TOL_LSE, TOL_MAX_ABS, TOL_MEAN_ABS, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def loom():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_29219_gb300 as m
    fn = m.capi().loom_attn_decode_noalloc
    vp, i32 = ctypes.c_void_p, ctypes.c_int
    fn.argtypes = [vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, ctypes.c_float, i32, vp]
    fn.restype = i32
    return m


def _case(seed, B, Hq, Hkv, Skv, D, lens):
    import torch
    q = to_dev(synth.bf16_normal(seed, synth.STREAM_Q, (B, Hq, 1, D)))
    k = to_dev(synth.bf16_normal(seed, synth.STREAM_K, (B, Hkv, Skv, D)))
    v = to_dev(synth.bf16_normal(seed, synth.STREAM_V, (B, Hkv, Skv, D)))
    sl = torch.from_numpy(np.asarray(lens, np.int32)).cuda()
    return q, k, v, sl


def _noalloc(loom, q, k, v, sl, num_splits):
    import torch
    B, Hq, _, D = q.shape
    Hkv, Skv = k.shape[1], k.shape[2]
    o = torch.empty_like(q)
    lse = torch.empty((B, Hq), dtype=torch.float32, device=q.device)
    st = loom.capi().loom_attn_decode_noalloc(
        q.data_ptr(), k.data_ptr(), v.data_ptr(), sl.data_ptr(), o.data_ptr(), lse.data_ptr(),
        B, Hq, Hkv, Skv, D, ctypes.c_float(D ** -0.5), num_splits,
        torch.cuda.current_stream().cuda_stream)
    assert st == 0, loom.loom_status_string(st)
    loom.loom_attn_check_error()
    return o, lse


def _compare(o, lse, o_ref, lse_ref):
    a = o.float().cpu().numpy().astype(np.float64)
    b = o_ref.float().cpu().numpy().astype(np.float64)
    err = np.abs(a - b)
    assert err.max() <= TOL_MAX_ABS and err.mean() <= TOL_MEAN_ABS
    la, lb = lse.cpu().numpy(), lse_ref.cpu().numpy()
    assert np.array_equal(np.isneginf(la), np.isneginf(lb))
    fin = np.isfinite(lb)
    assert np.all(np.abs(la[fin] - lb[fin]) <= TOL_LSE)


def test_noalloc_matches_workspace_entry_point_twice(loom):
    cases = [
        (21, 16, 32, 8, 8192, 128, synth.decode_lengths(21, 16, 4096, 8192), 16),
        (22, 5, 16, 2, 3000, 64, [0, 1, 65, 2999, 3000], 0),
    ]
    for seed, B, Hq, Hkv, Skv, D, lens, splits in cases:
        q, k, v, sl = _case(seed, B, Hq, Hkv, Skv, D, lens)
        o_ref, lse_ref = loom.loom_attn_decode(q, k, v, sl, num_splits=splits, return_lse=True)
        loom.loom_attn_check_error()
        o, lse = _noalloc(loom, q, k, v, sl, splits)
        _compare(o, lse, o_ref, lse_ref)


def test_noalloc_rejects_problems_beyond_its_scratch(loom):
    import torch
    B, Hq, Hkv, Skv, D, splits = 64, 64, 8, 65536, 128, 1024
    need = loom.loom_attn_decode_workspace_bytes(B, Hq, Hkv, Skv, D, splits)
    assert need > 8 << 20
    dummy = torch.empty(64, dtype=torch.bfloat16, device="cuda")
    p = dummy.data_ptr()
    st = loom.capi().loom_attn_decode_noalloc(p, p, p, None, p, None, B, Hq, Hkv, Skv, D,
                                             ctypes.c_float(0.08), splits, None)
    assert st == 4  # LOOM_ERR_WORKSPACE, nothing launched
