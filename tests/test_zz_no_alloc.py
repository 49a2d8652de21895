"""loom_attn_decode_noalloc: the decode entry point for callers that cannot allocate.

Callers such as serving engines that reserve all device memory up front (cudaMalloc on
the request path would synchronise the device and may fail) or plug-in hosts that hand
over only the call's tensors cannot supply a decode workspace.  This test calls the
no-allocation entry point directly through the C ABI, twice in a row with different
inputs.  It runs the same kernels on the same inputs as loom_attn_decode with a
caller-provided workspace, so each result must equal that entry point's bit for bit; a
partial left over from the previous call in the shared scratch array would show up as a
difference.  One case is also checked against the fp64 oracle.  The file runs last (its
name) and also passes alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import assert_parity, o_to_f64, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def loom():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_29219_gb300 as m
    return m


def _case(seed, B, Hq, Hkv, Skv, D, lens):
    q = synth.bf16_normal(seed, synth.STREAM_Q, (B, Hq, 1, D))
    k = synth.bf16_normal(seed, synth.STREAM_K, (B, Hkv, Skv, D))
    v = synth.bf16_normal(seed, synth.STREAM_V, (B, Hkv, Skv, D))
    return q, k, v, np.asarray(lens, np.int32)


def _noalloc(loom, q, k, v, sl, num_splits):
    """One call of the C entry point (the raw ctypes function, no Python wrapper)."""
    import torch
    B, Hq, _, D = q.shape
    Hkv, Skv = k.shape[1], k.shape[2]
    o = torch.full_like(q, float("nan"))
    lse = torch.full((B, Hq), float("nan"), dtype=torch.float32, device=q.device)
    st = loom.capi().loom_attn_decode_noalloc(
        q.data_ptr(), k.data_ptr(), v.data_ptr(), sl.data_ptr(), o.data_ptr(), lse.data_ptr(),
        B, Hq, Hkv, Skv, D, ctypes.c_float(D ** -0.5), num_splits,
        torch.cuda.current_stream().cuda_stream)
    assert st == 0, loom.loom_status_string(st)
    loom.loom_attn_check_error()
    return o, lse


def test_noalloc_equals_workspace_entry_point_twice(loom):
    import torch
    cases = [
        (21, 16, 32, 8, 8192, 128, synth.decode_lengths(21, 16, 4096, 8192), 16),
        (22, 5, 16, 2, 3000, 64, [0, 1, 65, 2999, 3000], 0),
    ]
    for i, (seed, B, Hq, Hkv, Skv, D, lens, splits) in enumerate(cases):
        qh, kh, vh, lh = _case(seed, B, Hq, Hkv, Skv, D, lens)
        q, k, v = to_dev(qh), to_dev(kh), to_dev(vh)
        sl = torch.from_numpy(lh).cuda()
        o_ref, lse_ref = loom.loom_attn_decode(q, k, v, sl, num_splits=splits, return_lse=True)
        loom.loom_attn_check_error()
        o, lse = _noalloc(loom, q, k, v, sl, splits)
        assert torch.equal(o.view(torch.int16), o_ref.view(torch.int16)), f"call {i}: O differs"
        assert torch.equal(lse, lse_ref), f"call {i}: LSE differs"
        if i == 1:  # the edge lengths (0, 1, 65, full) against the definition
            o_or, lse_or = oracle.attention(qh, kh, vh, seqlens_k=lh)
            assert_parity(o_to_f64(o), o_or, lse.cpu().numpy(), lse_or, "no-alloc decode vs oracle")


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
