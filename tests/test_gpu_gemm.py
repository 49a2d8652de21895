"""GPU parity of the BF16 GEMM (through the C ABI) against the fp64 oracle.

Bound: C is rounded to bf16 once (at most 2^-9 relative error, written here as 2^-8 for
margin), and the fp32 accumulation over K adds at most ~K * 2^-24 * sum_k |a_ik b_kj|,
which for N(0,1) inputs stays below 1e-6 * K in absolute terms at these sizes."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import to_dev

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


@pytest.fixture(autouse=True, params=[0, 64, 128, 192, 256], ids=["model", "bn64", "bn128", "bn192", "bn256"])
def tile_n(request, loom):
    loom.loom_debug_gemm_tile_n(request.param)
    yield request.param
    loom.loom_debug_gemm_tile_n(0)


def _inputs(seed, M, K, N):
    return synth.bf16_normal(seed, synth.STREAM_Q, (M, K)), synth.bf16_normal(seed, synth.STREAM_K, (K, N))


def _check(c_gpu, c_ref, K, what):
    diff = np.abs(c_gpu - c_ref)
    bound = 2.0 ** -8 * np.abs(c_ref) + 1e-6 * K + 1e-6
    worst = np.max(diff - bound)
    assert worst <= 0, f"{what}: max excess {worst:.3g} (max |diff| {diff.max():.3g})"


def _run(loom, a, b):
    import torch
    c = loom.loom_gemm_bf16(to_dev(a), to_dev(b))
    loom.loom_attn_check_error()
    return c.float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("M,K,N", [(128, 64, 256), (1, 8, 8), (200, 136, 304), (130, 72, 264), (255, 1000, 520),
                                   (1000, 1000, 1000), (64, 4096, 64), (2048, 256, 256)])
def test_full_parity(loom, M, K, N):
    a, b = _inputs(M + K + N, M, K, N)
    _check(_run(loom, a, b), oracle.gemm(a, b), K, f"{M}x{K}x{N}")


@pytest.mark.parametrize("M,K,N", [(4096, 4096, 4096), (8192, 2048, 1024)])
def test_large_sampled_rows(loom, M, K, N):
    a, b = _inputs(7, M, K, N)
    c = _run(loom, a, b)
    rng = np.random.default_rng(0)
    rows = np.unique(np.concatenate([[0, 127, 128, M - 1], rng.integers(0, M, 60)]))
    _check(c[rows], oracle.gemm(a, b, rows=rows), K, f"{M}x{K}x{N} sampled")


def test_identity_and_zeros(loom):
    K, N = 256, 512
    eye = np.zeros((K, K), np.uint16)
    eye[np.arange(K), np.arange(K)] = 0x3F80
    b = synth.bf16_normal(3, synth.STREAM_V, (K, N))
    np.testing.assert_array_equal(_run(loom, eye, b), oracle.bf16_to_f64(b))  # exact: one product per entry
    z = np.zeros((K, N), np.uint16)
    np.testing.assert_array_equal(_run(loom, eye, z), 0.0)


def test_timeout_is_reported_and_context_survives(loom, tile_n):
    if tile_n not in (0, 256):
        pytest.skip("one tile width is enough")
    M, K, N = 256, 1024, 512
    a, b = _inputs(11, M, K, N)
    ad, bd = to_dev(a), to_dev(b)
    loom.loom_attn_check_error()
    loom.loom_debug_set_timeout_ns(50_000_000)
    try:
        loom.loom_debug_inject(3)
        loom.loom_gemm_bf16(ad, bd)
        with pytest.raises(loom.LoomError) as e:
            loom.loom_attn_check_error()
        assert e.value.status == 6
    finally:
        loom.loom_debug_inject(0)
        loom.loom_debug_set_timeout_ns(0)
    c = loom.loom_gemm_bf16(ad, bd)
    loom.loom_attn_check_error()
    _check(c.float().cpu().numpy().astype(np.float64), oracle.gemm(a, b), K, "after timeout")
