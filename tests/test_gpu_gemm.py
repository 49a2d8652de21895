"""GPU parity of the BF16 GEMM (through the C ABI) against the fp64 oracle.

Bound: C is rounded to bf16 once (at most 2^-9 relative error, written here as 2^-8 for
margin), and the fp32 accumulation over K adds at most ~K * 2^-24 * sum_k |a_ik b_kj|,
which for N(0,1) inputs stays below 1e-6 * K in absolute terms at these sizes.  The same
bound holds for every split count: the split only regroups the fp32 sum."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import to_dev

pytestmark = pytest.mark.gpu

TILE_WIDTHS = (64, 128, 192, 256)
SPLITS = (2, 4, 8, 16)


@pytest.fixture(scope="module")
def loom():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_29219_gb300 as m
    yield m
    m.loom_debug_gemm_tile_n(0)
    m.loom_debug_gemm_splits(0)
    m.loom_debug_gemm_cta_pair(0)
    m.loom_debug_inject(0)
    m.loom_debug_set_timeout_ns(0)


@pytest.fixture
def forced(loom):
    """forced(tile_n, splits, pair): pin the kernel variant for one test (0 = the model's
    choice; pair 1 = CTA-pair 256 x 256 tiles, -1 = single-CTA kernels only)."""
    def set_(tile_n=0, splits=0, pair=None):
        if pair is None:
            pair = -1 if (tile_n or splits) else 0
        loom.loom_debug_gemm_tile_n(tile_n)
        loom.loom_debug_gemm_splits(splits)
        loom.loom_debug_gemm_cta_pair(pair)
        assert tile_n == 0 or loom.loom_gemm_tile_n(8, 8, 8) == tile_n
        assert pair != 1 or loom.loom_gemm_cta_pair(8, 8, 8) == 1
    yield set_
    loom.loom_debug_gemm_tile_n(0)
    loom.loom_debug_gemm_splits(0)
    loom.loom_debug_gemm_cta_pair(0)


def _inputs(seed, M, K, N):
    return synth.bf16_normal(seed, synth.STREAM_Q, (M, K)), synth.bf16_normal(seed, synth.STREAM_K, (K, N))


def _check(c_gpu, c_ref, K, what):
    assert np.all(np.isfinite(c_gpu)), f"{what}: non-finite output"
    diff = np.abs(c_gpu - c_ref)
    bound = 2.0 ** -8 * np.abs(c_ref) + 1e-6 * K + 1e-6
    worst = np.max(diff - bound)
    assert worst <= 0, f"{what}: max excess {worst:.3g} (max |diff| {diff.max():.3g})"


def _run_dev(loom, ad, bd):
    c = loom.loom_gemm_bf16(ad, bd)
    loom.loom_attn_check_error()
    return c


def _run(loom, a, b):
    return _run_dev(loom, to_dev(a), to_dev(b)).float().cpu().numpy().astype(np.float64)


# ---------------------------------------------------------------- persistent tiles (S = 1)
@pytest.mark.parametrize("tile_n", [0, *TILE_WIDTHS, "pair"], ids=["model", *[f"bn{b}" for b in TILE_WIDTHS], "pair"])
@pytest.mark.parametrize("M,K,N", [(128, 64, 256), (1, 8, 8), (200, 136, 304), (130, 72, 264), (255, 1000, 520),
                                   (1000, 1000, 1000), (64, 4096, 64), (2048, 256, 256), (384, 320, 768),
                                   (200, 136, 320), (1000, 1000, 960)])
def test_full_parity(loom, forced, tile_n, M, K, N):
    if tile_n == "pair":
        forced(0, 0, 1)
    else:
        forced(tile_n, 1 if tile_n else 0)
    a, b = _inputs(M + K + N, M, K, N)
    _check(_run(loom, a, b), oracle.gemm(a, b), K, f"{M}x{K}x{N} bn={tile_n}")


_LARGE = {}


def _large_case(M, K, N):
    """Inputs and the oracle's product of one large shape, computed once and shared by the
    kernel variants (every element is compared)."""
    if (M, K, N) not in _LARGE:
        a, b = _inputs(7, M, K, N)
        _LARGE[(M, K, N)] = (a, b, oracle.gemm(a, b))
    return _LARGE[(M, K, N)]


@pytest.mark.parametrize("tile_n", [0, 64, 256, "pair"], ids=["model", "bn64", "bn256", "pair"])
@pytest.mark.parametrize("M,K,N", [(4096, 4096, 4096), (8192, 2048, 1024)])
def test_large_full(loom, forced, tile_n, M, K, N):
    if tile_n == "pair":
        forced(0, 0, 1)
    else:
        forced(tile_n, 1 if tile_n else 0)
    a, b, c_ref = _large_case(M, K, N)
    _check(_run(loom, a, b), c_ref, K, f"{M}x{K}x{N} bn={tile_n}")


# ---------------------------------------------------------------- split-K clusters
@pytest.mark.parametrize("splits", SPLITS, ids=[f"s{s}" for s in SPLITS])
@pytest.mark.parametrize("tile_n", TILE_WIDTHS, ids=[f"bn{b}" for b in TILE_WIDTHS])
@pytest.mark.parametrize("M,K,N", [(128, 1024, 256), (200, 1000, 304), (130, 4096, 520), (384, 2048, 1000),
                                   (200, 1000, 320)])
def test_split_parity(loom, forced, tile_n, splits, M, K, N):
    forced(tile_n, splits)
    a, b = _inputs(3 * M + K + N, M, K, N)
    _check(_run(loom, a, b), oracle.gemm(a, b), K, f"{M}x{K}x{N} bn={tile_n} S={splits}")


@pytest.mark.parametrize("splits", SPLITS, ids=[f"s{s}" for s in SPLITS])
def test_split_with_idle_ctas(loom, forced, splits):
    """K = 64 is one stage: all but one CTA of each cluster get no stage and add zeros."""
    forced(64, splits)
    M, K, N = 256, 64, 192
    a, b = _inputs(5, M, K, N)
    _check(_run(loom, a, b), oracle.gemm(a, b), K, f"idle CTAs S={splits}")


@pytest.mark.parametrize("M,K,N", [(256, 16384, 256), (256, 16384, 2048), (2048, 2048, 256)])
def test_model_choice_long_k(loom, forced, M, K, N):
    """Shapes with few tiles and long K, on whatever (tile width, split) the model picks."""
    forced(0, 0)
    a, b = _inputs(9, M, K, N)
    c = _run(loom, a, b)
    rows = np.unique(np.concatenate([[0, 1, 127, 128, M - 1], np.random.default_rng(1).integers(0, M, 40)]))
    _check(c[rows], oracle.gemm(a, b, rows=rows), K,
           f"{M}x{K}x{N} model bn={loom.loom_gemm_tile_n(M, N, K)} S={loom.loom_gemm_splits(M, N, K)}")


@pytest.mark.parametrize("splits", [1, 4, 16, "pair"])
def test_deterministic(loom, forced, splits):
    if splits == "pair":
        forced(0, 0, 1)
    else:
        forced(128, splits)
    a, b = _inputs(13, 384, 4096, 512)
    ad, bd = to_dev(a), to_dev(b)
    import torch
    x1 = _run_dev(loom, ad, bd).view(torch.int16).cpu().numpy()
    x2 = _run_dev(loom, ad, bd).view(torch.int16).cpu().numpy()
    np.testing.assert_array_equal(x1, x2)


def test_identity_and_zeros(loom, forced):
    K, N = 256, 512
    eye = np.zeros((K, K), np.uint16)
    eye[np.arange(K), np.arange(K)] = 0x3F80
    b = synth.bf16_normal(3, synth.STREAM_V, (K, N))
    for tile_n, splits, pair in [(0, 0, 0), (64, 2, -1), (256, 4, -1), (0, 0, 1)]:
        forced(tile_n, splits, pair)
        np.testing.assert_array_equal(_run(loom, eye, b), oracle.bf16_to_f64(b))  # one product per entry
        np.testing.assert_array_equal(_run(loom, eye, np.zeros((K, N), np.uint16)), 0.0)


# ---------------------------------------------------------------- bounded waits
@pytest.mark.parametrize("tile_n,splits,pair", [(256, 1, -1), (64, 4, -1), (0, 0, 1)])
def test_timeout_is_reported_and_context_survives(loom, forced, tile_n, splits, pair):
    """The loader skips one stage (per CTA; for CTA pairs the even CTA never arms it); the
    waits on it run out, every CTA (and every cluster) unwinds, the error word says TIMEOUT,
    and the next call is correct."""
    forced(tile_n, splits, pair)
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
    c = _run_dev(loom, ad, bd)
    _check(c.float().cpu().numpy().astype(np.float64), oracle.gemm(a, b), K, "after timeout")


@pytest.mark.parametrize("M,K,N", [(1, 64, 512), (257, 128, 248), (3000, 640, 40), (512, 2048, 8)])
def test_pair_tiles_on_thin_shapes(loom, forced, M, K, N):
    """CTA-pair tiles on shapes far from 256 x 256 multiples: the odd CTA's rows (or most
    columns) fall outside C and are neither stored nor allowed to disturb the even CTA."""
    forced(0, 0, 1)
    a, b = _inputs(M * 7 + N, M, K, N)
    _check(_run(loom, a, b), oracle.gemm(a, b), K, f"pair {M}x{K}x{N}")


@pytest.mark.parametrize("variant", ["model", "bn128", "bn256", "split4", "pair"])
@pytest.mark.parametrize("M,K,N", [(200, 136, 304), (1000, 1000, 1000), (256, 4096, 264), (130, 64, 8)])
def test_transposed_b(loom, forced, variant, M, K, N):
    """b given [N, K] (C = A b^T): its tiles are K-major, in every kernel."""
    forced(*{"model": (0, 0, 0), "bn128": (128, 1, -1), "bn256": (256, 1, -1), "split4": (128, 4, -1),
             "pair": (0, 0, 1)}[variant])
    a = synth.bf16_normal(M + 5, synth.STREAM_Q, (M, K))
    bt = synth.bf16_normal(M + 5, synth.STREAM_K, (N, K))
    c = loom.loom_gemm_bf16(to_dev(a), to_dev(bt), b_transposed=True)
    loom.loom_attn_check_error()
    _check(c.float().cpu().numpy().astype(np.float64), oracle.gemm(a, bt, b_transposed=True), K,
           f"A B^T {M}x{K}x{N} {variant}")


def test_transposed_b_matches_plain_layout_bitwise(loom, forced):
    """The same product from B and from B^T stored [N, K]: identical fp32 sums, identical bits."""
    import torch
    forced(0, 0, 0)
    M, K, N = 512, 1024, 768
    a = to_dev(synth.bf16_normal(2, synth.STREAM_Q, (M, K)))
    b = to_dev(synth.bf16_normal(2, synth.STREAM_K, (K, N)))
    c1 = loom.loom_gemm_bf16(a, b)
    c2 = loom.loom_gemm_bf16(a, b.t().contiguous(), b_transposed=True)
    loom.loom_attn_check_error()
    assert torch.equal(c1.view(torch.int16), c2.view(torch.int16))


@pytest.mark.parametrize("group,k_alt", [(16, 1), (1, 1), (3, -1), (8, -1)])
@pytest.mark.parametrize("tile_n", [256, "pair"])
def test_tile_orders(loom, forced, group, k_alt, tile_n):
    """Other tile orders (rows per group, K walked backwards every other round) compute the
    same product: several rounds of tiles per CTA, a ragged K tail and ragged edges."""
    if tile_n == "pair":
        forced(0, 0, 1)
    else:
        forced(tile_n, 1)
    loom.loom_debug_gemm_order(group, k_alt)
    try:
        for M, K, N in [(4000, 328, 4096), (1000, 200, 2040)]:
            a, b = _inputs(M + group, M, K, N)
            _check(_run(loom, a, b), oracle.gemm(a, b), K, f"{M}x{K}x{N} group={group} k_alt={k_alt} {tile_n}")
    finally:
        loom.loom_debug_gemm_order(0, 0)


@pytest.mark.parametrize("M,K,N", [(2304, 200, 2304), (2300, 136, 2296), (520, 1000, 264)])
def test_pair_last_round_in_halves(loom, forced, M, K, N):
    """CTA pairs whose last round of tiles is thinly filled take those tiles as two 256 x 128
    halves (81 tiles on 76 pairs; few tiles): full tiles, then halves, ragged edges."""
    forced(0, 0, 1)
    a, b = _inputs(M + K, M, K, N)
    _check(_run(loom, a, b), oracle.gemm(a, b), K, f"{M}x{K}x{N} pair, halved last round")
    bt = np.ascontiguousarray(b.T)
    c = loom.loom_gemm_bf16(to_dev(a), to_dev(bt), b_transposed=True)
    loom.loom_attn_check_error()
    _check(c.float().cpu().numpy().astype(np.float64), oracle.gemm(a, b), K, f"{M}x{K}x{N} pair B^T")
