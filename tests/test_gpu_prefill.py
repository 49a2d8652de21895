"""GPU parity of the prefill kernel (through the C ABI) against the fp64 oracle."""
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


@pytest.fixture(autouse=True, params=[2, 1, 3, 4], ids=["two_tiles", "one_tile_double_s", "s_ring", "three_tiles"])
def design(request, loom):
    """Run every prefill test with each kernel design: two alternating query tiles; one
    query tile with S double-buffered in TMEM; two query tiles sharing a ring of three S
    buffers; three alternating query tiles over 96-key KV tiles (the last two D = 64 only:
    at D = 128 the call runs the two-tile design)."""
    loom.loom_debug_prefill_design(request.param)
    yield request.param
    loom.loom_debug_prefill_design(0)


def _inputs(seed, B, Hq, Hkv, Sq, Skv, D):
    return (synth.bf16_normal(seed, synth.STREAM_Q, (B, Hq, Sq, D)),
            synth.bf16_normal(seed, synth.STREAM_K, (B, Hkv, Skv, D)),
            synth.bf16_normal(seed, synth.STREAM_V, (B, Hkv, Skv, D)))


def _run(loom, q, k, v, causal, scale=None):
    o, lse = loom.loom_attn_fwd(to_dev(q), to_dev(k), to_dev(v), causal=causal, scale=scale,
                                return_lse=True)
    loom.loom_attn_check_error()
    return o, lse


@pytest.mark.parametrize("causal", [False, True])
def test_tiny_config(loom, causal):
    # B=1, H=2, Sq=Skv=128, D=64, seed 0
    q, k, v = _inputs(0, 1, 2, 2, 128, 128, 64)
    o, lse = _run(loom, q, k, v, causal)
    o_ref, lse_ref = oracle.attention(q, k, v, causal=causal)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"tiny causal={causal}")


def test_tiny_config_matches_golden_rows(loom):
    # the stored oracle rows of tests/golden/tiny_attention_seed0.txt
    import os
    import sys
    here = os.path.dirname(os.path.abspath(__file__))
    sys.path.insert(0, os.path.join(here, "golden"))
    import make_golden
    from tests.test_golden import load
    _, rows = load()
    q, k, v = make_golden.inputs()
    for causal in (False, True):
        o, lse = _run(loom, q, k, v, causal)
        o = o_to_f64(o)
        lse = lse.cpu().numpy()
        for c, h, r, vals in rows:
            if c != int(causal):
                continue
            assert abs(lse[0, h, r] - vals[0]) <= 1e-3, (causal, h, r)
            got = [o[0, h, r, col] for col in make_golden.COLS]
            assert np.max(np.abs(np.asarray(got) - np.asarray(vals[1:]))) <= 2e-2, (causal, h, r)


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("causal", [False, True])
@pytest.mark.parametrize("S", [1, 127, 129, 255, 257, 384, 515])
def test_ragged_lengths(loom, D, causal, S):
    q, k, v = _inputs(S + D, 1, 2, 1, S, S, D)
    o, lse = _run(loom, q, k, v, causal)
    o_ref, lse_ref = oracle.attention(q, k, v, causal=causal)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"S={S} D={D} causal={causal}")


@pytest.mark.parametrize("Hq,Hkv", [(1, 1), (4, 1), (8, 2), (4, 4), (6, 3)])
def test_gqa_and_batches(loom, Hq, Hkv):
    q, k, v = _inputs(Hq * 10 + Hkv, 3, Hq, Hkv, 200, 200, 128)
    for causal in (False, True):
        o, lse = _run(loom, q, k, v, causal)
        o_ref, lse_ref = oracle.attention(q, k, v, causal=causal)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"Hq={Hq} Hkv={Hkv} causal={causal}")


@pytest.mark.parametrize("Sq,Skv", [(100, 300), (256, 1000), (1, 700), (300, 301)])
def test_more_keys_than_queries(loom, Sq, Skv):
    q, k, v = _inputs(Sq + Skv, 2, 4, 2, Sq, Skv, 128)
    for causal in (False, True):
        o, lse = _run(loom, q, k, v, causal)
        o_ref, lse_ref = oracle.attention(q, k, v, causal=causal)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"Sq={Sq} Skv={Skv} causal={causal}")


def test_scale_and_large_scores(loom):
    # a large scale makes the row max jump between tiles (exercises the O rescale path)
    q, k, v = _inputs(77, 1, 2, 2, 300, 900, 64)
    for scale in (0.02, 0.5, 1.3):
        o, lse = _run(loom, q, k, v, False, scale=scale)
        o_ref, lse_ref = oracle.attention(q, k, v, scale=scale)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"scale={scale}")


def test_increasing_scores_force_rescales(loom):
    # keys grow along the sequence so every KV tile raises the running max
    B, H, S, D = 1, 1, 256, 64
    q = synth.f32_to_bf16(np.full((B, H, S, D), 0.5, np.float32))
    ramp = np.linspace(0.0, 4.0, S, dtype=np.float32)[None, None, :, None]
    k = synth.f32_to_bf16(np.broadcast_to(ramp, (B, H, S, D)).copy())
    v = synth.bf16_normal(5, synth.STREAM_V, (B, H, S, D))
    o, lse = _run(loom, q, k, v, False, scale=1.0)
    o_ref, lse_ref = oracle.attention(q, k, v, scale=1.0)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, "ramp")


@pytest.mark.parametrize("B,H,S", [(4, 32, 2048), (1, 16, 8192), (1, 3, 1000), (2, 64, 512)])
def test_causal_work_order_covers_every_row(loom, B, H, S):
    # the causal work order (blocks of planes aligned to round pairs, a merged final
    # block) must hand out every (plane, query tile) exactly once: O and LSE start as NaN
    # and no NaN may survive
    import torch
    D = 128
    q = torch.randn(B, H, S, D, device="cuda").to(torch.bfloat16)
    o = torch.full_like(q, float("nan"))
    lse = torch.full((B, H, S), float("nan"), device="cuda")
    loom.loom_attn_fwd(q, q, q, o, lse, causal=True)
    loom.loom_attn_check_error()
    assert torch.isfinite(o.float()).all() and torch.isfinite(lse).all()


# The full-size configurations are compared on every row of O and LSE.  Their inputs and
# the oracle's results are computed once per configuration and shared by the three
# prefill designs (the oracle takes ~3-10 s per configuration on the host cores).
_FULL = {}


def _full_case(B, Hq, Hkv, S, D, causal):
    key = (B, Hq, Hkv, S, D, causal)
    if key not in _FULL:
        q, k, v = _inputs(0, B, Hq, Hkv, S, S, D)
        o_ref, lse_ref = oracle.attention(q, k, v, causal=causal)
        _FULL[key] = (q, k, v, o_ref, lse_ref)
    return _FULL[key]


@pytest.mark.slow
@pytest.mark.parametrize("causal", [False, True])
def test_prefill_config_full_size(loom, causal):
    # B=4, Hq=Hkv=32, Sq=Skv=2048, D=128 (the benchmarked prefill workload), all rows
    q, k, v, o_ref, lse_ref = _full_case(4, 32, 32, 2048, 128, causal)
    o, lse = _run(loom, q, k, v, causal)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"B4 H32 S2048 causal={causal}")


@pytest.mark.slow
@pytest.mark.parametrize("Hq,Hkv,D", [(32, 8, 128), (64, 16, 64)])
def test_long_prefill_full_size(loom, Hq, Hkv, D):
    # B=1, S=8192, causal, GQA group 4, all rows
    q, k, v, o_ref, lse_ref = _full_case(1, Hq, Hkv, 8192, D, True)
    o, lse = _run(loom, q, k, v, True)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"S8192 Hq={Hq} Hkv={Hkv} D={D}")
