"""GPU parity of the kernel variants compiled for the block-size ablation: every neighbour
of the analytic model's ring depth or stage plan that the ablation measures computes the
same attention (or product) as the model's choice, checked against the fp64 oracle."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import assert_parity, o_to_f64, to_dev

pytestmark = pytest.mark.gpu

DECODE_PLANS = [(32, 2, 2), (32, 3, 2), (32, 4, 2), (64, 2, 2), (64, 4, 1), (128, 2, 1), (128, 3, 1)]


@pytest.fixture(scope="module")
def loom():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_29219_gb300 as m
    yield m
    m.loom_debug_prefill_slots(64, 0)
    m.loom_debug_decode_stage_plan(0)
    m.loom_debug_gemm_stages(0)
    m.loom_debug_gemm_cta_pair(0)
    m.loom_debug_gemm_tile_n(0)
    m.loom_debug_gemm_splits(0)


def _qkv(seed, B, Hq, Hkv, Sq, Skv, D):
    return (synth.bf16_normal(seed, synth.STREAM_Q, (B, Hq, Sq, D)),
            synth.bf16_normal(seed, synth.STREAM_K, (B, Hkv, Skv, D)),
            synth.bf16_normal(seed, synth.STREAM_V, (B, Hkv, Skv, D)))


@pytest.mark.parametrize("D,slots", [(128, 2), (64, 3), (64, 6), (64, 9)])
@pytest.mark.parametrize("causal", [False, True])
def test_prefill_ring_depths(loom, D, slots, causal):
    assert loom.loom_debug_prefill_slots(D, slots)
    try:
        for S, Hq, Hkv in [(515, 4, 1), (1100, 2, 2)]:
            q, k, v = _qkv(S + slots, 2, Hq, Hkv, S, S, D)
            o, lse = loom.loom_attn_fwd(to_dev(q), to_dev(k), to_dev(v), causal=causal, return_lse=True)
            loom.loom_attn_check_error()
            o_ref, lse_ref = oracle.attention(q, k, v, causal=causal)
            assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"D={D} slots={slots} S={S}")
    finally:
        loom.loom_debug_prefill_slots(D, 0)


def test_prefill_rejects_depths_not_compiled(loom):
    assert not loom.loom_debug_prefill_slots(128, 4)   # does not fit in shared memory
    assert not loom.loom_debug_prefill_slots(64, 11)
    assert loom.loom_debug_prefill_slots(128, 0)


@pytest.mark.parametrize("plan", DECODE_PLANS, ids=[f"t{t}s{s}c{c}" for t, s, c in DECODE_PLANS])
def test_decode_stage_plans(loom, plan):
    import torch
    assert loom.loom_debug_decode_stage_plan(*plan)
    try:
        B, Hq, Hkv, Skv, D = 6, 8, 2, 3000, 128
        q = synth.bf16_normal(4, synth.STREAM_Q, (B, Hq, 1, D))
        k = synth.bf16_normal(4, synth.STREAM_K, (B, Hkv, Skv, D))
        v = synth.bf16_normal(4, synth.STREAM_V, (B, Hkv, Skv, D))
        lens = np.array([0, 1, 33, 65, 2999, 3000], np.int32)
        o_ref, lse_ref = oracle.attention(q, k, v, seqlens_k=lens)
        sl = torch.from_numpy(lens).cuda()
        for splits in (1, 3, 16):
            o, lse = loom.loom_attn_decode(to_dev(q), to_dev(k), to_dev(v), sl, num_splits=splits, return_lse=True)
            loom.loom_attn_check_error()
            assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"plan={plan} splits={splits}")
    finally:
        loom.loom_debug_decode_stage_plan(0)


def test_decode_rejects_plans_not_compiled(loom):
    assert not loom.loom_debug_decode_stage_plan(64, 4, 2)  # 128 KB rings: one CTA per SM only
    assert loom.loom_debug_decode_stage_plan(0)


def _gemm_check(loom, M, K, N, what):
    a = synth.bf16_normal(M + N, synth.STREAM_Q, (M, K))
    b = synth.bf16_normal(M + N, synth.STREAM_K, (K, N))
    c = loom.loom_gemm_bf16(to_dev(a), to_dev(b))
    loom.loom_attn_check_error()
    c = c.float().cpu().numpy().astype(np.float64)
    ref = oracle.gemm(a, b)
    bound = 2.0 ** -8 * np.abs(ref) + 1e-6 * K + 1e-6
    assert np.all(np.abs(c - ref) <= bound), what


@pytest.mark.parametrize("kernel,stages", [("pair", 5), (256, 3), (128, 5)])
def test_gemm_ring_depths(loom, kernel, stages):
    if kernel == "pair":
        loom.loom_debug_gemm_cta_pair(1)
    else:
        loom.loom_debug_gemm_cta_pair(-1)
        loom.loom_debug_gemm_tile_n(kernel)
        loom.loom_debug_gemm_splits(1)
    loom.loom_debug_gemm_stages(stages)
    try:
        for M, K, N in [(1000, 1000, 1000), (300, 4096, 520), (2048, 256, 768)]:
            _gemm_check(loom, M, K, N, f"{kernel} stages={stages} {M}x{K}x{N}")
    finally:
        loom.loom_debug_gemm_stages(0)
        loom.loom_debug_gemm_cta_pair(0)
        loom.loom_debug_gemm_tile_n(0)
        loom.loom_debug_gemm_splits(0)
