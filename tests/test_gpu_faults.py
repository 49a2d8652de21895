"""Failure detection without a GPU fault.

Every mbarrier wait in the kernels is bounded by %globaltimer.  The host-side test hook
loom_debug_inject makes a kernel's loader skip one copy, so that the waits on it run out;
the kernel then unwinds (drains the copies it issued, waits for its issued MMAs, frees
TMEM) and sets the device error word.  These tests check that loom_attn_check_error
reports LOOM_ERR_TIMEOUT and that the context stays usable: the very next normal call
matches the oracle and reports no error.
"""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import assert_parity, o_to_f64, to_dev

pytestmark = pytest.mark.gpu

TIMEOUT_NS = 50_000_000  # 50 ms per wait while the hook is on


@pytest.fixture(scope="module")
def loom():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_29219_gb300 as m
    yield m
    m.loom_debug_inject(0)
    m.loom_debug_set_timeout_ns(0)


def _expect_timeout(loom, call):
    loom.loom_attn_check_error()  # nothing pending
    loom.loom_debug_set_timeout_ns(TIMEOUT_NS)
    try:
        call()
        with pytest.raises(loom.LoomError) as e:
            loom.loom_attn_check_error()
        assert e.value.status == 6, e.value
    finally:
        loom.loom_debug_inject(0)
        loom.loom_debug_set_timeout_ns(0)
    loom.loom_attn_check_error()  # the word was cleared


@pytest.mark.parametrize("tensor_cores", [1, 2, 0], ids=["tc_persistent", "tc_per_split", "cuda_core"])
def test_decode_skipped_stage_times_out_and_context_survives(loom, tensor_cores):
    """The split kernel on the tensor cores (persistent, or one CTA per split) and on the
    CUDA cores: a stage whose copy is never issued times out, the kernel returns (its
    copies and MMAs drained, TMEM released) and the next call is correct."""
    B, Hq, Hkv, Skv, D = 1, 4, 1, 2048, 128  # one split of 32 stages, one CTA
    q = synth.bf16_normal(31, synth.STREAM_Q, (B, Hq, 1, D))
    k = synth.bf16_normal(31, synth.STREAM_K, (B, Hkv, Skv, D))
    v = synth.bf16_normal(31, synth.STREAM_V, (B, Hkv, Skv, D))
    qd, kd, vd = to_dev(q), to_dev(k), to_dev(v)

    def bad():
        loom.loom_debug_inject(1)
        loom.loom_attn_decode(qd, kd, vd, None, num_splits=1)

    loom.loom_debug_decode_tensor_cores(tensor_cores)
    try:
        _expect_timeout(loom, bad)
        o, lse = loom.loom_attn_decode(qd, kd, vd, None, num_splits=1, return_lse=True)
        loom.loom_attn_check_error()
    finally:
        loom.loom_debug_decode_tensor_cores(1)
    o_ref, lse_ref = oracle.attention(q, k, v)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, "decode after timeout")


@pytest.mark.parametrize("lens,splits", [(2048, 2), (160, 2)], ids=["all_items_abort", "one_item_aborts"])
def test_persistent_decode_skipped_stage_times_out_and_context_survives(loom, lens, splits):
    """The persistent split kernel: the CTA whose second stage is never filled gives up on
    it and unwinds; the next call on the same context is correct."""
    import torch
    B, Hq, Hkv, Skv, D = 1, 4, 1, 2048, 128
    q = synth.bf16_normal(38, synth.STREAM_Q, (B, Hq, 1, D))
    k = synth.bf16_normal(38, synth.STREAM_K, (B, Hkv, Skv, D))
    v = synth.bf16_normal(38, synth.STREAM_V, (B, Hkv, Skv, D))
    qd, kd, vd = to_dev(q), to_dev(k), to_dev(v)
    sl_h = np.array([lens], np.int32)
    sl = torch.from_numpy(sl_h).cuda()
    loom.loom_debug_decode_form(2)
    try:
        assert loom.loom_attn_decode_form(B, Hq, Hkv, Skv, D, splits)[0] == 2

        def bad():
            loom.loom_debug_inject(1)
            loom.loom_attn_decode(qd, kd, vd, sl, num_splits=splits)

        _expect_timeout(loom, bad)
        o, lse = loom.loom_attn_decode(qd, kd, vd, sl, num_splits=splits, return_lse=True)
        loom.loom_attn_check_error()
    finally:
        loom.loom_debug_decode_form(0)
    o_ref, lse_ref = oracle.attention(q, k, v, seqlens_k=sl_h)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, "persistent decode after timeout")


@pytest.mark.parametrize("lens,splits", [(2048, 2), (160, 2), (2048, 16)], ids=["both_abort", "one_aborts", "c16"])
def test_cluster_decode_skipped_stage_times_out_and_context_survives(loom, lens, splits):
    """The single-kernel cluster form (one cluster of `splits` CTAs): every CTA with a
    second stage gives up on it and unwinds; its peers give up on the partial it never
    signals; all CTAs still meet at the final cluster barrier, so the launch ends and the
    next call is correct."""
    import torch
    B, Hq, Hkv, Skv, D = 1, 4, 1, 2048, 128
    q = synth.bf16_normal(37, synth.STREAM_Q, (B, Hq, 1, D))
    k = synth.bf16_normal(37, synth.STREAM_K, (B, Hkv, Skv, D))
    v = synth.bf16_normal(37, synth.STREAM_V, (B, Hkv, Skv, D))
    qd, kd, vd = to_dev(q), to_dev(k), to_dev(v)
    sl_h = np.array([lens], np.int32)
    sl = torch.from_numpy(sl_h).cuda()
    loom.loom_debug_decode_form(3, splits)
    try:
        assert loom.loom_attn_decode_form(B, Hq, Hkv, Skv, D, splits) == (3, splits)

        def bad():
            loom.loom_debug_inject(1)
            loom.loom_attn_decode(qd, kd, vd, sl, num_splits=splits)

        _expect_timeout(loom, bad)
        o, lse = loom.loom_attn_decode(qd, kd, vd, sl, num_splits=splits, return_lse=True)
        loom.loom_attn_check_error()
    finally:
        loom.loom_debug_decode_form(0)
    o_ref, lse_ref = oracle.attention(q, k, v, seqlens_k=sl_h)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, "cluster decode after timeout")


@pytest.mark.parametrize("design,D", [(2, 128), (1, 128), (1, 64), (3, 64), (4, 64)])
def test_prefill_skipped_tile_times_out_and_context_survives(loom, design, D):
    loom.loom_debug_prefill_design(design)
    try:
        _prefill_fault_case(loom, D)
    finally:
        loom.loom_debug_prefill_design(0)


def _prefill_fault_case(loom, D):
    B, H, S = 1, 2, 512  # 2 to 4 work items, each with 4 KV tiles
    q = synth.bf16_normal(32, synth.STREAM_Q, (B, H, S, D))
    k = synth.bf16_normal(32, synth.STREAM_K, (B, H, S, D))
    v = synth.bf16_normal(32, synth.STREAM_V, (B, H, S, D))
    qd, kd, vd = to_dev(q), to_dev(k), to_dev(v)

    def bad():
        loom.loom_debug_inject(2)
        loom.loom_attn_fwd(qd, kd, vd)

    _expect_timeout(loom, bad)
    for causal in (False, True):
        o, lse = loom.loom_attn_fwd(qd, kd, vd, causal=causal, return_lse=True)
        loom.loom_attn_check_error()
        o_ref, lse_ref = oracle.attention(q, k, v, causal=causal)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"prefill after timeout causal={causal}")


def test_no_false_timeouts_under_default_limit(loom):
    # a full-size call with the default 2 s limit never trips the error word
    B, H, S, D = 4, 32, 2048, 128
    import torch
    q = torch.randn(B, H, S, D, device="cuda").to(torch.bfloat16)
    for causal in (False, True):
        loom.loom_attn_fwd(q, q, q, causal=causal)
    loom.loom_attn_check_error()


@pytest.mark.parametrize("tensor_cores", [1, 0], ids=["tc_persistent", "cuda_core"])
def test_paged_decode_skipped_stage_times_out_and_context_survives(loom, tensor_cores):
    """The split kernel over a paged cache (64-key pages, in a shuffled order): a stage
    whose copies are never issued times out, the kernel unwinds, and the next call on the
    same context matches the oracle."""
    import torch
    B, Hq, Hkv, P, D = 2, 8, 2, 64, 128
    lens = np.array([1000, 333], np.int32)
    npg = [(int(n) + P - 1) // P for n in lens]
    max_pages = max(npg)
    kc = synth.bf16_normal(41, synth.STREAM_K, (sum(npg), P, Hkv, D))
    vc = synth.bf16_normal(41, synth.STREAM_V, (sum(npg), P, Hkv, D))
    q = synth.bf16_normal(41, synth.STREAM_Q, (B, Hq, 1, D))
    order = np.random.default_rng(41).permutation(sum(npg)).astype(np.int32)
    table = np.full((B, max_pages), -1, np.int32)
    table[0, :npg[0]] = order[:npg[0]]
    table[1, :npg[1]] = order[npg[0]:]
    qd, kd, vd = to_dev(q), to_dev(kc), to_dev(vc)
    td, sl = torch.from_numpy(table).cuda(), torch.from_numpy(lens).cuda()
    loom.loom_debug_decode_tensor_cores(tensor_cores)
    try:
        def bad():
            loom.loom_debug_inject(1)
            loom.loom_attn_decode_paged(qd, kd, vd, td, sl, num_splits=2)

        _expect_timeout(loom, bad)
        o, lse = loom.loom_attn_decode_paged(qd, kd, vd, td, sl, num_splits=2, return_lse=True)
        loom.loom_attn_check_error()
    finally:
        loom.loom_debug_decode_tensor_cores(1)
    o_ref, lse_ref = oracle.decode_paged(q, kc, vc, table, lens, page_size=P)
    assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, "paged decode after timeout")
