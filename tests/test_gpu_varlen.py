"""GPU parity of the ragged-batch (varlen) prefill (through the C ABI) against the fp64
oracle (``oracle.attention_varlen``), plus bit equality with the dense kernel when every
sequence has the same length (both load identical tiles and run identical arithmetic)."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import assert_parity, to_dev

pytestmark = pytest.mark.gpu


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


def case(seed, lq, lk, Hq, Hkv, D):
    cq = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    ck = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    q = synth.bf16_normal(seed, synth.STREAM_Q, (int(cq[-1]), Hq, D))
    k = synth.bf16_normal(seed, synth.STREAM_K, (max(int(ck[-1]), 1), Hkv, D))[:int(ck[-1])]
    v = synth.bf16_normal(seed, synth.STREAM_V, (max(int(ck[-1]), 1), Hkv, D))[:int(ck[-1])]
    return q, k, v, cq, ck


def run(loom, q, k, v, cq, ck, causal):
    import torch
    o, lse = loom.loom_attn_fwd_varlen(to_dev(q), to_dev(k), to_dev(v), torch.from_numpy(cq).cuda(),
                                       torch.from_numpy(ck).cuda(), int(np.diff(cq).max()), causal=causal,
                                       return_lse=True)
    loom.loom_attn_check_error()
    return o.float().cpu().numpy().astype(np.float64), lse.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("causal", [False, True], ids=["nc", "causal"])
@pytest.mark.parametrize("D", [64, 128])
def test_mixed_lengths(loom, D, causal):
    lens = [1, 127, 128, 129, 255, 256, 257, 700, 33]
    q, k, v, cq, ck = case(D + causal, lens, lens, 4, 2, D)
    o, lse = run(loom, q, k, v, cq, ck, causal)
    o_ref, lse_ref = oracle.attention_varlen(q, k, v, cq, ck, causal=causal)
    assert_parity(o, o_ref, lse, lse_ref, f"mixed D={D} causal={causal}")


@pytest.mark.parametrize("causal", [False, True], ids=["nc", "causal"])
def test_queries_and_keys_differ(loom, causal):
    """Per-sequence Sq != Skv, both ways (causal rows before Skv - Sq... see no key: O = 0,
    LSE = -inf), an empty query run, and a sequence without keys."""
    lq, lk = [100, 300, 5, 0, 64, 513], [300, 100, 5, 7, 0, 1000]
    q, k, v, cq, ck = case(7, lq, lk, 8, 8, 128)
    o, lse = run(loom, q, k, v, cq, ck, causal)
    o_ref, lse_ref = oracle.attention_varlen(q, k, v, cq, ck, causal=causal)
    assert_parity(o, o_ref, lse, lse_ref, f"q/k differ causal={causal}")


@pytest.mark.parametrize("G", [1, 4, 8])
def test_gqa(loom, G):
    lens = [300, 77, 1024]
    q, k, v, cq, ck = case(G, lens, lens, 2 * G, 2, 128)
    o, lse = run(loom, q, k, v, cq, ck, True)
    o_ref, lse_ref = oracle.attention_varlen(q, k, v, cq, ck, causal=True)
    assert_parity(o, o_ref, lse, lse_ref, f"G={G}")


@pytest.mark.parametrize("causal", [False, True], ids=["nc", "causal"])
@pytest.mark.parametrize("S", [384, 1000])
def test_equal_lengths_match_dense_kernel_bitwise(loom, S, causal):
    import torch
    B, H, D = 3, 4, 128
    q, k, v, cq, ck = case(S, [S] * B, [S] * B, H, H, D)
    o, lse = loom.loom_attn_fwd_varlen(to_dev(q), to_dev(k), to_dev(v), torch.from_numpy(cq).cuda(),
                                       torch.from_numpy(ck).cuda(), S, causal=causal, return_lse=True)
    loom.loom_attn_check_error()
    dense = [to_dev(np.ascontiguousarray(x.reshape(B, S, H, D).transpose(0, 2, 1, 3))) for x in (q, k, v)]
    od, ld = loom.loom_attn_fwd(*dense, causal=causal, return_lse=True)
    loom.loom_attn_check_error()
    od = od.permute(0, 2, 1, 3).reshape(B * S, H, D)
    ld = ld.permute(1, 0, 2).reshape(H, B * S)
    assert torch.equal(o.view(torch.int16), od.contiguous().view(torch.int16))
    assert torch.equal(lse, ld.contiguous())


def test_large_ragged_batch_full(loom):
    """12 sequences of U[512, 4096] tokens, Hq = 32, Hkv = 8, D = 128, causal: every row
    of O and LSE against the oracle."""
    rng = np.random.default_rng(3)
    lens = rng.integers(512, 4097, 12)
    Hq, Hkv, D = 32, 8, 128
    q, k, v, cq, ck = case(11, lens, lens, Hq, Hkv, D)
    o, lse = run(loom, q, k, v, cq, ck, True)
    o_ref, lse_ref = oracle.attention_varlen(q, k, v, cq, ck, causal=True)
    assert_parity(o, o_ref, lse, lse_ref, f"12 sequences, {int(cq[-1])} tokens")


def test_timeout_is_reported_and_context_survives(loom):
    import torch
    lens = [600, 300]
    q, k, v, cq, ck = case(5, lens, lens, 4, 4, 128)
    args = (to_dev(q), to_dev(k), to_dev(v), torch.from_numpy(cq).cuda(), torch.from_numpy(ck).cuda(), 600)
    loom.loom_attn_check_error()
    loom.loom_debug_set_timeout_ns(50_000_000)
    try:
        loom.loom_debug_inject(2)
        loom.loom_attn_fwd_varlen(*args, causal=True)
        with pytest.raises(loom.LoomError) as e:
            loom.loom_attn_check_error()
        assert e.value.status == 6
    finally:
        loom.loom_debug_inject(0)
        loom.loom_debug_set_timeout_ns(0)
    o, lse = loom.loom_attn_fwd_varlen(*args, causal=True, return_lse=True)
    loom.loom_attn_check_error()
    o_ref, lse_ref = oracle.attention_varlen(q, k, v, cq, ck, causal=True)
    assert_parity(o.float().cpu().numpy(), o_ref, lse.cpu().numpy(), lse_ref, "after timeout")


@pytest.mark.parametrize("causal", [False, True], ids=["nc", "causal"])
def test_many_short_sequences(loom, causal):
    """300 sequences of 0-300 tokens (many empty or single-token), D = 64: the sequence
    cursor steps over empty runs and items never cross a sequence."""
    rng = np.random.default_rng(17)
    lens = rng.integers(0, 301, 300)
    lens[rng.integers(0, 300, 40)] = 0
    lens[rng.integers(0, 300, 40)] = 1
    q, k, v, cq, ck = case(23, lens, lens, 4, 1, 64)
    o, lse = run(loom, q, k, v, cq, ck, causal)
    o_ref, lse_ref = oracle.attention_varlen(q, k, v, cq, ck, causal=causal)
    assert_parity(o, o_ref, lse, lse_ref, f"300 short sequences causal={causal}")


def test_cross_attention_lengths(loom):
    """Every sequence has its own query and key counts (cross attention, non-causal)."""
    rng = np.random.default_rng(29)
    lq = rng.integers(1, 700, 10)
    lk = rng.integers(1, 1500, 10)
    q, k, v, cq, ck = case(31, lq, lk, 8, 2, 128)
    o, lse = run(loom, q, k, v, cq, ck, False)
    o_ref, lse_ref = oracle.attention_varlen(q, k, v, cq, ck, causal=False)
    assert_parity(o, o_ref, lse, lse_ref, "cross attention")
