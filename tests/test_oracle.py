"""Pins for the fp64 oracle, checked against facts the mathematics fixes.

The paper prints no attention values, so every pin here is a closed form, an
invariant, a special case that reduces to a library routine, or brute force with an
independent naive formula.  Each is chosen so that a plausible slip in the oracle
(a dropped scale, a transposed operand, a wrong GQA head map, a wrong causal offset,
a missing max subtraction, a wrong merge weight) fails at least one of them.
"""
import numpy as np
import pytest
from scipy.special import logsumexp, softmax

import synth

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _inputs(seed, B, Hq, Hkv, Sq, Skv, D):
    q = synth.bf16_normal(seed, synth.STREAM_Q, (B, Hq, Sq, D))
    k = synth.bf16_normal(seed, synth.STREAM_K, (B, Hkv, Skv, D))
    v = synth.bf16_normal(seed, synth.STREAM_V, (B, Hkv, Skv, D))
    return q, k, v


def _f64(bits):
    return synth.bf16_to_f32(bits).astype(np.float64)


def _const_bits(value, shape):
    return np.full(shape, synth.f32_to_bf16(np.array([value], np.float32))[0], dtype=np.uint16)


def _scipy_attention(q, k, v, causal, scale, seqlens=None):
    """Library-routine restatement: scipy softmax / logsumexp on explicit score matrices."""
    qf, kf, vf = _f64(q), _f64(k), _f64(v)
    B, Hq, Sq, D = qf.shape
    Hkv, Skv = kf.shape[1], kf.shape[2]
    G = Hq // Hkv
    kf = np.repeat(kf, G, axis=1)  # head h reads kv head h // G
    vf = np.repeat(vf, G, axis=1)
    s = scale * np.einsum("bhid,bhjd->bhij", qf, kf)
    o = np.zeros_like(qf)
    lse = np.full((B, Hq, Sq), -np.inf)
    for b in range(B):
        length = Skv if seqlens is None else int(seqlens[b])
        mask = np.zeros((Sq, Skv), bool)
        mask[:, :length] = True
        if causal:  # bottom-right aligned: key j visible to query i iff j <= i + (len - Sq)
            mask &= np.tril(np.ones((Sq, Skv), bool), k=length - Sq)
        for h in range(Hq):
            sb = np.where(mask, s[b, h], -np.inf)
            for i in range(Sq):
                if not mask[i].any():
                    continue
                o[b, h, i] = softmax(sb[i]) @ vf[b, h]
                lse[b, h, i] = logsumexp(sb[i])
    return o, lse


@pytest.mark.parametrize("B,Hq,Hkv,Sq,Skv,D,causal", [
    (1, 2, 2, 5, 7, 8, False),
    (2, 4, 1, 6, 6, 16, True),
    (1, 4, 2, 3, 9, 8, True),     # Sq < Skv: bottom-right causal offset
    (2, 8, 2, 17, 33, 32, False),
    (1, 2, 1, 33, 40, 64, True),
])
def test_matches_scipy_softmax(oracle_mod, B, Hq, Hkv, Sq, Skv, D, causal):
    q, k, v = _inputs(1, B, Hq, Hkv, Sq, Skv, D)
    scale = 1.0 / np.sqrt(D)
    o, lse = oracle_mod.attention(q, k, v, causal=causal, scale=scale)
    o_ref, lse_ref = _scipy_attention(q, k, v, causal, scale)
    np.testing.assert_allclose(o, o_ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lse_ref, rtol=0, atol=1e-12)


@pytest.mark.parametrize("causal", [False, True])
def test_brute_force_naive_long_double(oracle_mod, causal):
    for seed, (B, Hq, Hkv, Sq, Skv, D) in enumerate([(1, 1, 1, 1, 1, 4), (1, 2, 1, 4, 8, 4),
                                                     (2, 4, 2, 8, 8, 8), (1, 3, 3, 5, 7, 6)]):
        q, k, v = _inputs(seed + 10, B, Hq, Hkv, Sq, Skv, D)
        o, lse = oracle_mod.attention(q, k, v, causal=causal)
        o_n, lse_n = oracle_mod.attention_naive(q, k, v, causal=causal)
        np.testing.assert_allclose(o, o_n, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, lse_n, rtol=0, atol=1e-12)


def test_rows_sum_to_one(oracle_mod):
    # V = 1 everywhere: every output element is the row's probability mass.
    q, k, _ = _inputs(2, 2, 4, 2, 19, 23, 16)
    ones = _const_bits(1.0, k.shape)
    for causal in (False, True):
        o, _ = oracle_mod.attention(q, k, ones, causal=causal)
        np.testing.assert_allclose(o, 1.0, rtol=0, atol=1e-12)


def test_constant_value_row_is_returned(oracle_mod):
    q, k, v = _inputs(3, 1, 2, 1, 11, 29, 32)
    row = v[0, 0, 5]
    vc = np.broadcast_to(row, v.shape).copy()
    o, _ = oracle_mod.attention(q, k, vc)
    np.testing.assert_allclose(o, np.broadcast_to(_f64(row), o.shape), rtol=0, atol=1e-12)


def test_single_key(oracle_mod):
    q, k, v = _inputs(4, 2, 4, 2, 7, 1, 64)
    scale = 0.37
    o, lse = oracle_mod.attention(q, k, v, scale=scale)
    G = 2
    for h in range(4):
        np.testing.assert_array_equal(o[:, h], np.broadcast_to(_f64(v[:, h // G, 0])[:, None, :], o[:, h].shape))
        dots = np.einsum("bid,bd->bi", _f64(q[:, h]), _f64(k[:, h // G, 0]))
        np.testing.assert_allclose(lse[:, h], scale * dots, rtol=0, atol=1e-12)


def test_causal_first_query_sees_only_key0(oracle_mod):
    q, k, v = _inputs(5, 1, 2, 2, 16, 16, 32)
    o, lse = oracle_mod.attention(q, k, v, causal=True)
    np.testing.assert_array_equal(o[:, :, 0], _f64(v[:, :, 0]))
    dots = np.einsum("bhd,bhd->bh", _f64(q[:, :, 0]), _f64(k[:, :, 0]))
    np.testing.assert_allclose(lse[:, :, 0], dots / np.sqrt(32), rtol=0, atol=1e-12)
    # the last query sees every key, i.e. equals the non-causal result
    o_nc, lse_nc = oracle_mod.attention(q, k, v, causal=False)
    np.testing.assert_allclose(o[:, :, -1], o_nc[:, :, -1], rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse[:, :, -1], lse_nc[:, :, -1], rtol=0, atol=1e-13)


def test_zero_scale_and_zero_query_give_mean_of_values(oracle_mod):
    q, k, v = _inputs(6, 1, 2, 2, 9, 13, 16)
    for qq, scale in ((q, 0.0), (np.zeros_like(q), 0.125)):
        for causal in (False, True):
            o, lse = oracle_mod.attention(qq, k, v, causal=causal, scale=scale)
            for i in range(9):
                n = 13 if not causal else i + 13 - 9 + 1
                np.testing.assert_allclose(o[0, :, i], _f64(v[0, :, :n]).mean(axis=1), rtol=0, atol=1e-12)
                np.testing.assert_allclose(lse[0, :, i], np.log(n), rtol=0, atol=1e-12)


def test_hard_attention_limit_needs_max_subtraction(oracle_mod):
    # With a huge scale the softmax becomes one-hot on the largest score; exp(s) alone
    # would overflow to inf/inf = nan.
    q, k, v = _inputs(7, 1, 1, 1, 4, 50, 16)
    scale = 1e4
    o, lse = oracle_mod.attention(q, k, v, scale=scale)
    dots = _f64(q[0, 0]) @ _f64(k[0, 0]).T
    best = dots.argmax(axis=1)
    second = np.sort(dots, axis=1)[:, -2]
    assert np.all(scale * (dots.max(axis=1) - second) > 50)  # gap makes the one-hot exact in fp64
    np.testing.assert_allclose(o[0, 0], _f64(v[0, 0])[best], rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse[0, 0], scale * dots.max(axis=1), rtol=1e-15, atol=1e-9)


def test_key_permutation_invariance(oracle_mod):
    q, k, v = _inputs(8, 2, 4, 2, 12, 37, 32)
    perm = np.random.default_rng(0).permutation(37)
    o, lse = oracle_mod.attention(q, k, v)
    o_p, lse_p = oracle_mod.attention(q, k[:, :, perm], v[:, :, perm])
    np.testing.assert_allclose(o, o_p, rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse, lse_p, rtol=0, atol=1e-13)


def test_duplicated_keys_shift_lse_by_ln2(oracle_mod):
    q, k, v = _inputs(9, 1, 2, 1, 10, 21, 16)
    o, lse = oracle_mod.attention(q, k, v)
    o2, lse2 = oracle_mod.attention(q, np.concatenate([k, k], axis=2), np.concatenate([v, v], axis=2))
    np.testing.assert_allclose(o2, o, rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse2, lse + np.log(2.0), rtol=0, atol=1e-12)


def test_gqa_equals_repeated_kv_heads(oracle_mod):
    q, k, v = _inputs(10, 2, 8, 2, 6, 14, 16)
    o, lse = oracle_mod.attention(q, k, v, causal=True)
    o_r, lse_r = oracle_mod.attention(q, np.repeat(k, 4, axis=1), np.repeat(v, 4, axis=1), causal=True)
    np.testing.assert_array_equal(o, o_r)
    np.testing.assert_array_equal(lse, lse_r)


def test_row_sampling_matches_full(oracle_mod):
    q, k, v = _inputs(11, 2, 4, 2, 33, 47, 32)
    o, lse = oracle_mod.attention(q, k, v, causal=True)
    rows = np.array([0, 5, 32, 33, 100, 2 * 4 * 33 - 1])
    o_s, lse_s = oracle_mod.attention(q, k, v, causal=True, rows=rows)
    np.testing.assert_array_equal(o_s, o.reshape(-1, 32)[rows])
    np.testing.assert_array_equal(lse_s, lse.reshape(-1)[rows])


def test_empty_rows_are_zero_with_minus_inf_lse(oracle_mod):
    q, k, v = _inputs(12, 3, 2, 1, 1, 40, 16)
    lens = np.array([0, 1, 40], np.int32)
    o, lse = oracle_mod.attention(q, k, v, seqlens_k=lens)
    assert np.all(o[0] == 0) and np.all(np.isneginf(lse[0]))
    np.testing.assert_array_equal(o[1, :, 0], np.broadcast_to(_f64(v[1, 0, 0]), (2, 16)))
    assert np.all(np.isfinite(o)) and np.all(np.isfinite(lse[1:]))
    # causal with more queries than keys: the first Sq - Skv rows see nothing
    q2, k2, v2 = _inputs(13, 1, 1, 1, 6, 4, 8)
    o2, lse2 = oracle_mod.attention(q2, k2, v2, causal=True)
    assert np.all(o2[0, 0, :2] == 0) and np.all(np.isneginf(lse2[0, 0, :2]))
    np.testing.assert_array_equal(o2[0, 0, 2], _f64(v2[0, 0, 0]))


@pytest.mark.parametrize("chunk_align", [1, 64])
def test_split_merge_equals_unsplit_for_every_split_count(oracle_mod, chunk_align):
    B, Hq, Hkv, Skv, D = 2, 4, 2, 150, 32
    q, k, v = _inputs(14, B, Hq, Hkv, 1, Skv, D)
    lens = np.array([150, 97], np.int32)
    o_ref, lse_ref = oracle_mod.attention(q, k, v, seqlens_k=lens)
    for splits in range(1, 160, 7):
        o, lse, o_part, lse_part = oracle_mod.decode_split_merge(
            q, k, v, num_splits=splits, seqlens_k=lens, chunk_align=chunk_align)
        np.testing.assert_allclose(o, o_ref[:, :, 0], rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, lse_ref[:, :, 0], rtol=0, atol=1e-12)
        # partials of non-empty splits are themselves attention over their chunk
        c = oracle_mod.decode_chunk(97, splits, chunk_align)
        j0, j1 = 0, min(c, 97)
        o_c, lse_c = oracle_mod.attention(q[1:], k[1:, :, j0:j1], v[1:, :, j0:j1])
        np.testing.assert_allclose(o_part[1, :, 0], o_c[0, :, 0], rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse_part[1, :, 0], lse_c[0, :, 0], rtol=0, atol=1e-12)


def test_split_merge_edge_lengths(oracle_mod):
    B, Hq, Hkv, Skv, D = 5, 2, 1, 200, 16
    q, k, v = _inputs(15, B, Hq, Hkv, 1, Skv, D)
    lens = np.array([0, 1, 63, 65, 200], np.int32)  # empty, single key, chunk-1, chunk+1, full
    o_ref, lse_ref = oracle_mod.attention(q, k, v, seqlens_k=lens)
    for splits in (1, 2, 4, 16):
        o, lse, _, lse_part = oracle_mod.decode_split_merge(q, k, v, num_splits=splits, seqlens_k=lens)
        assert np.all(o[0] == 0) and np.all(np.isneginf(lse[0]))
        assert np.all(np.isneginf(lse_part[0]))
        np.testing.assert_allclose(o[1:], o_ref[1:, :, 0], rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse[1:], lse_ref[1:, :, 0], rtol=0, atol=1e-12)


def test_decode_chunk_rule(oracle_mod):
    assert oracle_mod.decode_chunk(0, 16, 64) == 0
    assert oracle_mod.decode_chunk(1, 16, 64) == 64
    assert oracle_mod.decode_chunk(4096, 16, 64) == 256
    assert oracle_mod.decode_chunk(4097, 16, 64) == 320
    assert oracle_mod.decode_chunk(131072, 19, 64) == 6912
    assert oracle_mod.decode_chunk(100, 7, 1) == 15


def test_generator_is_counter_based_and_normal():
    a = synth.bf16_normal(0, synth.STREAM_K, (1 << 23) + 1000)
    b = synth.bf16_normal(0, synth.STREAM_K, 1000, start=(1 << 23) - 500)
    np.testing.assert_array_equal(a[(1 << 23) - 500:(1 << 23) + 500], b)
    f = synth.bf16_to_f32(a).astype(np.float64)
    assert abs(f.mean()) < 2e-3 and abs(f.std() - 1) < 2e-3
    # bf16 rounding is round-to-nearest-even on the fp32 pattern
    x = np.array([1.0, 1.00390625, 1.01171875, -2.5, 3.0e38], np.float32)
    np.testing.assert_array_equal(synth.f32_to_bf16(x), np.array([0x3F80, 0x3F80, 0x3F82, 0xC020, 0x7F62], np.uint16))
    lens = synth.decode_lengths(0, 4096, 4096, 8192)
    assert lens.min() >= 4096 and lens.max() <= 8192
