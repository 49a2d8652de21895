"""Pins of the paged-KV decode oracle (``oracle.paged_gather`` + ``oracle.decode_paged``)
against what does not depend on it: a pure-Python brute force that walks the block table
key by key, the contiguous decode when the pages are laid out in order, the Flash Decode
split/merge form of the C++ oracle, invariance under a permutation of physical pages,
garbage in pages and rows that no sequence reaches, and empty sequences."""
import math

import numpy as np
import pytest

import oracle
import synth


def _paged_case(seed, B, Hq, Hkv, P, max_pages, lens, D=16, spare=3):
    """Random cache with pages dealt to sequences in a shuffled order, plus spare pages."""
    rng = np.random.default_rng(seed)
    need = [(int(n) + P - 1) // P for n in lens]
    npages = sum(need) + spare
    k_cache = synth.bf16_normal(seed, synth.STREAM_K, (npages, P, Hkv, D))
    v_cache = synth.bf16_normal(seed, synth.STREAM_V, (npages, P, Hkv, D))
    q = synth.bf16_normal(seed, synth.STREAM_Q, (B, Hq, 1, D))
    perm = rng.permutation(npages)
    table = np.full((B, max_pages), -7, dtype=np.int32)  # entries past a sequence's end: junk
    i = 0
    for b in range(B):
        table[b, :need[b]] = perm[i:i + need[b]]
        i += need[b]
    return q, k_cache, v_cache, table, np.asarray(lens, dtype=np.int32)


def _brute(q, k_cache, v_cache, table, lens, P, scale):
    """Per (b, h): walk keys t < len, fetch row t % P of page table[b][t // P], softmax."""
    B, Hq, _, D = q.shape
    Hkv = k_cache.shape[2]
    f = oracle.bf16_to_f64
    o = np.zeros((B, Hq, D))
    lse = np.full((B, Hq), -np.inf)
    for b in range(B):
        for h in range(Hq):
            hk = h // (Hq // Hkv)
            qv = [float(x) for x in f(q[b, h, 0])]
            scores, vals = [], []
            for t in range(int(lens[b])):
                page, row = int(table[b][t // P]), t % P
                kv = [float(x) for x in f(k_cache[page, row, hk])]
                scores.append(scale * sum(a * c for a, c in zip(qv, kv)))
                vals.append([float(x) for x in f(v_cache[page, row, hk])])
            if not scores:
                continue
            m = max(scores)
            w = [math.exp(s - m) for s in scores]
            z = sum(w)
            lse[b, h] = m + math.log(z)
            for d in range(D):
                o[b, h, d] = sum(wi * vi[d] for wi, vi in zip(w, vals)) / z
    return o, lse


@pytest.mark.parametrize("P,lens", [(4, [5, 12, 1]), (8, [16, 9, 0]), (16, [33, 16, 47])])
def test_matches_brute_force(P, lens):
    B, Hq, Hkv = 3, 4, 2
    max_pages = max((n + P - 1) // P for n in lens) + 1
    q, kc, vc, table, sl = _paged_case(P, B, Hq, Hkv, P, max_pages, lens)
    scale = 0.3
    o, lse = oracle.decode_paged(q, kc, vc, table, sl, page_size=P, scale=scale)
    ob, lb = _brute(q, kc, vc, table, sl, P, scale)
    np.testing.assert_allclose(o, ob, rtol=0, atol=1e-12)
    np.testing.assert_array_equal(np.isneginf(lse), np.isneginf(lb))
    fin = np.isfinite(lb)
    np.testing.assert_allclose(lse[fin], lb[fin], rtol=0, atol=1e-12)
    assert np.all(o[np.isneginf(lb)] == 0.0)


def test_in_order_pages_equal_contiguous_decode():
    """Pages dealt in order, one sequence after another, reproduce the contiguous cache;
    the result must equal the C++ oracle's Flash Decode split/merge form."""
    B, Hq, Hkv, P, S, D = 2, 8, 2, 16, 96, 32
    k = synth.bf16_normal(1, synth.STREAM_K, (B, Hkv, S, D))
    v = synth.bf16_normal(1, synth.STREAM_V, (B, Hkv, S, D))
    q = synth.bf16_normal(1, synth.STREAM_Q, (B, Hq, 1, D))
    npg = S // P
    kc = k.reshape(B, Hkv, npg, P, D).transpose(0, 2, 3, 1, 4).reshape(B * npg, P, Hkv, D).copy()
    vc = v.reshape(B, Hkv, npg, P, D).transpose(0, 2, 3, 1, 4).reshape(B * npg, P, Hkv, D).copy()
    table = np.arange(B * npg, dtype=np.int32).reshape(B, npg)
    lens = np.array([S, 70], dtype=np.int32)
    o, lse = oracle.decode_paged(q, kc, vc, table, lens, page_size=P, scale=0.2)
    o2, lse2, _, _ = oracle.decode_split_merge(q, k, v, num_splits=3, scale=0.2, seqlens_k=lens)
    np.testing.assert_allclose(o, o2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lse2, rtol=0, atol=1e-12)


def test_page_permutation_invariance():
    B, Hq, Hkv, P = 2, 4, 1, 8
    q, kc, vc, table, sl = _paged_case(5, B, Hq, Hkv, P, 6, [40, 23], D=32)
    o, lse = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
    perm = np.random.default_rng(9).permutation(kc.shape[0])
    inv = np.argsort(perm)
    t2 = table.copy()
    live = t2 >= 0
    t2[live] = inv[t2[live]]
    o2, lse2 = oracle.decode_paged(q, kc[perm], vc[perm], t2, sl, page_size=P)
    np.testing.assert_array_equal(o, o2)
    np.testing.assert_array_equal(lse, lse2)


def test_unreached_pages_and_rows_are_ignored():
    B, Hq, Hkv, P = 2, 2, 1, 8
    q, kc, vc, table, sl = _paged_case(7, B, Hq, Hkv, P, 4, [13, 8], D=16)
    o, lse = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
    kc2, vc2 = kc.copy(), vc.copy()
    used = set()
    for b in range(B):
        for j in range((int(sl[b]) + P - 1) // P):
            used.add(int(table[b, j]))
            kc2[table[b, j], int(sl[b]) - j * P:] = 0x7FC0  # NaN past the sequence's end
            vc2[table[b, j], int(sl[b]) - j * P:] = 0x7FC0
    for p in range(kc.shape[0]):
        if p not in used:
            kc2[p] = 0x7FC0
            vc2[p] = 0x7F80  # +inf
    o2, lse2 = oracle.decode_paged(q, kc2, vc2, table, sl, page_size=P)
    np.testing.assert_array_equal(o, o2)
    np.testing.assert_array_equal(lse, lse2)


def test_empty_sequence_and_bad_table():
    q, kc, vc, table, sl = _paged_case(3, 2, 2, 1, 8, 3, [0, 9], D=16)
    o, lse = oracle.decode_paged(q, kc, vc, table, sl, page_size=8)
    assert np.all(o[0] == 0.0) and np.all(np.isneginf(lse[0])) and np.all(np.isfinite(lse[1]))
    bad = table.copy()
    bad[1, 1] = kc.shape[0]
    with pytest.raises(ValueError):
        oracle.decode_paged(q, kc, vc, bad, sl, page_size=8)


def _mutant_gather(kind):
    def gather(cache, block_table, seqlens, page_size, layout="nhd"):
        cache = np.asarray(cache, dtype=np.uint16)
        table = np.asarray(block_table, dtype=np.int64)
        npages, P, Hkv, D = cache.shape
        B, max_pages = table.shape
        out = np.zeros((B, Hkv, max_pages * P, D), dtype=np.uint16)
        for b in range(B):
            for t in range(int(seqlens[b])):
                page = int(table[b, t // P]) if kind != "page_mod" else int(table[b, t % max_pages])
                row = t % P if kind != "row_div" else (t // P) % P
                if kind == "head_row_swap":
                    out[b, :, t, :] = cache[page, :, row % Hkv, :][:Hkv] if P >= Hkv else 0
                else:
                    out[b, :, t, :] = cache[page, row]
        return out
    return gather


@pytest.mark.parametrize("kind", ["page_mod", "row_div", "head_row_swap"])
def test_brute_force_catches_planted_gather_mistakes(kind, monkeypatch):
    """A mistake planted in the gather (on the CPU) must break the brute-force pin."""
    P, lens = 4, [11, 7]
    q, kc, vc, table, sl = _paged_case(21, 2, 4, 2, P, 4, lens)
    ob, _ = _brute(q, kc, vc, table, sl, P, 0.3)
    monkeypatch.setattr(oracle, "paged_gather", _mutant_gather(kind))
    o, _ = oracle.decode_paged(q, kc, vc, table, sl, page_size=P, scale=0.3)
    assert not np.allclose(o, ob, atol=1e-6)


def test_hnd_layout_is_the_same_cache_transposed():
    """The head-major page layout [pages, Hkv, page_size, D] holds the same keys: gathering
    it equals gathering its NHD transpose, and the brute force agrees."""
    P, lens = 8, [13, 30]
    q, kc, vc, table, sl = _paged_case(51, 2, 4, 2, P, 5, lens, D=16)
    kh = np.ascontiguousarray(kc.transpose(0, 2, 1, 3))
    vh = np.ascontiguousarray(vc.transpose(0, 2, 1, 3))
    np.testing.assert_array_equal(oracle.paged_gather(kh, table, sl, P, "hnd"), oracle.paged_gather(kc, table, sl, P))
    o, lse = oracle.decode_paged(q, kh, vh, table, sl, page_size=P, scale=0.3, layout="hnd")
    ob, lb = _brute(q, kc, vc, table, sl, P, 0.3)
    np.testing.assert_allclose(o, ob, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lb, rtol=0, atol=1e-12)
    with pytest.raises(ValueError):
        oracle.paged_gather(kc, table, sl, P, "nhwd")
