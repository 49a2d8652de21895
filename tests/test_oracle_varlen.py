"""Pins of the ragged-batch (varlen) attention oracle against what does not depend on
it: a pure-Python brute force over the packed tokens, the dense oracle when all sequences
have one length, a permutation of the sequences, causal rows with no visible key, empty
sequences, and the independence of a sequence from its neighbours' tokens."""
import math

import numpy as np
import pytest

import oracle
import synth


def _case(seed, lq, lk, Hq, Hkv, D):
    cq = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    ck = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    q = synth.bf16_normal(seed, synth.STREAM_Q, (int(cq[-1]), Hq, D))
    k = synth.bf16_normal(seed, synth.STREAM_K, (int(ck[-1]), Hkv, D))
    v = synth.bf16_normal(seed, synth.STREAM_V, (int(ck[-1]), Hkv, D))
    return q, k, v, cq, ck


def _brute(q, k, v, cq, ck, causal, scale):
    f = oracle.bf16_to_f64
    total_q, Hq, D = q.shape
    Hkv = k.shape[1]
    o = np.zeros((total_q, Hq, D))
    lse = np.full((Hq, total_q), -np.inf)
    for b in range(len(cq) - 1):
        sq, sk = int(cq[b + 1] - cq[b]), int(ck[b + 1] - ck[b])
        for h in range(Hq):
            hk = h // (Hq // Hkv)
            for i in range(sq):
                qi = [float(x) for x in f(q[cq[b] + i, h])]
                sc, vs = [], []
                for j in range(sk):
                    if causal and j > i + (sk - sq):
                        continue
                    kj = [float(x) for x in f(k[ck[b] + j, hk])]
                    sc.append(scale * sum(a * c for a, c in zip(qi, kj)))
                    vs.append([float(x) for x in f(v[ck[b] + j, hk])])
                if not sc:
                    continue
                m = max(sc)
                w = [math.exp(s - m) for s in sc]
                z = sum(w)
                lse[h, cq[b] + i] = m + math.log(z)
                for d in range(D):
                    o[cq[b] + i, h, d] = sum(wi * vv[d] for wi, vv in zip(w, vs)) / z
    return o, lse


@pytest.mark.parametrize("causal", [False, True])
def test_matches_brute_force(causal):
    lq, lk = [3, 0, 7, 5, 2], [3, 4, 9, 2, 0]  # includes Sq > Skv (causal: rows with no key) and empty sequences
    q, k, v, cq, ck = _case(1, lq, lk, 4, 2, 8)
    o, lse = oracle.attention_varlen(q, k, v, cq, ck, causal=causal, scale=0.4)
    ob, lb = _brute(q, k, v, cq, ck, causal, 0.4)
    np.testing.assert_allclose(o, ob, rtol=0, atol=1e-12)
    np.testing.assert_array_equal(np.isneginf(lse), np.isneginf(lb))
    fin = np.isfinite(lb)
    np.testing.assert_allclose(lse[fin], lb[fin], rtol=0, atol=1e-12)


@pytest.mark.parametrize("causal", [False, True])
def test_equal_lengths_equal_dense(causal):
    B, S, Hq, Hkv, D = 3, 40, 4, 2, 16
    q, k, v, cq, ck = _case(2, [S] * B, [S] * B, Hq, Hkv, D)
    o, lse = oracle.attention_varlen(q, k, v, cq, ck, causal=causal)
    qd = np.ascontiguousarray(q.reshape(B, S, Hq, D).transpose(0, 2, 1, 3))
    kd = np.ascontiguousarray(k.reshape(B, S, Hkv, D).transpose(0, 2, 1, 3))
    vd = np.ascontiguousarray(v.reshape(B, S, Hkv, D).transpose(0, 2, 1, 3))
    od, ld = oracle.attention(qd, kd, vd, causal=causal)
    np.testing.assert_array_equal(o, od.transpose(0, 2, 1, 3).reshape(B * S, Hq, D))
    np.testing.assert_array_equal(lse, ld.transpose(1, 0, 2).reshape(Hq, B * S))


def test_sequence_permutation():
    lq, lk = [5, 9, 2], [6, 9, 4]
    q, k, v, cq, ck = _case(3, lq, lk, 2, 1, 16)
    o, lse = oracle.attention_varlen(q, k, v, cq, ck, causal=True)
    perm = [2, 0, 1]
    qp = np.concatenate([q[cq[b]:cq[b + 1]] for b in perm])
    kp = np.concatenate([k[ck[b]:ck[b + 1]] for b in perm])
    vp = np.concatenate([v[ck[b]:ck[b + 1]] for b in perm])
    cq2 = np.concatenate([[0], np.cumsum([lq[b] for b in perm])])
    ck2 = np.concatenate([[0], np.cumsum([lk[b] for b in perm])])
    o2, lse2 = oracle.attention_varlen(qp, kp, vp, cq2, ck2, causal=True)
    for i, b in enumerate(perm):
        np.testing.assert_array_equal(o2[cq2[i]:cq2[i + 1]], o[cq[b]:cq[b + 1]])
        np.testing.assert_array_equal(lse2[:, cq2[i]:cq2[i + 1]], lse[:, cq[b]:cq[b + 1]])


def test_neighbours_do_not_leak():
    lq, lk = [4, 6, 3], [5, 6, 7]
    q, k, v, cq, ck = _case(4, lq, lk, 2, 2, 16)
    o, lse = oracle.attention_varlen(q, k, v, cq, ck)
    q2, k2, v2 = q.copy(), k.copy(), v.copy()
    q2[cq[0]:cq[1]] = 0x3F80
    k2[ck[2]:ck[3]] = 0xBF80
    v2[ck[0]:ck[1]] = 0x4000
    o2, lse2 = oracle.attention_varlen(q2, k2, v2, cq, ck)
    np.testing.assert_array_equal(o2[cq[1]:cq[2]], o[cq[1]:cq[2]])
    np.testing.assert_array_equal(lse2[:, cq[1]:cq[2]], lse[:, cq[1]:cq[2]])


def test_rejects_bad_offsets():
    q, k, v, cq, ck = _case(5, [2, 3], [2, 3], 1, 1, 8)
    with pytest.raises(ValueError):
        oracle.attention_varlen(q, k, v, cq[::-1].copy(), ck)
    with pytest.raises(ValueError):
        oracle.attention_varlen(q, k, v, cq + 1, ck)
