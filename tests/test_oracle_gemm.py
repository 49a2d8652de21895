"""Pins of the GEMM oracle (C = A B in fp64 from bf16 inputs) against what does not
depend on it: a pure-Python triple loop, and closed forms (identity, all-ones,
transposition, rank one, row selection)."""
import numpy as np
import pytest

import oracle
import synth

ONE = np.uint16(0x3F80)  # bf16 1.0


def _bits(seed, stream, shape):
    return synth.bf16_normal(seed, stream, shape)


def test_matches_triple_loop():
    M, K, N = 5, 7, 3
    a, b = _bits(1, 0, (M, K)), _bits(1, 1, (K, N))
    A, B = oracle.bf16_to_f64(a), oracle.bf16_to_f64(b)
    ref = [[sum(A[i][k] * B[k][j] for k in range(K)) for j in range(N)] for i in range(M)]
    np.testing.assert_allclose(oracle.gemm(a, b), np.array(ref), rtol=1e-13, atol=1e-13)


def test_bf16_widening_is_exact():
    # 1.0, -2.0, the smallest normal and the largest finite bfloat16
    bits = np.array([0x3F80, 0xC000, 0x0080, 0x7F7F], np.uint16)
    np.testing.assert_array_equal(oracle.bf16_to_f64(bits), [1.0, -2.0, 2.0 ** -126, (2 - 2 ** -7) * 2.0 ** 127])


def test_identity_returns_b():
    K, N = 16, 9
    eye = np.zeros((K, K), np.uint16)
    eye[np.arange(K), np.arange(K)] = ONE
    b = _bits(2, 1, (K, N))
    np.testing.assert_array_equal(oracle.gemm(eye, b), oracle.bf16_to_f64(b))


def test_ones_give_row_sums():
    M, K, N = 6, 33, 4
    a = _bits(3, 0, (M, K))
    ones = np.full((K, N), ONE, np.uint16)
    c = oracle.gemm(a, ones)
    sums = oracle.bf16_to_f64(a).sum(axis=1)
    for j in range(N):
        np.testing.assert_allclose(c[:, j], sums, rtol=1e-13, atol=1e-13)


def test_transpose_identity():
    M, K, N = 8, 12, 5
    a, b = _bits(4, 0, (M, K)), _bits(4, 1, (K, N))
    np.testing.assert_allclose(oracle.gemm(a, b).T, oracle.gemm(b.T.copy(), a.T.copy()), rtol=1e-13, atol=1e-13)


def test_rank_one():
    u, v = _bits(5, 0, (7, 1)), _bits(5, 1, (1, 6))
    c = oracle.gemm(u, v)
    np.testing.assert_array_equal(c, np.outer(oracle.bf16_to_f64(u)[:, 0], oracle.bf16_to_f64(v)[0]))


def test_row_selection():
    a, b = _bits(6, 0, (20, 16)), _bits(6, 1, (16, 8))
    rows = [0, 3, 19, 7]
    np.testing.assert_array_equal(oracle.gemm(a, b, rows=rows), oracle.gemm(a, b)[rows])


def test_shape_mismatch_rejected():
    with pytest.raises(ValueError):
        oracle.gemm(_bits(7, 0, (4, 5)), _bits(7, 1, (6, 3)))


def test_transposed_b_matches_triple_loop():
    """b given [N, K]: c_ij = sum_k a_ik b_jk, checked element by element in plain Python."""
    rng = np.random.default_rng(7)
    M, K, N = 5, 7, 3
    a = synth.f32_to_bf16(rng.standard_normal((M, K)).astype(np.float32))
    bt = synth.f32_to_bf16(rng.standard_normal((N, K)).astype(np.float32))
    c = oracle.gemm(a, bt, b_transposed=True)
    A, Bt = oracle.bf16_to_f64(a), oracle.bf16_to_f64(bt)
    for i in range(M):
        for j in range(N):
            ref = sum(float(A[i, k]) * float(Bt[j, k]) for k in range(K))
            assert abs(c[i, j] - ref) <= 1e-12 * max(1.0, abs(ref))
    with pytest.raises(ValueError):
        oracle.gemm(a, bt)  # [N, K] taken as [K, N]: the inner sizes disagree
