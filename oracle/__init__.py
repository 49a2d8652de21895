"""ctypes front end of the fp64 CPU oracle (``oracle.cpp``).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py``, never by the product package.  It shares no code
with the CUDA library; the only common dependency is the seeded input generator
(``synth``), which holds no attention arithmetic.

Arrays are numpy: Q [B, Hq, Sq, D], K/V [B, Hkv, Skv, D] (and the GEMM operands A [M, K],
B [K, N]; a paged KV cache [num_pages, page_size, Hkv, D]; packed ragged batches
[total_tokens, H, D]) as uint16 bfloat16 bit patterns, results in float64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.cpp")
_LIB_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_LIB_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

_u16p = np.ctypeslib.ndpointer(dtype=np.uint16, flags="C_CONTIGUOUS")
_f64p = np.ctypeslib.ndpointer(dtype=np.float64, flags="C_CONTIGUOUS")


def build(force: bool = False) -> str:
    """Compile ``oracle.cpp`` into ``_build/liboracle.so`` (plain g++, no fast-math)."""
    os.makedirs(_LIB_DIR, exist_ok=True)
    stale = (not os.path.exists(_LIB)) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-pthread", "-o", tmp, _SRC]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _bind(path: str):
    """Open a compiled oracle library and declare its C signatures."""
    lib = ctypes.CDLL(path)
    i32, i64, dbl = ctypes.c_int, ctypes.c_int64, ctypes.c_double
    vp = ctypes.c_void_p
    lib.oracle_attention.argtypes = [_u16p, _u16p, _u16p, i32, i32, i32, i32, i32, i32,
                                     i32, dbl, vp, vp, i64, _f64p, _f64p, i32]
    lib.oracle_attention.restype = i32
    lib.oracle_decode_split_merge.argtypes = [_u16p, _u16p, _u16p, i32, i32, i32, i32, i32,
                                              dbl, vp, i32, i32, vp, vp, _f64p, _f64p, i32]
    lib.oracle_decode_split_merge.restype = i32
    lib.oracle_attention_naive.argtypes = [_u16p, _u16p, _u16p, i32, i32, i32, i32, i32,
                                           i32, i32, dbl, _f64p, _f64p]
    lib.oracle_attention_naive.restype = i32
    lib.oracle_decode_chunk.argtypes = [i64, i32, i32]
    lib.oracle_decode_chunk.restype = i64
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(build())
    return _lib


def _shapes(q, k, v):
    if q.ndim != 4 or k.ndim != 4 or v.shape != k.shape:
        raise ValueError("expected Q [B,Hq,Sq,D] and K/V [B,Hkv,Skv,D]")
    B, Hq, Sq, D = q.shape
    Bk, Hkv, Skv, Dk = k.shape
    if Bk != B or Dk != D:
        raise ValueError("batch or head-dim mismatch between Q and K/V")
    return B, Hq, Hkv, Sq, Skv, D


def _u16(a):
    return np.ascontiguousarray(a, dtype=np.uint16)


def attention(q, k, v, *, causal=False, scale=None, seqlens_k=None, rows=None, nthreads=0):
    """Attention by definition in fp64.

    ``rows`` optionally lists flat row indices ``(b*Hq + h)*Sq + i``; the result then
    holds only those rows.  Returns ``(o, lse)``: o [B,Hq,Sq,D] (or [nrows, D]) and
    lse [B,Hq,Sq] (or [nrows]).
    """
    q, k, v = _u16(q), _u16(k), _u16(v)
    B, Hq, Hkv, Sq, Skv, D = _shapes(q, k, v)
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    sl = None if seqlens_k is None else np.ascontiguousarray(seqlens_k, dtype=np.int32)
    if rows is None:
        nrows = B * Hq * Sq
        rp = None
    else:
        rows = np.ascontiguousarray(rows, dtype=np.int64)
        nrows = rows.size
        rp = rows.ctypes.data
    o = np.zeros((max(nrows, 1), D), dtype=np.float64)
    lse = np.zeros(max(nrows, 1), dtype=np.float64)
    rc = _load().oracle_attention(q, k, v, B, Hq, Hkv, Sq, Skv, D, int(bool(causal)), float(scale),
                                  None if sl is None else sl.ctypes.data, rp, nrows, o, lse,
                                  int(nthreads))
    if rc != 0:
        raise ValueError("oracle_attention rejected its arguments")
    o, lse = o[:nrows], lse[:nrows]
    if rows is None:
        return o.reshape(B, Hq, Sq, D), lse.reshape(B, Hq, Sq)
    return o, lse


def decode_chunk(length: int, num_splits: int, chunk_align: int = 64) -> int:
    """Chunk length of the Flash Decode split rule (see ``oracle.cpp``)."""
    return int(_load().oracle_decode_chunk(int(length), int(num_splits), int(chunk_align)))


def decode_split_merge(q, k, v, *, num_splits, scale=None, seqlens_k=None, chunk_align=64,
                       nthreads=0):
    """Flash Decode in fp64: per-split partials then the log-sum-exp merge.

    q [B,Hq,1,D].  Returns ``(o [B,Hq,D], lse [B,Hq], o_part [B,Hq,S,D], lse_part [B,Hq,S])``.
    """
    q, k, v = _u16(q), _u16(k), _u16(v)
    B, Hq, Hkv, Sq, Skv, D = _shapes(q, k, v)
    if Sq != 1:
        raise ValueError("decode takes Sq == 1")
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    sl = None if seqlens_k is None else np.ascontiguousarray(seqlens_k, dtype=np.int32)
    o = np.zeros((B * Hq, D), dtype=np.float64)
    lse = np.zeros(max(B * Hq, 1), dtype=np.float64)
    o_part = np.zeros((B * Hq * num_splits, D), dtype=np.float64)
    lse_part = np.zeros(max(B * Hq * num_splits, 1), dtype=np.float64)
    rc = _load().oracle_decode_split_merge(q, k, v, B, Hq, Hkv, Skv, D, float(scale),
                                           None if sl is None else sl.ctypes.data,
                                           int(num_splits), int(chunk_align),
                                           o_part.ctypes.data, lse_part.ctypes.data, o, lse,
                                           int(nthreads))
    if rc != 0:
        raise ValueError("oracle_decode_split_merge rejected its arguments")
    return (o.reshape(B, Hq, D), lse[:B * Hq].reshape(B, Hq),
            o_part.reshape(B, Hq, num_splits, D), lse_part[:B * Hq * num_splits].reshape(B, Hq, num_splits))


def attention_naive(q, k, v, *, causal=False, scale=None):
    """Long-double naive attention (no max subtraction); tiny inputs only."""
    q, k, v = _u16(q), _u16(k), _u16(v)
    B, Hq, Hkv, Sq, Skv, D = _shapes(q, k, v)
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    o = np.zeros((max(B * Hq * Sq, 1), D), dtype=np.float64)
    lse = np.zeros(max(B * Hq * Sq, 1), dtype=np.float64)
    rc = _load().oracle_attention_naive(q, k, v, B, Hq, Hkv, Sq, Skv, D, int(bool(causal)),
                                        float(scale), o, lse)
    if rc != 0:
        raise ValueError("oracle_attention_naive rejected its arguments")
    n = B * Hq * Sq
    return o[:n].reshape(B, Hq, Sq, D), lse[:n].reshape(B, Hq, Sq)


def bf16_to_f64(bits):
    """Exact widening of bfloat16 bit patterns (uint16) to float64."""
    bits = np.asarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def gemm(a, b, *, rows=None, b_transposed=False):
    """C = A B in fp64 from bf16 A [M, K] and B [K, N] (the paper's third kernel, evaluated
    on GEMM shapes): the definition, c_ij = sum_k a_ik b_kj, with the exactly widened
    inputs and a library matmul as its one step.  ``b_transposed``: b is given [N, K] and
    C = A b^T (c_ij = sum_k a_ik b_jk).  ``rows`` optionally selects rows of C."""
    A = bf16_to_f64(a)
    Bm = bf16_to_f64(b)
    if b_transposed:
        Bm = Bm.T
    if A.ndim != 2 or Bm.ndim != 2 or A.shape[1] != Bm.shape[0]:
        raise ValueError("expected A [M, K] and B [K, N] ([N, K] when transposed)")
    if rows is not None:
        A = A[np.asarray(rows, dtype=np.int64)]
    return A @ Bm


def paged_gather(cache, block_table, seqlens, page_size, layout="nhd"):
    """The logical K (or V) [B, Hkv, Skv_max, D] of a paged cache: key t of sequence b is
    row t mod page_size of physical page block_table[b, t div page_size] (the usual
    paged-KV convention; the paper has none).  layout "nhd": cache [num_pages, page_size,
    Hkv, D]; "hnd": cache [num_pages, Hkv, page_size, D].  Skv_max = block_table.shape[1] *
    page_size; positions at or past seqlens[b] are left zero, and their table entries are
    not read (they may be anything)."""
    cache = _u16(cache)
    if layout == "hnd":
        cache = cache.transpose(0, 2, 1, 3)
    elif layout != "nhd":
        raise ValueError("layout is 'nhd' or 'hnd'")
    table = np.asarray(block_table, dtype=np.int64)
    lens = np.asarray(seqlens, dtype=np.int64)
    npages, P, Hkv, D = cache.shape
    if P != page_size:
        raise ValueError("cache rows per page != page_size")
    B, max_pages = table.shape
    out = np.zeros((B, Hkv, max_pages * P, D), dtype=np.uint16)
    for b in range(B):
        n = int(min(max(lens[b], 0), max_pages * P))
        for j in range((n + P - 1) // P):
            page = int(table[b, j])
            if not 0 <= page < npages:
                raise ValueError(f"block_table[{b}, {j}] = {page} is not a page of the cache")
            r = min(P, n - j * P)
            out[b, :, j * P:j * P + r, :] = cache[page, :r].transpose(1, 0, 2)
    return out


def decode_paged(q, k_cache, v_cache, block_table, seqlens, *, page_size, scale=None, nthreads=0, layout="nhd"):
    """Decode (one query row per head) over a paged KV cache: the attention definition on
    the logical K/V that ``paged_gather`` assembles.  q [B, Hq, 1, D].  Returns
    ``(o [B, Hq, D], lse [B, Hq])``."""
    k = paged_gather(k_cache, block_table, seqlens, page_size, layout)
    v = paged_gather(v_cache, block_table, seqlens, page_size, layout)
    o, lse = attention(q, k, v, scale=scale, seqlens_k=np.asarray(seqlens, dtype=np.int32), nthreads=nthreads)
    return o[:, :, 0, :], lse[:, :, 0]


def attention_varlen(q, k, v, cu_seqlens_q, cu_seqlens_k, *, causal=False, scale=None, nthreads=0):
    """Attention over a ragged batch packed token-major: q [total_q, Hq, D], k/v
    [total_k, Hkv, D]; sequence b owns query tokens cu_seqlens_q[b] .. cu_seqlens_q[b+1]
    and key tokens cu_seqlens_k[b] .. cu_seqlens_k[b+1] (the packed-varlen convention; the
    paper has none).  Each sequence is the attention definition on its own tokens, causal
    masking bottom-right aligned per sequence.  Returns ``(o [total_q, Hq, D],
    lse [Hq, total_q])``; a query with no visible key has O = 0 and LSE = -inf."""
    q, k, v = _u16(q), _u16(k), _u16(v)
    cq = np.asarray(cu_seqlens_q, dtype=np.int64)
    ck = np.asarray(cu_seqlens_k, dtype=np.int64)
    total_q, Hq, D = q.shape
    total_k, Hkv, Dk = k.shape
    if v.shape != k.shape or Dk != D or cq.shape != ck.shape or cq.ndim != 1 or cq.size < 2:
        raise ValueError("expected q [total_q, Hq, D], k/v [total_k, Hkv, D], cu_seqlens [B + 1]")
    if cq[0] != 0 or ck[0] != 0 or cq[-1] != total_q or ck[-1] != total_k or np.any(np.diff(cq) < 0) \
            or np.any(np.diff(ck) < 0):
        raise ValueError("cu_seqlens must run from 0 to the token totals without decreasing")
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    o = np.zeros((total_q, Hq, D), dtype=np.float64)
    lse = np.full((Hq, total_q), -np.inf, dtype=np.float64)
    for b in range(cq.size - 1):
        q0, q1, k0, k1 = int(cq[b]), int(cq[b + 1]), int(ck[b]), int(ck[b + 1])
        if q1 == q0:
            continue
        if k1 == k0:
            continue  # no keys: O = 0, LSE = -inf
        qb = np.ascontiguousarray(q[q0:q1].transpose(1, 0, 2))[None]
        kb = np.ascontiguousarray(k[k0:k1].transpose(1, 0, 2))[None]
        vb = np.ascontiguousarray(v[k0:k1].transpose(1, 0, 2))[None]
        if causal and q1 - q0 > k1 - k0:
            # rows with no visible key (i < Sq - Skv) are left at O = 0, LSE = -inf; the
            # others see keys j <= i + (Skv - Sq) as in the definition
            skip = (q1 - q0) - (k1 - k0)
            ob, lb = attention(qb[:, :, skip:], kb, vb, causal=True, scale=scale, nthreads=nthreads)
            o[q0 + skip:q1] = ob[0].transpose(1, 0, 2)
            lse[:, q0 + skip:q1] = lb[0]
        else:
            ob, lb = attention(qb, kb, vb, causal=causal, scale=scale, nthreads=nthreads)
            o[q0:q1] = ob[0].transpose(1, 0, 2)
            lse[:, q0:q1] = lb[0]
    return o, lse
