"""Host-side checks of the C ABI that need no GPU: the library builds for sm_103a,
loads, exports every function include/loom_attn.h declares, and rejects bad
arguments before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "loom_attn.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_29219_gb300 import build
    build.build()
    import paper_2609_29219_gb300 as loom
    return loom.capi()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(loom_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("loom_attn_fwd", "loom_attn_decode", "loom_attn_decode_workspace_bytes",
                     "loom_attn_check_error", "loom_status_string"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, f"not exported: {missing}"


def test_status_strings(lib):
    import paper_2609_29219_gb300 as loom
    for code, name in loom.STATUS.items():
        assert loom.loom_status_string(code) == name


FAKE = 0x10000  # aligned, never dereferenced: every call below is rejected during validation


@pytest.mark.parametrize("args,expect", [
    ((0, FAKE, FAKE, FAKE, None, 1, 2, 2, 128, 128, 64, 0, 0.125), 1),     # null q
    ((FAKE, FAKE, FAKE, FAKE, None, 0, 2, 2, 128, 128, 64, 0, 0.125), 1),  # B = 0
    ((FAKE, FAKE, FAKE, FAKE, None, 1, 3, 2, 128, 128, 64, 0, 0.125), 1),  # Hq % Hkv
    ((FAKE, FAKE, FAKE, FAKE, None, 1, 2, 2, 256, 128, 64, 1, 0.125), 1),  # causal Sq > Skv
    ((FAKE, FAKE, FAKE, FAKE, None, 1, 2, 2, 128, 128, 64, 0, float("nan")), 1),
    ((FAKE, FAKE, FAKE, FAKE, None, 1, 2, 2, 128, 128, 64, 0, 0.0), 1),
    ((FAKE, FAKE, FAKE, FAKE, None, 1, 2, 2, 128, 128, 64, 2, 0.125), 1),  # causal not 0/1
    ((FAKE, FAKE, FAKE, FAKE, None, 1, 2, 2, 128, 128, 96, 0, 0.125), 2),  # D unsupported
    ((FAKE + 8, FAKE, FAKE, FAKE, None, 1, 2, 2, 128, 128, 64, 0, 0.125), 3),  # misaligned
    ((FAKE, FAKE, FAKE, FAKE, FAKE + 2, 1, 2, 2, 128, 128, 64, 0, 0.125), 3),  # misaligned lse
])
def test_fwd_rejects_bad_arguments(lib, args, expect):
    assert lib.loom_attn_fwd(*args, None) == expect


def test_decode_rejects_bad_arguments(lib):
    ok = (FAKE, FAKE, FAKE, None, FAKE, None, FAKE, 1 << 20, 2, 8, 2, 1024, 128, 0.08, 4, None)

    def call(**kw):
        names = ["q", "k", "v", "sl", "o", "lse", "ws", "wsb", "B", "Hq", "Hkv", "Skv", "D", "scale",
                 "splits", "stream"]
        a = dict(zip(names, ok))
        a.update(kw)
        return lib.loom_attn_decode(*[a[n] for n in names])

    assert call(q=0) == 1
    assert call(Hq=7) == 1
    assert call(scale=-1.0) == 1
    assert call(splits=-1) == 1
    assert call(D=80) == 2
    assert call(splits=5000) == 2
    assert call(v=FAKE + 4) == 3
    assert call(sl=FAKE + 2) == 3
    assert call(ws=0) == 4
    assert call(wsb=100) == 4


def test_workspace_size_formula(lib):
    # O_i [B,Hq,S,D] fp32 + lse_i [B,Hq,S] fp32, each padded to 256 bytes, + 256 bytes
    # for the persistent split kernel's item counter
    B, Hq, D, S = 3, 8, 128, 7
    rows = B * Hq * S
    expect = (rows * D * 4 + 255) // 256 * 256 + (rows * 4 + 255) // 256 * 256 + 256
    assert lib.loom_attn_decode_workspace_bytes(B, Hq, 2, 4096, D, S) == expect
    assert lib.loom_attn_decode_workspace_bytes(B, Hq, 2, 4096, 96, S) == 0
    assert lib.loom_attn_decode_workspace_bytes(B, Hq, 2, 4096, D, 2000) == 0


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    import paper_2609_29219_gb300 as loom
    monkeypatch.setattr(loom, "_lib", None)
    monkeypatch.setattr(loom, "_LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="no fallback"):
        loom.capi()


def test_gemm_rejects_bad_arguments(lib):
    # every call is rejected during validation, before any device work
    odd = FAKE + 8
    assert lib.loom_gemm_bf16(None, FAKE, FAKE, 8, 8, 8, None) == 1   # INVALID_ARG: null
    assert lib.loom_gemm_bf16(FAKE, FAKE, FAKE, 0, 8, 8, None) == 1   # INVALID_ARG: M = 0
    assert lib.loom_gemm_bf16(FAKE, odd, FAKE, 8, 8, 8, None) == 3    # MISALIGNED
    assert lib.loom_gemm_bf16(FAKE, FAKE, FAKE, 8, 8, 12, None) == 2  # UNSUPPORTED: K % 8
    assert lib.loom_gemm_bf16(FAKE, FAKE, FAKE, 8, 20, 8, None) == 2  # UNSUPPORTED: N % 8


def test_gemm_choice_is_supported(lib):
    for M, N, K in [(1, 8, 8), (128, 256, 64), (4096, 4096, 4096), (8192, 1024, 8192), (256, 256, 16384)]:
        assert lib.loom_gemm_tile_n(M, N, K) in (64, 128, 192, 256)
        assert lib.loom_gemm_splits(M, N, K) in (1, 2, 4, 8, 16)
    assert lib.loom_gemm_tile_n(0, 8, 8) == 0
    assert lib.loom_gemm_splits(8, 0, 8) == 0


def test_gemm_splits_only_when_tiles_are_few(lib):
    # few C tiles and a long K: the model splits K over clusters
    assert lib.loom_gemm_splits(256, 256, 16384) > 1
    assert lib.loom_gemm_splits(256, 2048, 16384) > 1
    # enough tiles for every SM, or a single K stage: no split
    assert lib.loom_gemm_splits(16384, 16384, 16384) == 1
    assert lib.loom_gemm_splits(256, 256, 64) == 1
    t1 = lib.loom_model_gemm_time_us(256, 256, 16384, 64, 1, 152)
    t8 = lib.loom_model_gemm_time_us(256, 256, 16384, 64, 8, 152)
    assert 0 < t8 < t1
    assert lib.loom_model_gemm_time_us(256, 256, 16384, 64, 3, 152) < 0  # unsupported split
    assert lib.loom_model_gemm_time_us(256, 256, 16384, 96, 1, 152) < 0  # unsupported width


def test_gemm_pair_tiles_for_large_shapes(lib):
    # operand traffic per SM decides: CTA pairs for large C, never for a single K stage tile
    assert lib.loom_gemm_cta_pair(16384, 16384, 16384) == 1
    assert lib.loom_gemm_tile_n(16384, 16384, 16384) == 256
    assert lib.loom_gemm_cta_pair(256, 256, 16384) == 0
    tp = lib.loom_model_gemm_time_us(16384, 16384, 16384, 512, 1, 152)
    t1 = lib.loom_model_gemm_time_us(16384, 16384, 16384, 256, 1, 152)
    assert 0 < tp < t1


def test_paged_decode_rejects_bad_arguments(lib):
    ok = dict(q=FAKE, k=FAKE, v=FAKE, tbl=FAKE, sl=FAKE, o=FAKE, lse=None, ws=FAKE, wsb=1 << 24, B=2, Hq=8,
              Hkv=2, npages=64, P=16, maxp=8, layout=0, D=128, scale=0.08, splits=4, stream=None)
    names = list(ok)

    def call(**kw):
        a = dict(ok)
        a.update(kw)
        return lib.loom_attn_decode_paged(*[a[n] for n in names])

    assert call(tbl=None) == 1
    assert call(sl=None) == 1
    assert call(P=0) == 1
    assert call(Hq=7) == 1
    assert call(layout=2) == 1      # INVALID_ARG layout
    assert call(P=24) == 2          # UNSUPPORTED page size
    assert call(P=96) == 2
    assert call(D=80) == 2
    assert call(npages=1 << 30, P=64) == 2
    assert call(tbl=FAKE + 2) == 3  # MISALIGNED
    assert call(q=FAKE + 8) == 3
    assert call(wsb=16) == 4        # WORKSPACE


def test_varlen_prefill_rejects_bad_arguments(lib):
    ok = dict(q=FAKE, k=FAKE, v=FAKE, o=FAKE, lse=None, cq=FAKE, ck=FAKE, B=2, Hq=8, Hkv=2, tq=100, tk=100,
              maxq=60, D=128, causal=1, scale=0.08, stream=None)
    names = list(ok)

    def call(**kw):
        a = dict(ok)
        a.update(kw)
        return lib.loom_attn_fwd_varlen(*[a[n] for n in names])

    assert call(cq=None) == 1
    assert call(B=0) == 1
    assert call(tq=-1) == 1
    assert call(Hq=7) == 1
    assert call(scale=0.0) == 1
    assert call(D=96) == 2
    assert call(tk=0) == 2          # queries but no keys at all
    assert call(q=FAKE + 8) == 3
    assert call(ck=FAKE + 2) == 3
    assert call(tq=0) == 0          # nothing to do


def test_noalloc_decode_checks_arguments_before_its_scratch_size(lib):
    # a problem far beyond the built-in scratch array: argument errors are still reported
    # first, in loom_attn_decode's order; only valid arguments get LOOM_ERR_WORKSPACE
    ok = dict(q=FAKE, k=FAKE, v=FAKE, sl=None, o=FAKE, lse=None, B=64, Hq=64, Hkv=8, Skv=65536, D=128,
              scale=0.08, splits=1024, stream=None)
    names = list(ok)

    def call(**kw):
        a = dict(ok)
        a.update(kw)
        return lib.loom_attn_decode_noalloc(*[a[n] for n in names])

    assert call(q=None) == 1
    assert call(Hq=7) == 1
    assert call(D=80) == 2
    assert call(o=FAKE + 8) == 3
    assert call(sl=FAKE + 2) == 3
    assert call() == 4
