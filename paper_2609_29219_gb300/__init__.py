"""GB300 fused attention (prefill + Flash Decode): thin Python binding of ``libloomattn.so``.

Every function here only marshals arguments (tensor data pointers, sizes, the current
CUDA stream) into the C ABI declared in ``include/loom_attn.h``; all computation runs
in the library's CUDA kernels.  There is no fallback: if the compiled library is
missing, every call raises.

Two layers:

* ``capi()`` returns the ``ctypes.CDLL`` with argument types declared -- the raw C ABI,
  taking integer device pointers.
* Functions with the C names (``loom_attn_fwd``, ``loom_attn_decode``, ...) that take
  torch tensors, check their dtype/device/layout, and raise ``LoomError`` on a non-OK
  status.
"""
from __future__ import annotations

import ctypes
import os
import threading

__all__ = [
    "LoomError", "capi", "library_path", "STATUS",
    "loom_attn_fwd", "loom_attn_decode", "loom_attn_decode_noalloc", "loom_attn_decode_workspace_bytes",
    "loom_attn_decode_num_splits", "loom_attn_check_error", "loom_status_string",
    "loom_debug_set_timeout_ns", "loom_debug_inject", "loom_model_fwd_plan",
    "loom_model_fwd_time_us", "loom_model_decode_time_us", "FwdPlan", "loom_debug_prefill_design",
    "loom_model_fwd_plan_variant", "loom_model_heg_pipe", "loom_model_fwd_time_us_design",
    "loom_attn_decode_paged", "loom_attn_fwd_varlen", "loom_gemm_bf16", "loom_gemm_bf16_bt", "loom_gemm_tile_n", "loom_gemm_splits", "loom_gemm_cta_pair", "loom_model_gemm_time_us", "loom_debug_gemm_tile_n",
    "loom_debug_gemm_splits", "loom_debug_gemm_cta_pair", "loom_model_decode_cluster_time_us",
    "loom_attn_decode_form", "loom_decode_max_clusters", "loom_decode_persistent_slots", "loom_debug_decode_form",
    "loom_model_decode_persistent_time_us", "loom_model_decode_tc_time_us", "DECODE_SPLIT_MERGE", "DECODE_PERSISTENT", "DECODE_CLUSTER",
    "loom_debug_prefill_slots", "loom_debug_decode_stage_plan", "loom_debug_gemm_stages",
    "loom_debug_gemm_order", "loom_debug_decode_tensor_cores",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libloomattn.so")
_lock = threading.Lock()
_lib = None

STATUS = {
    0: "LOOM_OK", 1: "LOOM_ERR_INVALID_ARG", 2: "LOOM_ERR_UNSUPPORTED", 3: "LOOM_ERR_MISALIGNED",
    4: "LOOM_ERR_WORKSPACE", 5: "LOOM_ERR_CUDA", 6: "LOOM_ERR_TIMEOUT",
}


class FwdPlan(ctypes.Structure):
    """Mirror of ``loom_fwd_plan`` (include/loom_attn.h)."""
    _fields_ = [(n, ctypes.c_int) for n in ("design", "bm", "bn", "q_tiles", "s_buffers", "kv_slots",
                                             "b_lm", "b_ms", "smem_bytes", "tmem_cols")] + \
               [(n, ctypes.c_double) for n in ("t_load_ns", "t_mma_ns", "t_softmax_ns", "t_iter_ns")]

    def as_dict(self):
        return {n: getattr(self, n) for n, _ in self._fields_}


class LoomError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)}")


def library_path() -> str:
    return _LIB_PATH


def capi() -> ctypes.CDLL:
    """The compiled library with its C signatures declared (raises if it is missing)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(_LIB_PATH):
                raise RuntimeError(
                    f"{_LIB_PATH} is missing: build it with paper_2609_29219_gb300.build.build() "
                    "(there is no fallback implementation)")
            lib = ctypes.CDLL(_LIB_PATH)
            vp, i32, f32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
            lib.loom_attn_fwd.argtypes = [vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i32, f32, vp]
            lib.loom_attn_fwd.restype = i32
            lib.loom_attn_decode_num_splits.argtypes = [i32, i32, i32, i32, i32]
            lib.loom_attn_decode_num_splits.restype = i32
            lib.loom_attn_decode_workspace_bytes.argtypes = [i32, i32, i32, i32, i32, i32]
            lib.loom_attn_decode_workspace_bytes.restype = sz
            lib.loom_attn_decode.argtypes = [vp, vp, vp, vp, vp, vp, vp, sz, i32, i32, i32, i32, i32,
                                             f32, i32, vp]
            lib.loom_attn_decode.restype = i32
            lib.loom_attn_decode_noalloc.argtypes = [vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, f32, i32,
                                                     vp]
            lib.loom_attn_decode_noalloc.restype = i32
            lib.loom_attn_check_error.argtypes = [vp]
            lib.loom_attn_check_error.restype = i32
            lib.loom_status_string.argtypes = [i32]
            lib.loom_status_string.restype = ctypes.c_char_p
            lib.loom_debug_set_timeout_ns.argtypes = [ctypes.c_uint64]
            lib.loom_debug_set_timeout_ns.restype = None
            lib.loom_debug_inject.argtypes = [i32]
            lib.loom_debug_inject.restype = None
            lib.loom_debug_prefill_design.argtypes = [i32]
            lib.loom_debug_prefill_design.restype = None
            lib.loom_model_fwd_plan.argtypes = [i32, ctypes.POINTER(FwdPlan)]
            lib.loom_model_fwd_plan.restype = i32
            lib.loom_model_fwd_plan_variant.argtypes = [i32, i32, ctypes.POINTER(FwdPlan)]
            lib.loom_model_fwd_plan_variant.restype = i32
            lib.loom_model_heg_pipe.argtypes = [ctypes.c_double] * 3 + [i32, i32]
            lib.loom_model_heg_pipe.restype = ctypes.c_double
            lib.loom_model_fwd_time_us.argtypes = [i32, i32, i32, i32, i32, i32]
            lib.loom_model_fwd_time_us.restype = ctypes.c_double
            lib.loom_model_fwd_time_us_design.argtypes = [i32] * 7
            lib.loom_model_fwd_time_us_design.restype = ctypes.c_double
            lib.loom_attn_decode_paged.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, sz, i32, i32, i32, i32,
                                                   i32, i32, i32, i32, f32, i32, vp]
            lib.loom_attn_decode_paged.restype = i32
            lib.loom_attn_fwd_varlen.argtypes = [vp, vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i32,
                                                 i32, f32, vp]
            lib.loom_attn_fwd_varlen.restype = i32
            lib.loom_gemm_bf16.argtypes = [vp, vp, vp, i32, i32, i32, vp]
            lib.loom_gemm_bf16.restype = i32
            lib.loom_gemm_bf16_bt.argtypes = [vp, vp, vp, i32, i32, i32, vp]
            lib.loom_gemm_bf16_bt.restype = i32
            lib.loom_gemm_tile_n.argtypes = [i32, i32, i32]
            lib.loom_gemm_tile_n.restype = i32
            lib.loom_gemm_splits.argtypes = [i32, i32, i32]
            lib.loom_gemm_splits.restype = i32
            lib.loom_gemm_cta_pair.argtypes = [i32, i32, i32]
            lib.loom_gemm_cta_pair.restype = i32
            lib.loom_model_gemm_time_us.argtypes = [i32] * 6
            lib.loom_model_gemm_time_us.restype = ctypes.c_double
            lib.loom_debug_gemm_tile_n.argtypes = [i32]
            lib.loom_debug_gemm_tile_n.restype = None
            lib.loom_debug_gemm_splits.argtypes = [i32]
            lib.loom_debug_gemm_splits.restype = None
            lib.loom_debug_gemm_cta_pair.argtypes = [i32]
            lib.loom_debug_gemm_cta_pair.restype = None
            lib.loom_model_decode_time_us.argtypes = [i32, i32, i32, i32, i32, i32, i32]
            lib.loom_model_decode_time_us.restype = ctypes.c_double
            lib.loom_model_decode_cluster_time_us.argtypes = [i32] * 8
            lib.loom_model_decode_cluster_time_us.restype = ctypes.c_double
            lib.loom_model_decode_persistent_time_us.argtypes = [i32] * 7
            lib.loom_model_decode_persistent_time_us.restype = ctypes.c_double
            lib.loom_model_decode_tc_time_us.argtypes = [i32] * 7
            lib.loom_model_decode_tc_time_us.restype = ctypes.c_double
            lib.loom_attn_decode_form.argtypes = [i32] * 7 + [ctypes.POINTER(i32)]
            lib.loom_attn_decode_form.restype = i32
            lib.loom_decode_max_clusters.argtypes = [i32, i32, i32]
            lib.loom_decode_max_clusters.restype = i32
            lib.loom_decode_persistent_slots.argtypes = [i32, i32]
            lib.loom_decode_persistent_slots.restype = i32
            lib.loom_debug_decode_form.argtypes = [i32, i32]
            lib.loom_debug_decode_form.restype = None
            lib.loom_debug_prefill_slots.argtypes = [i32, i32]
            lib.loom_debug_prefill_slots.restype = i32
            lib.loom_debug_decode_stage_plan.argtypes = [i32, i32, i32]
            lib.loom_debug_decode_stage_plan.restype = i32
            lib.loom_debug_gemm_stages.argtypes = [i32]
            lib.loom_debug_gemm_stages.restype = None
            lib.loom_debug_gemm_order.argtypes = [i32, i32]
            lib.loom_debug_gemm_order.restype = None
            lib.loom_debug_decode_tensor_cores.argtypes = [i32]
            lib.loom_debug_decode_tensor_cores.restype = None
            _lib = lib
    return _lib


# ------------------------------------------------------------------ marshalling helpers
def _torch():
    import torch
    return torch


def _dev_ptr(t, name, dtype=None, ndim=None):
    torch = _torch()
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got shape {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _stream_ptr(stream, device):
    torch = _torch()
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _check(status: int, where: str):
    if status != 0:
        raise LoomError(status, where)


# ------------------------------------------------------------------ C-ABI functions
def loom_attn_fwd(q, k, v, o=None, lse=None, *, causal=False, scale=None, stream=None,
                  return_lse=False):
    """Prefill attention.  q [B,Hq,Sq,D], k/v [B,Hkv,Skv,D] bf16 CUDA tensors.

    Writes ``o`` ([B,Hq,Sq,D] bf16, allocated if None) and, if given (or
    ``return_lse``), ``lse`` ([B,Hq,Sq] fp32).  Returns ``o`` or ``(o, lse)``.
    """
    torch = _torch()
    bf16 = torch.bfloat16
    qp = _dev_ptr(q, "q", bf16, 4)
    kp = _dev_ptr(k, "k", bf16, 4)
    vp_ = _dev_ptr(v, "v", bf16, 4)
    B, Hq, Sq, D = q.shape
    Bk, Hkv, Skv, Dk = k.shape
    if tuple(v.shape) != tuple(k.shape) or Bk != B or Dk != D:
        raise ValueError("q/k/v shapes disagree")
    if o is None:
        o = torch.empty_like(q)
    if tuple(o.shape) != tuple(q.shape):
        raise ValueError("o must have q's shape")
    op = _dev_ptr(o, "o", bf16, 4)
    if lse is None and return_lse:
        lse = torch.empty((B, Hq, Sq), dtype=torch.float32, device=q.device)
    lp = None
    if lse is not None:
        if tuple(lse.shape) != (B, Hq, Sq):
            raise ValueError("lse must be [B, Hq, Sq]")
        lp = _dev_ptr(lse, "lse", torch.float32)
    if scale is None:
        scale = D ** -0.5
    st = capi().loom_attn_fwd(qp, kp, vp_, op, lp, B, Hq, Hkv, Sq, Skv, D, int(bool(causal)),
                              float(scale), _stream_ptr(stream, q.device))
    _check(st, "loom_attn_fwd")
    return (o, lse) if (return_lse or lse is not None) else o


def loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D) -> int:
    return int(capi().loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D))


def loom_attn_decode_workspace_bytes(B, Hq, Hkv, Skv, D, num_splits=0) -> int:
    return int(capi().loom_attn_decode_workspace_bytes(B, Hq, Hkv, Skv, D, num_splits))


def _decode_operands(q, k_cache, v_cache, seqlens_k, o, lse, return_lse):
    """Pointers and sizes of the contiguous decode entry points' tensor arguments."""
    torch = _torch()
    bf16 = torch.bfloat16
    qp = _dev_ptr(q, "q", bf16, 4)
    kp = _dev_ptr(k_cache, "k_cache", bf16, 4)
    vp_ = _dev_ptr(v_cache, "v_cache", bf16, 4)
    B, Hq, Sq, D = q.shape
    Bk, Hkv, Skv, Dk = k_cache.shape
    if Sq != 1 or tuple(v_cache.shape) != tuple(k_cache.shape) or Bk != B or Dk != D:
        raise ValueError("decode takes q [B,Hq,1,D] and k/v caches [B,Hkv,Skv,D]")
    sp = None
    if seqlens_k is not None:
        if tuple(seqlens_k.shape) != (B,):
            raise ValueError("seqlens_k must be [B]")
        sp = _dev_ptr(seqlens_k, "seqlens_k", torch.int32)
    if o is None:
        o = torch.empty_like(q)
    op = _dev_ptr(o, "o", bf16, 4)
    if lse is None and return_lse:
        lse = torch.empty((B, Hq), dtype=torch.float32, device=q.device)
    lp = None
    if lse is not None:
        if lse.numel() != B * Hq:
            raise ValueError("lse must hold B*Hq values")
        lp = _dev_ptr(lse, "lse", torch.float32)
    return (qp, kp, vp_, sp, op, lp), (B, Hq, Hkv, Skv, D), o, lse


def loom_attn_decode(q, k_cache, v_cache, seqlens_k=None, o=None, lse=None, workspace=None, *,
                     scale=None, num_splits=0, stream=None, return_lse=False):
    """Flash Decode.  q [B,Hq,1,D], k_cache/v_cache [B,Hkv,Skv,D] bf16, seqlens_k [B] int32.

    ``workspace`` is a CUDA uint8 tensor of at least ``loom_attn_decode_workspace_bytes``
    bytes (allocated here if None).  Returns ``o`` or ``(o, lse)``.
    """
    torch = _torch()
    (qp, kp, vp_, sp, op, lp), (B, Hq, Hkv, Skv, D), o, lse = _decode_operands(
        q, k_cache, v_cache, seqlens_k, o, lse, return_lse)
    if workspace is None:
        need = loom_attn_decode_workspace_bytes(B, Hq, Hkv, Skv, D, num_splits)
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=q.device)
    wp = _dev_ptr(workspace, "workspace")
    if scale is None:
        scale = D ** -0.5
    st = capi().loom_attn_decode(qp, kp, vp_, sp, op, lp, wp, workspace.numel() * workspace.element_size(),
                                 B, Hq, Hkv, Skv, D, float(scale), int(num_splits),
                                 _stream_ptr(stream, q.device))
    _check(st, "loom_attn_decode")
    return (o, lse) if (return_lse or lse is not None) else o


def loom_attn_decode_noalloc(q, k_cache, v_cache, seqlens_k=None, o=None, lse=None, *, scale=None,
                             num_splits=0, stream=None, return_lse=False):
    """Flash Decode with the partials in the library's built-in scratch array (no
    workspace argument, no device allocation by the library).  Arguments and results as
    ``loom_attn_decode``; problems whose partials exceed the array raise LOOM_ERR_WORKSPACE."""
    (qp, kp, vp_, sp, op, lp), (B, Hq, Hkv, Skv, D), o, lse = _decode_operands(
        q, k_cache, v_cache, seqlens_k, o, lse, return_lse)
    if scale is None:
        scale = D ** -0.5
    st = capi().loom_attn_decode_noalloc(qp, kp, vp_, sp, op, lp, B, Hq, Hkv, Skv, D, float(scale),
                                         int(num_splits), _stream_ptr(stream, q.device))
    _check(st, "loom_attn_decode_noalloc")
    return (o, lse) if (return_lse or lse is not None) else o


def loom_attn_fwd_varlen(q, k, v, cu_seqlens_q, cu_seqlens_k, max_seqlen_q, o=None, lse=None, *, causal=False,
                         scale=None, stream=None, return_lse=False):
    """Prefill over a ragged batch.  q [total_q, Hq, D], k/v [total_k, Hkv, D] bf16;
    cu_seqlens_q / cu_seqlens_k [B + 1] int32 on the device; max_seqlen_q an int.
    Returns ``o`` ([total_q, Hq, D]) or ``(o, lse)`` with lse [Hq, total_q]."""
    torch = _torch()
    bf16 = torch.bfloat16
    qp = _dev_ptr(q, "q", bf16, 3)
    kp = _dev_ptr(k, "k", bf16, 3)
    vp_ = _dev_ptr(v, "v", bf16, 3)
    total_q, Hq, D = q.shape
    total_k, Hkv, Dk = k.shape
    if tuple(v.shape) != tuple(k.shape) or Dk != D:
        raise ValueError("varlen prefill takes q [total_q, Hq, D] and k/v [total_k, Hkv, D]")
    cqp = _dev_ptr(cu_seqlens_q, "cu_seqlens_q", torch.int32, 1)
    ckp = _dev_ptr(cu_seqlens_k, "cu_seqlens_k", torch.int32, 1)
    if cu_seqlens_q.numel() != cu_seqlens_k.numel() or cu_seqlens_q.numel() < 2:
        raise ValueError("cu_seqlens_q and cu_seqlens_k must both be [B + 1]")
    B = cu_seqlens_q.numel() - 1
    if o is None:
        o = torch.empty_like(q)
    op = _dev_ptr(o, "o", bf16, 3)
    if lse is None and return_lse:
        lse = torch.empty((Hq, total_q), dtype=torch.float32, device=q.device)
    lp = None
    if lse is not None:
        if lse.numel() != Hq * total_q:
            raise ValueError("lse must hold Hq*total_q values")
        lp = _dev_ptr(lse, "lse", torch.float32)
    if scale is None:
        scale = D ** -0.5
    st = capi().loom_attn_fwd_varlen(qp, kp, vp_, op, lp, cqp, ckp, B, Hq, Hkv, total_q, total_k,
                                     int(max_seqlen_q), D, int(bool(causal)), float(scale),
                                     _stream_ptr(stream, q.device))
    _check(st, "loom_attn_fwd_varlen")
    return (o, lse) if (return_lse or lse is not None) else o


def loom_attn_decode_paged(q, k_cache, v_cache, block_table, seqlens_k, o=None, lse=None, workspace=None, *,
                           scale=None, num_splits=0, stream=None, return_lse=False, layout="nhd"):
    """Flash Decode over a paged cache.  q [B,Hq,1,D]; k_cache/v_cache bf16, [num_pages,
    page_size, Hkv, D] (layout "nhd") or [num_pages, Hkv, page_size, D] (layout "hnd");
    block_table [B, max_pages] int32; seqlens_k [B] int32 (all on the device).  Returns
    ``o`` or ``(o, lse)``."""
    torch = _torch()
    bf16 = torch.bfloat16
    qp = _dev_ptr(q, "q", bf16, 4)
    kp = _dev_ptr(k_cache, "k_cache", bf16, 4)
    vp_ = _dev_ptr(v_cache, "v_cache", bf16, 4)
    B, Hq, Sq, D = q.shape
    if layout not in ("nhd", "hnd"):
        raise ValueError("layout is 'nhd' or 'hnd'")
    if layout == "nhd":
        num_pages, page_size, Hkv, Dk = k_cache.shape
    else:
        num_pages, Hkv, page_size, Dk = k_cache.shape
    if Sq != 1 or tuple(v_cache.shape) != tuple(k_cache.shape) or Dk != D:
        raise ValueError("paged decode takes q [B,Hq,1,D] and two caches of one shape")
    if block_table.dim() != 2 or block_table.shape[0] != B:
        raise ValueError("block_table must be [B, max_pages]")
    max_pages = block_table.shape[1]
    tp = _dev_ptr(block_table, "block_table", torch.int32, 2)
    if tuple(seqlens_k.shape) != (B,):
        raise ValueError("seqlens_k must be [B]")
    sp = _dev_ptr(seqlens_k, "seqlens_k", torch.int32)
    if o is None:
        o = torch.empty_like(q)
    op = _dev_ptr(o, "o", bf16, 4)
    if lse is None and return_lse:
        lse = torch.empty((B, Hq), dtype=torch.float32, device=q.device)
    lp = None
    if lse is not None:
        if lse.numel() != B * Hq:
            raise ValueError("lse must hold B*Hq values")
        lp = _dev_ptr(lse, "lse", torch.float32)
    Skv = max_pages * page_size
    if workspace is None:
        need = loom_attn_decode_workspace_bytes(B, Hq, Hkv, Skv, D, num_splits)
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=q.device)
    wp = _dev_ptr(workspace, "workspace")
    if scale is None:
        scale = D ** -0.5
    st = capi().loom_attn_decode_paged(qp, kp, vp_, tp, sp, op, lp, wp, workspace.numel() * workspace.element_size(),
                                       B, Hq, Hkv, num_pages, page_size, max_pages, 0 if layout == "nhd" else 1,
                                       D, float(scale),
                                       int(num_splits), _stream_ptr(stream, q.device))
    _check(st, "loom_attn_decode_paged")
    return (o, lse) if (return_lse or lse is not None) else o


def loom_attn_check_error(stream=None, device=None):
    """Synchronise and raise ``LoomError`` if a kernel abandoned a bounded wait."""
    st = capi().loom_attn_check_error(_stream_ptr(stream, device))
    _check(st, "loom_attn_check_error")


def loom_status_string(status: int) -> str:
    return capi().loom_status_string(int(status)).decode()


def loom_debug_set_timeout_ns(ns: int):
    capi().loom_debug_set_timeout_ns(int(ns))


def loom_debug_inject(mode: int):
    capi().loom_debug_inject(int(mode))


def loom_debug_prefill_design(design: int):
    capi().loom_debug_prefill_design(int(design))


def loom_model_fwd_plan(D: int) -> dict:
    plan = FwdPlan()
    _check(capi().loom_model_fwd_plan(int(D), ctypes.byref(plan)), "loom_model_fwd_plan")
    return plan.as_dict()


def loom_model_fwd_plan_variant(D: int, design: int):
    """Best plan of one prefill design (1, 2 or 3), or None if the design is infeasible at D."""
    plan = FwdPlan()
    st = capi().loom_model_fwd_plan_variant(int(D), int(design), ctypes.byref(plan))
    if st == 2:  # LOOM_ERR_UNSUPPORTED
        return None
    _check(st, "loom_model_fwd_plan_variant")
    return plan.as_dict()


def loom_model_heg_pipe(l: float, m: float, s: float, b_lm: int, b_ms: int) -> float:
    return float(capi().loom_model_heg_pipe(float(l), float(m), float(s), int(b_lm), int(b_ms)))


def loom_gemm_bf16(a, b, c=None, *, stream=None, b_transposed=False):
    """C = A B (bf16, fp32 accumulation): a [M, K] and b [K, N] bf16 CUDA tensors, or with
    ``b_transposed`` b [N, K] and C = A b^T (a linear layer's weight); writes and returns c
    ([M, N] bf16, allocated if None)."""
    torch = _torch()
    bf16 = torch.bfloat16
    ap = _dev_ptr(a, "a", bf16, 2)
    bp = _dev_ptr(b, "b", bf16, 2)
    M, K = a.shape
    if b_transposed:
        N, K2 = b.shape
    else:
        K2, N = b.shape
    if K2 != K:
        raise ValueError(f"a is [M, {K}] but b has {K2} along K")
    if c is None:
        c = torch.empty((M, N), dtype=bf16, device=a.device)
    cp = _dev_ptr(c, "c", bf16, 2)
    if tuple(c.shape) != (M, N):
        raise ValueError("c must be [M, N]")
    fn = capi().loom_gemm_bf16_bt if b_transposed else capi().loom_gemm_bf16
    _check(fn(ap, bp, cp, M, N, K, _stream_ptr(stream, a.device)), "loom_gemm_bf16")
    return c


def loom_gemm_tile_n(M, N, K) -> int:
    return int(capi().loom_gemm_tile_n(M, N, K))


def loom_gemm_splits(M, N, K) -> int:
    return int(capi().loom_gemm_splits(M, N, K))


def loom_model_gemm_time_us(M, N, K, tile_n, splits, num_sms) -> float:
    return float(capi().loom_model_gemm_time_us(M, N, K, tile_n, splits, num_sms))


def loom_debug_gemm_tile_n(tile_n: int):
    capi().loom_debug_gemm_tile_n(int(tile_n))


def loom_debug_gemm_splits(splits: int):
    capi().loom_debug_gemm_splits(int(splits))


def loom_gemm_cta_pair(M, N, K) -> int:
    return int(capi().loom_gemm_cta_pair(M, N, K))


def loom_debug_gemm_cta_pair(mode: int):
    capi().loom_debug_gemm_cta_pair(int(mode))


def loom_model_fwd_time_us_design(design, B, Hq, Sq, Skv, D, causal) -> float:
    """Modeled prefill time (us) with one design forced; negative if the design is infeasible."""
    return float(capi().loom_model_fwd_time_us_design(design, B, Hq, Sq, Skv, D, int(bool(causal))))


def loom_model_fwd_time_us(B, Hq, Sq, Skv, D, causal) -> float:
    return float(capi().loom_model_fwd_time_us(B, Hq, Sq, Skv, D, int(bool(causal))))


def loom_model_decode_time_us(splits, B, Hq, Hkv, Skv, D, num_sms) -> float:
    return float(capi().loom_model_decode_time_us(splits, B, Hq, Hkv, Skv, D, num_sms))


def loom_model_decode_cluster_time_us(splits, cluster, B, Hq, Hkv, Skv, D, clusters) -> float:
    return float(capi().loom_model_decode_cluster_time_us(splits, cluster, B, Hq, Hkv, Skv, D, clusters))


DECODE_SPLIT_MERGE, DECODE_PERSISTENT, DECODE_CLUSTER = 1, 2, 3


def loom_attn_decode_form(B, Hq, Hkv, Skv, D, num_splits=0, paged=False):
    """(form, cluster size) a decode call with these sizes runs: DECODE_SPLIT_MERGE,
    DECODE_PERSISTENT or DECODE_CLUSTER (with its cluster size; 0 otherwise); form -1 on
    invalid sizes."""
    cs = ctypes.c_int(0)
    f = int(capi().loom_attn_decode_form(B, Hq, Hkv, Skv, D, num_splits, int(bool(paged)), ctypes.byref(cs)))
    return f, int(cs.value)


def loom_model_decode_persistent_time_us(splits, B, Hq, Hkv, Skv, D, ctas) -> float:
    return float(capi().loom_model_decode_persistent_time_us(splits, B, Hq, Hkv, Skv, D, ctas))


def loom_model_decode_tc_time_us(splits, B, Hq, Hkv, Skv, D, num_sms) -> float:
    return float(capi().loom_model_decode_tc_time_us(splits, B, Hq, Hkv, Skv, D, num_sms))


def loom_decode_persistent_slots(D, G) -> int:
    return int(capi().loom_decode_persistent_slots(D, G))


def loom_decode_max_clusters(D, G, cluster) -> int:
    return int(capi().loom_decode_max_clusters(D, G, cluster))


def loom_debug_decode_form(form: int, cluster: int = 0) -> None:
    """Pin the Flash Decode form (DECODE_*; 0: the model's) and the cluster size (0: the model's)."""
    capi().loom_debug_decode_form(int(form), int(cluster))


def loom_debug_prefill_slots(D: int, slots: int) -> bool:
    """Pin the two-tile prefill's K/V ring depth (0: the model's); False if not compiled."""
    return bool(capi().loom_debug_prefill_slots(int(D), int(slots)))


def loom_debug_decode_stage_plan(tokens: int, stages: int = 0, ctas_per_sm: int = 0) -> bool:
    """Pin the decode split kernel's stage plan (tokens 0: the model's); False if not compiled."""
    return bool(capi().loom_debug_decode_stage_plan(int(tokens), int(stages), int(ctas_per_sm)))


def loom_debug_gemm_stages(stages: int) -> None:
    """Pin the GEMM's K-stage ring depth where a neighbour is compiled (0: the model's)."""
    capi().loom_debug_gemm_stages(int(stages))


def loom_debug_decode_tensor_cores(mode) -> None:
    """Split kernel of the split + merge decode on a contiguous cache: 1 / True (default)
    tensor cores, persistent; 2 tensor cores, one CTA per split; 0 / False CUDA cores."""
    capi().loom_debug_decode_tensor_cores(int(mode))


def loom_debug_gemm_order(group_rows: int = 0, k_alternate: int = 0) -> None:
    """Pin the GEMM's tile order: tile rows per group (0: the default) and the CTA-pair
    kernel's alternating K direction (-1: off; 0, 1: on)."""
    capi().loom_debug_gemm_order(int(group_rows), int(k_alternate))
