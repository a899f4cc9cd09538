"""Python binding of libnld (include/nld.h), with the C entry points' names.

Marshalling only: each function checks tensor dtypes, shapes and devices,
passes raw device pointers and the current CUDA stream to the C ABI, and
raises ``NldError`` on a non-OK status. Every step of the computation runs
in the library's CUDA kernels; there is no CPU fallback. If the library has
not been built, ``lib()`` raises instead of computing anything elsewhere.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional

import numpy as np
import torch

from . import build as _build

NLD_OK = 0
NLD_MODE_DIFFUSION = 0
NLD_MODE_VERIFY = 1
NLD_DEVERR_PREFIX_RANGE = 0x1
NLD_DEVERR_PAGE_RANGE = 0x2
NLD_DEVERR_WAIT_TIMEOUT = 0x4
NLD_ATTN_PREFIX_READY = 0x1
NLD_ATTN_NO_CLUSTER = 0x4

HEADER = os.path.join(_build.INCLUDE, "nld.h")


class NldError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {status_name(status)} ({status})")
        self.status = status


class AttnParams(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("num_q_heads", ctypes.c_int), ("num_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("page_size", ctypes.c_int), ("num_pages", ctypes.c_int),
                ("max_pages_per_seq", ctypes.c_int), ("num_splits", ctypes.c_int),
                ("softmax_scale", ctypes.c_float), ("flags", ctypes.c_uint)]


_lib = None


def lib(path: Optional[str] = None):
    """Load libnld.so (built by ``paper_2607_05722_gb300.build``)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or _build.LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libnld.so is not built ({p}); run __graft_entry__.build() first")
    L = ctypes.CDLL(p)
    V, I, Sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    PP = ctypes.POINTER(AttnParams)
    L.nld_block_attn_num_splits.argtypes = [PP, I]
    L.nld_block_attn_num_splits.restype = I
    L.nld_block_attn_workspace_size.argtypes = [PP, I]
    L.nld_block_attn_workspace_size.restype = Sz
    L.nld_block_attn.argtypes = [PP, V, V, V, V, V, I, I, V, V, V, Sz, V]
    L.nld_block_attn.restype = I
    L.nld_block_attn_partials.argtypes = [PP, V, V, V, V, V, I, I, V, V, V, Sz, V]
    L.nld_block_attn_partials.restype = I
    L.nld_block_attn_static_scratch.argtypes = [PP, V, V, V, V, V, I, I, V, V, V]
    L.nld_block_attn_static_scratch.restype = I
    L.nld_split_kv_combine.argtypes = [V, V, I, I, I, I, I, V, V, V]
    L.nld_split_kv_combine.restype = I
    L.nld_accept.argtypes = [V, V, I, I, V, V]
    L.nld_accept.restype = I
    L.nld_unmask.argtypes = [V, I, I, I, V, V, V]
    L.nld_unmask_threshold.argtypes = [V, I, I, ctypes.c_float, V, V, V]
    L.nld_unmask_threshold.restype = I
    L.nld_greedy_accept.argtypes = [V, V, V, I, I, V, V, V]
    L.nld_greedy_accept.restype = I
    L.nld_logits_argmax.argtypes = [V, I, I, I, V, V, V]
    L.nld_logits_argmax.restype = I
    L.nld_logits_ensemble_argmax.argtypes = [V, V, I, I, I, ctypes.c_float, V, V, V]
    L.nld_logits_ensemble_argmax.restype = I
    L.nld_kv_commit.argtypes = [PP, V, V, V, V, V, I, I, V, V, V]
    L.nld_kv_commit.restype = I
    L.nld_block_attn_masked.argtypes = [PP, V, V, V, V, V, I, V, V, V, V, Sz, V]
    L.nld_block_attn_masked.restype = I
    L.nld_quadss_block_mask.argtypes = [I, V]
    L.nld_quadss_block_mask.restype = I
    L.nld_unmask.restype = I
    L.nld_status_string.argtypes = [I]
    L.nld_status_string.restype = ctypes.c_char_p
    L.nld_device_error.argtypes = [ctypes.POINTER(ctypes.c_uint32), I]
    L.nld_device_error.restype = I
    L.nld_rescale_count.argtypes = [ctypes.POINTER(ctypes.c_uint64), I]
    L.nld_rescale_count.restype = I
    L.nld_check_wait_timeout.argtypes = [ctypes.c_uint64, V]
    L.nld_check_wait_timeout.restype = I
    L.nld_block_attn_kernels.argtypes = [PP, I]
    L.nld_block_attn_kernels.restype = I
    L.nld_block_attn_plan.argtypes = [PP, I, I, ctypes.POINTER(ctypes.c_int32)]
    L.nld_block_attn_plan.restype = I
    if path is None:
        _lib = L
    return L


def header_functions():
    """Names of the functions include/nld.h declares."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w]+\s*\**\s*(nld_\w+)\s*\(", text, flags=re.M)))


def status_name(status: int) -> str:
    try:
        return lib().nld_status_string(int(status)).decode()
    except RuntimeError:
        return str(status)


def _check(status: int, what: str):
    if status != NLD_OK:
        raise NldError(status, what)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _expect(t: torch.Tensor, dtype, shape, name):
    if t.dtype != dtype:
        raise TypeError(f"{name}: dtype {t.dtype}, expected {dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: shape {tuple(t.shape)}, expected {tuple(shape)}")
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name}: must be a contiguous CUDA tensor")


def make_params(batch, num_q_heads, num_kv_heads, head_dim, page_size, num_pages, max_pages_per_seq,
                num_splits=0, softmax_scale=0.0, flags=0) -> AttnParams:
    return AttnParams(batch, num_q_heads, num_kv_heads, head_dim, page_size, num_pages, max_pages_per_seq,
                      num_splits, softmax_scale, flags)


def params_for(q_block: torch.Tensor, k_pages: torch.Tensor, page_table: torch.Tensor, num_splits=0,
               softmax_scale=0.0, flags=0) -> AttnParams:
    B, bl, Hq, D = q_block.shape
    num_pages, Hkv, P, _ = k_pages.shape
    return make_params(B, Hq, Hkv, D, P, num_pages, page_table.shape[1], num_splits, softmax_scale, flags)


def nld_block_attn_num_splits(params: AttnParams, block_len: int) -> int:
    return int(lib().nld_block_attn_num_splits(ctypes.byref(params), block_len))


def nld_block_attn_kernels(params: AttnParams, block_len: int) -> int:
    """Kernels one nld_block_attn call launches (1 or 2) on the current device."""
    n = int(lib().nld_block_attn_kernels(ctypes.byref(params), block_len))
    if n < 0:
        raise NldError(1, "nld_block_attn_kernels")
    return n


def nld_block_attn_workspace_size(params: AttnParams, block_len: int) -> int:
    n = int(lib().nld_block_attn_workspace_size(ctypes.byref(params), block_len))
    if n == ctypes.c_size_t(-1).value:
        raise NldError(1, "nld_block_attn_workspace_size")
    return n


def workspace_views(params: AttnParams, block_len: int, workspace):
    """(o_part bf16 [S,B,Hq,bl,D], lse_part fp32 [S,B,Hq,bl]) views of a workspace laid out
    as include/nld.h documents, or None when the plan has one split."""
    S = nld_block_attn_num_splits(params, block_len)
    if S <= 1:
        return None
    B, Hq, D = params.batch, params.num_q_heads, params.head_dim
    n_o = S * B * Hq * block_len * D
    o0 = 0
    l0 = o0 + ((n_o * 2 + 255) // 256) * 256
    flat = workspace.view(torch.uint8)
    o_part = flat[o0:o0 + n_o * 2].view(torch.bfloat16).view(S, B, Hq, block_len, D)
    lse_part = flat[l0:l0 + S * B * Hq * block_len * 4].view(torch.float32).view(S, B, Hq, block_len)
    return o_part, lse_part


def alloc_workspace(params: AttnParams, block_len: int, device="cuda"):
    """A workspace for these parameters (None when the plan needs none)."""
    n = nld_block_attn_workspace_size(params, block_len)
    return torch.zeros(n, dtype=torch.uint8, device=device) if n else None


def nld_block_attn(params: AttnParams, q_block, k_pages, v_pages, page_table, prefix_lens, block_len: int,
                   mode: int, out, lse=None, workspace=None, stream=None, _entry="nld_block_attn"):
    """Masked block attention over the paged KV cache (see include/nld.h)."""
    B, Hq, Hkv, D, P = params.batch, params.num_q_heads, params.num_kv_heads, params.head_dim, params.page_size
    _expect(q_block, torch.bfloat16, (B, block_len, Hq, D), "q_block")
    _expect(k_pages, torch.bfloat16, (params.num_pages, Hkv, P, D), "k_pages")
    _expect(v_pages, torch.bfloat16, (params.num_pages, Hkv, P, D), "v_pages")
    _expect(page_table, torch.int32, (B, params.max_pages_per_seq), "page_table")
    _expect(prefix_lens, torch.int32, (B,), "prefix_lens")
    _expect(out, torch.bfloat16, (B, block_len, Hq, D), "out")
    if lse is not None:
        _expect(lse, torch.float32, (B, Hq, block_len), "lse")
    ws_bytes = 0
    if workspace is not None:
        if not workspace.is_cuda or not workspace.is_contiguous():
            raise ValueError("workspace: must be a contiguous CUDA tensor")
        ws_bytes = workspace.numel() * workspace.element_size()
    st = getattr(lib(), _entry)(ctypes.byref(params), _ptr(q_block), _ptr(k_pages), _ptr(v_pages), _ptr(page_table),
                              _ptr(prefix_lens), int(block_len), int(mode), _ptr(out), _ptr(lse), _ptr(workspace),
                              ws_bytes, _stream(stream))
    _check(st, _entry)


def nld_block_attn_partials(params: AttnParams, q_block, k_pages, v_pages, page_table, prefix_lens,
                            block_len: int, mode: int, out, lse=None, workspace=None, stream=None):
    """The attention kernel alone; with several splits only the workspace partials are written."""
    nld_block_attn(params, q_block, k_pages, v_pages, page_table, prefix_lens, block_len, mode, out, lse,
                   workspace, stream, _entry="nld_block_attn_partials")



def nld_block_attn_masked(params: AttnParams, q_block, k_pages, v_pages, page_table, prefix_lens, block_len: int,
                          block_mask, out, lse=None, workspace=None, stream=None):
    """nld_block_attn with the block part of the mask from block_mask (uint32
    [block_len] as int32 on the device; bit j: block slot j visible)."""
    B, Hq, Hkv, D, P = params.batch, params.num_q_heads, params.num_kv_heads, params.head_dim, params.page_size
    _expect(q_block, torch.bfloat16, (B, block_len, Hq, D), "q_block")
    _expect(k_pages, torch.bfloat16, (params.num_pages, Hkv, P, D), "k_pages")
    _expect(v_pages, torch.bfloat16, (params.num_pages, Hkv, P, D), "v_pages")
    _expect(page_table, torch.int32, (B, params.max_pages_per_seq), "page_table")
    _expect(prefix_lens, torch.int32, (B,), "prefix_lens")
    _expect(block_mask, torch.int32, (block_len,), "block_mask")
    _expect(out, torch.bfloat16, (B, block_len, Hq, D), "out")
    if lse is not None:
        _expect(lse, torch.float32, (B, Hq, block_len), "lse")
    ws_bytes = 0
    if workspace is not None:
        if not workspace.is_cuda or not workspace.is_contiguous():
            raise ValueError("workspace: must be a contiguous CUDA tensor")
        ws_bytes = workspace.numel() * workspace.element_size()
    st = lib().nld_block_attn_masked(ctypes.byref(params), _ptr(q_block), _ptr(k_pages), _ptr(v_pages),
                                     _ptr(page_table), _ptr(prefix_lens), int(block_len), _ptr(block_mask),
                                     _ptr(out), _ptr(lse), _ptr(workspace), ws_bytes, _stream(stream))
    _check(st, "nld_block_attn_masked")


def nld_quadss_block_mask(k: int):
    """The quadratic self-speculation table: numpy uint32 [1 + k + k^2]."""
    out = np.zeros((32,), dtype=np.uint32)
    n = lib().nld_quadss_block_mask(int(k), out.ctypes.data)
    if n < 0:
        raise ValueError(f"k={k}: 1 + k + k^2 slots must be at most 32")
    return out[:n].copy()

def nld_block_attn_static_scratch(params: AttnParams, q_block, k_pages, v_pages, page_table, prefix_lens,
                                  block_len: int, mode: int, out, lse=None, stream=None):
    """nld_block_attn without a workspace: the split partials live in a fixed
    16 MiB device array inside the library (for callers that cannot allocate)."""
    B, Hq, Hkv, D, P = params.batch, params.num_q_heads, params.num_kv_heads, params.head_dim, params.page_size
    _expect(q_block, torch.bfloat16, (B, block_len, Hq, D), "q_block")
    _expect(k_pages, torch.bfloat16, (params.num_pages, Hkv, P, D), "k_pages")
    _expect(v_pages, torch.bfloat16, (params.num_pages, Hkv, P, D), "v_pages")
    _expect(page_table, torch.int32, (B, params.max_pages_per_seq), "page_table")
    _expect(prefix_lens, torch.int32, (B,), "prefix_lens")
    _expect(out, torch.bfloat16, (B, block_len, Hq, D), "out")
    if lse is not None:
        _expect(lse, torch.float32, (B, Hq, block_len), "lse")
    st = lib().nld_block_attn_static_scratch(ctypes.byref(params), _ptr(q_block), _ptr(k_pages), _ptr(v_pages),
                                             _ptr(page_table), _ptr(prefix_lens), int(block_len), int(mode),
                                             _ptr(out), _ptr(lse), _stream(stream))
    _check(st, "nld_block_attn_static_scratch")


def nld_split_kv_combine(o_part, lse_part, out, lse=None, stream=None):
    """Merge split partials o_part bf16 [S,B,Hq,bl,D], lse_part fp32 [S,B,Hq,bl] into out [B,bl,Hq,D]."""
    S, B, Hq, bl, D = o_part.shape
    _expect(o_part, torch.bfloat16, (S, B, Hq, bl, D), "o_part")
    _expect(lse_part, torch.float32, (S, B, Hq, bl), "lse_part")
    _expect(out, torch.bfloat16, (B, bl, Hq, D), "out")
    if lse is not None:
        _expect(lse, torch.float32, (B, Hq, bl), "lse")
    st = lib().nld_split_kv_combine(_ptr(o_part), _ptr(lse_part), S, B, Hq, bl, D, _ptr(out), _ptr(lse),
                                    _stream(stream))
    _check(st, "nld_split_kv_combine")


def nld_accept(draft_ids, verify_ids, accepted_len, stream=None):
    """accepted_len[b] = first mismatch of draft vs verify ids, or n."""
    B, n = draft_ids.shape
    _expect(draft_ids, torch.int32, (B, n), "draft_ids")
    _expect(verify_ids, torch.int32, (B, n), "verify_ids")
    _expect(accepted_len, torch.int32, (B,), "accepted_len")
    _check(lib().nld_accept(_ptr(draft_ids), _ptr(verify_ids), B, n, _ptr(accepted_len), _stream(stream)),
           "nld_accept")


def nld_unmask(confidences, k: int, positions, num_selected=None, stream=None):
    """positions[b] = the k most confident eligible positions in rank order."""
    B, n = confidences.shape
    _expect(confidences, torch.float32, (B, n), "confidences")
    _expect(positions, torch.int32, (B, k), "positions")
    if num_selected is not None:
        _expect(num_selected, torch.int32, (B,), "num_selected")
    _check(lib().nld_unmask(_ptr(confidences), B, n, int(k), _ptr(positions), _ptr(num_selected),
                            _stream(stream)), "nld_unmask")



def nld_unmask_threshold(confidences, threshold: float, positions, num_selected=None, stream=None):
    """Commit every masked position with confidence > threshold, else the top-1
    (positions ascending, then -1)."""
    B, n = confidences.shape
    _expect(confidences, torch.float32, (B, n), "confidences")
    _expect(positions, torch.int32, (B, n), "positions")
    if num_selected is not None:
        _expect(num_selected, torch.int32, (B,), "num_selected")
    _check(lib().nld_unmask_threshold(_ptr(confidences), B, n, float(threshold), _ptr(positions),
                                      _ptr(num_selected), _stream(stream)), "nld_unmask_threshold")


def nld_greedy_accept(pred_ids, target_ids, confidences, positions, num_selected=None, stream=None):
    """Commit every masked position whose prediction equals the target, else the
    top-1 (positions ascending, then -1)."""
    B, n = confidences.shape
    _expect(pred_ids, torch.int32, (B, n), "pred_ids")
    _expect(target_ids, torch.int32, (B, n), "target_ids")
    _expect(confidences, torch.float32, (B, n), "confidences")
    _expect(positions, torch.int32, (B, n), "positions")
    if num_selected is not None:
        _expect(num_selected, torch.int32, (B,), "num_selected")
    _check(lib().nld_greedy_accept(_ptr(pred_ids), _ptr(target_ids), _ptr(confidences), B, n, _ptr(positions),
                                   _ptr(num_selected), _stream(stream)), "nld_greedy_accept")


def nld_logits_argmax(logits, ids, conf, vocab=None, stream=None):
    """Per row of bf16 logits [rows, ld]: the argmax over the first `vocab`
    entries (lowest index on ties) and the max softmax probability."""
    if logits.dtype != torch.bfloat16 or logits.dim() != 2 or not logits.is_cuda or logits.stride(1) != 1:
        raise ValueError("logits: a CUDA bf16 [rows, ld] tensor with unit column stride")
    rows, ld = logits.shape[0], logits.stride(0)
    vocab = logits.shape[1] if vocab is None else int(vocab)
    _expect(ids, torch.int32, (rows,), "ids")
    _expect(conf, torch.float32, (rows,), "conf")
    _check(lib().nld_logits_argmax(_ptr(logits), rows, vocab, ld, _ptr(ids), _ptr(conf), _stream(stream)),
           "nld_logits_argmax")



def nld_logits_ensemble_argmax(ar_logits, diff_logits, lam: float, ids, conf, vocab=None, stream=None):
    """Lowest argmax and max of lam * softmax(ar) + (1 - lam) * softmax(diff) per row."""
    for name, t in (("ar_logits", ar_logits), ("diff_logits", diff_logits)):
        if t.dtype != torch.bfloat16 or t.dim() != 2 or not t.is_cuda or t.stride(1) != 1:
            raise ValueError(f"{name}: a CUDA bf16 [rows, ld] tensor with unit column stride")
    if ar_logits.shape != diff_logits.shape or ar_logits.stride(0) != diff_logits.stride(0):
        raise ValueError("ar_logits and diff_logits: same shape and row stride")
    rows, ld = ar_logits.shape[0], ar_logits.stride(0)
    vocab = ar_logits.shape[1] if vocab is None else int(vocab)
    _expect(ids, torch.int32, (rows,), "ids")
    _expect(conf, torch.float32, (rows,), "conf")
    _check(lib().nld_logits_ensemble_argmax(_ptr(ar_logits), _ptr(diff_logits), rows, vocab, ld, float(lam),
                                            _ptr(ids), _ptr(conf), _stream(stream)), "nld_logits_ensemble_argmax")

def nld_kv_commit(params: AttnParams, k_new, v_new, counts, page_table, prefix_lens, block_len: int, advance: bool,
                  k_pages, v_pages, stream=None):
    """Write rows j < counts[b] (all block_len rows when counts is None) of the
    block K/V [B, bl, Hkv, D] to slots prefix_lens[b] + j; advance the prefix."""
    B, Hkv, D, P = params.batch, params.num_kv_heads, params.head_dim, params.page_size
    _expect(k_new, torch.bfloat16, (B, block_len, Hkv, D), "k_new")
    _expect(v_new, torch.bfloat16, (B, block_len, Hkv, D), "v_new")
    if counts is not None:
        _expect(counts, torch.int32, (B,), "counts")
    _expect(page_table, torch.int32, (B, params.max_pages_per_seq), "page_table")
    _expect(prefix_lens, torch.int32, (B,), "prefix_lens")
    _expect(k_pages, torch.bfloat16, (params.num_pages, Hkv, P, D), "k_pages")
    _expect(v_pages, torch.bfloat16, (params.num_pages, Hkv, P, D), "v_pages")
    _check(lib().nld_kv_commit(ctypes.byref(params), _ptr(k_new), _ptr(v_new), _ptr(counts), _ptr(page_table),
                               _ptr(prefix_lens), int(block_len), int(bool(advance)), _ptr(k_pages), _ptr(v_pages),
                               _stream(stream)), "nld_kv_commit")

def nld_block_attn_plan(params: AttnParams, block_len: int, sm_count: int) -> dict:
    """Host-only split plan for sm_count SMs: explicit split counts as launched
    (clusters included); automatic plans as if no cluster were resident."""
    out = (ctypes.c_int32 * 4)()
    if lib().nld_block_attn_plan(ctypes.byref(params), block_len, sm_count, out) != 0:
        raise NldError(1, "nld_block_attn_plan")
    return {"splits": out[0], "chunk": out[1], "cluster": out[2], "partials": out[3]}


def nld_check_wait_timeout(limit_ns: int, stream=None) -> None:
    """Launch the bounded-wait check: one wait that nothing completes gives up
    after limit_ns and sets NLD_DEVERR_WAIT_TIMEOUT."""
    _check(lib().nld_check_wait_timeout(ctypes.c_uint64(int(limit_ns)), _stream(stream)),
           "nld_check_wait_timeout")


def nld_device_error(clear: bool = False) -> int:
    bits = ctypes.c_uint32(0)
    _check(lib().nld_device_error(ctypes.byref(bits), 1 if clear else 0), "nld_device_error")
    return int(bits.value)


def nld_rescale_count(clear: bool = False) -> int:
    """Running-max rescale events of the attention kernels on this device."""
    n = ctypes.c_uint64(0)
    _check(lib().nld_rescale_count(ctypes.byref(n), 1 if clear else 0), "nld_rescale_count")
    return int(n.value)


def nld_status_string(status: int) -> str:
    return lib().nld_status_string(int(status)).decode()
