"""ctypes binding of ``libzarya.so`` (include/zarya.h).

Argument marshalling only: every step of slot attention and KV append runs
in the library's CUDA kernels. PyTorch supplies device memory and streams.
If the library is missing the calls raise; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libzarya.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "zarya.h")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_DEVICE_FAULT = 0, 1, 2, 3, 4
MASK_BIDIR_BLOCK, MASK_SLOT_CAUSAL = 0, 1
BF16, FP32 = 0, 1
APPEND_STAGE, APPEND_COMMIT = 0, 1
DEVERR_NAMES = {0: "none", 1: "page id", 2: "rows", 3: "capacity", 4: "accept length",
                5: "timeout", 6: "mask mode"}
DEVERR_TIMEOUT = 5
DEBUG_STALL = 1


class ZaryaError(RuntimeError):
    def __init__(self, status: int, what: str):
        msg = f"{what}: {status_string(status)} (status {status})"
        if status == ERR_CUDA:
            msg += f" [{last_error()}]"
        super().__init__(msg)
        self.status = status


class AttnDesc(ctypes.Structure):
    """Mirror of ``zarya_attn_desc``."""
    _fields_ = [
        ("batch", ctypes.c_int32),
        ("n_q_heads", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("dtype", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("cache_capacity", ctypes.c_int32),
        ("n_pages", ctypes.c_int32),
        ("max_rows", ctypes.c_int32),
        ("total_rows", ctypes.c_int32),
        ("max_kv_len", ctypes.c_int32),
        ("kv_splits", ctypes.c_int32),
        ("scale", ctypes.c_float),
        ("q_row_offsets", ctypes.c_void_p),
        ("wait_limit_us", ctypes.c_int32),
        ("debug_flags", ctypes.c_int32),
    ]


class SampleDesc(ctypes.Structure):
    """Mirror of ``zarya_sample_desc``."""
    _fields_ = [
        ("batch", ctypes.c_int32),
        ("vocab", ctypes.c_int32),
        ("dtype", ctypes.c_int32),
        ("max_slots", ctypes.c_int32),
        ("total_rows", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
        ("row_stride", ctypes.c_int64),
        ("temperature", ctypes.c_float),
        ("slot_threshold", ctypes.c_float),
        ("token_threshold", ctypes.c_float),
        ("reserved2", ctypes.c_uint32),
        ("seed", ctypes.c_uint64),
        ("offset", ctypes.c_uint64),
        ("row_offsets", ctypes.c_void_p),
    ]


_lib = None


def load() -> ctypes.CDLL:
    """Load the library (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing; build it with __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    dp = ctypes.POINTER(AttnDesc)
    lib.zarya_slot_attn_workspace_size.argtypes = [dp]
    lib.zarya_slot_attn_workspace_size.restype = sz
    # plan queries (a library built before them lacks these two; every
    # declared function's presence is checked by the tests)
    if hasattr(lib, "zarya_slot_attn_kernel"):
        lib.zarya_slot_attn_kernel.argtypes = [dp]
        lib.zarya_slot_attn_kernel.restype = ctypes.c_char_p
    if hasattr(lib, "zarya_slot_attn_launches"):
        lib.zarya_slot_attn_launches.argtypes = [dp]
        lib.zarya_slot_attn_launches.restype = i32
    lib.zarya_slot_attn.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, dp, vp]
    lib.zarya_slot_attn.restype = ctypes.c_int
    lib.zarya_slot_attn_staged.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz,
                                           dp, vp]
    lib.zarya_slot_attn_staged.restype = ctypes.c_int
    lib.zarya_slot_attn_noalloc.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, dp, vp]
    lib.zarya_slot_attn_noalloc.restype = ctypes.c_int
    lib.zarya_kv_append.argtypes = [vp, vp, vp, vp, vp, vp, vp, i32, dp, vp]
    lib.zarya_kv_append.restype = ctypes.c_int
    lib.zarya_kv_append_commit_to.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, dp, vp]
    lib.zarya_kv_append_commit_to.restype = ctypes.c_int
    lib.zarya_kv_commit_staged.argtypes = [vp, vp, vp, dp, vp]
    lib.zarya_kv_commit_staged.restype = ctypes.c_int
    lib.zarya_sample_rows.argtypes = [vp, vp, vp, ctypes.POINTER(SampleDesc), vp]
    lib.zarya_sample_rows.restype = ctypes.c_int
    lib.zarya_mode_a_budget.argtypes = [vp, i32, i32, ctypes.c_float, ctypes.c_uint64,
                                        ctypes.c_uint64, i32, vp, vp, vp]
    lib.zarya_mode_a_budget.restype = ctypes.c_int
    lib.zarya_reorder.argtypes = [vp, vp, vp, vp, i32, i32, vp, vp, vp, vp]
    lib.zarya_reorder.restype = ctypes.c_int
    lib.zarya_restore.argtypes = [vp, vp, vp, i32, i32, vp, vp]
    lib.zarya_restore.restype = ctypes.c_int
    sp = ctypes.POINTER(SampleDesc)
    lib.zarya_draft_select.argtypes = [vp] * 11 + [sp, vp]
    lib.zarya_draft_select.restype = ctypes.c_int
    lib.zarya_verify_accept.argtypes = [vp] * 7 + [sp, vp]
    lib.zarya_verify_accept.restype = ctypes.c_int
    lib.zarya_repetition_penalty.argtypes = [vp, vp, vp, i32, ctypes.c_float, sp, vp]
    lib.zarya_repetition_penalty.restype = ctypes.c_int
    lib.zarya_top_p.argtypes = [vp, ctypes.c_float, sp, vp]
    lib.zarya_top_p.restype = ctypes.c_int
    lib.zarya_copy.argtypes = [vp, vp, sz, vp]
    lib.zarya_copy.restype = ctypes.c_int
    lib.zarya_check_device_error.argtypes = [vp, ctypes.POINTER(i32)]
    lib.zarya_check_device_error.restype = ctypes.c_int
    lib.zarya_last_error.argtypes = []
    lib.zarya_last_error.restype = ctypes.c_char_p
    lib.zarya_status_string.argtypes = [ctypes.c_int]
    lib.zarya_status_string.restype = ctypes.c_char_p
    lib.zarya_version.argtypes = []
    lib.zarya_version.restype = i32
    _lib = lib
    return lib


def header_functions() -> list:
    """Names of the functions ``include/zarya.h`` declares."""
    with open(HEADER) as f:
        text = f.read()
    return sorted(set(re.findall(r"\b(zarya_[a-z0-9_]+)\s*\(", text)))


def status_string(status: int) -> str:
    return load().zarya_status_string(int(status)).decode()


def last_error() -> str:
    """The library's message about the last CUDA failure on this thread."""
    return load().zarya_last_error().decode()


def version() -> int:
    return int(load().zarya_version())


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check_cuda(name: str, t: torch.Tensor, dtype=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")


def make_desc(*, batch: int, n_q_heads: int, n_kv_heads: int, head_dim: int, dtype: int,
              page_size: int, cache_capacity: int, n_pages: int, max_rows: int,
              total_rows: int, q_row_offsets: torch.Tensor, max_kv_len: int = 0,
              kv_splits: int = 0, scale: float = 0.0, wait_limit_us: int = 0,
              debug_flags: int = 0) -> AttnDesc:
    _check_cuda("q_row_offsets", q_row_offsets, torch.int32)
    d = AttnDesc()
    d.batch, d.n_q_heads, d.n_kv_heads, d.head_dim = batch, n_q_heads, n_kv_heads, head_dim
    d.dtype, d.page_size, d.cache_capacity, d.n_pages = dtype, page_size, cache_capacity, n_pages
    d.max_rows, d.total_rows, d.max_kv_len, d.kv_splits = max_rows, total_rows, max_kv_len, kv_splits
    d.scale = scale
    d.wait_limit_us, d.debug_flags = wait_limit_us, debug_flags
    d.q_row_offsets = q_row_offsets.data_ptr()
    d._keep = q_row_offsets  # keep the offsets alive as long as the descriptor
    return d


def slot_attn_kernel(desc: AttnDesc) -> str:
    """``zarya_slot_attn_kernel``: the kernel the plan for ``desc`` launches."""
    return load().zarya_slot_attn_kernel(ctypes.byref(desc)).decode()


def slot_attn_launches(desc: AttnDesc) -> int:
    """``zarya_slot_attn_launches``: kernels one attention call launches."""
    return int(load().zarya_slot_attn_launches(ctypes.byref(desc)))


def workspace_size(desc: AttnDesc) -> int:
    return int(load().zarya_slot_attn_workspace_size(ctypes.byref(desc)))


def slot_attn(q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len, mask_mode, out,
              desc: AttnDesc, workspace: Optional[torch.Tensor] = None, stream=None) -> None:
    """``zarya_slot_attn``: out <- slot attention of q over the cache (Sec. 5.2)."""
    for name, t in (("q", q), ("k_cache", k_cache), ("v_cache", v_cache), ("out", out)):
        _check_cuda(name, t)
    for name, t in (("cache_lens", cache_lens), ("n_slots", n_slots), ("slot_len", slot_len),
                    ("mask_mode", mask_mode)):
        _check_cuda(name, t, torch.int32)
    if page_table is not None:
        _check_cuda("page_table", page_table, torch.int32)
    ws_bytes = 0
    if workspace is not None:
        _check_cuda("workspace", workspace)
        ws_bytes = workspace.numel() * workspace.element_size()
    st = load().zarya_slot_attn(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(cache_lens),
                                _ptr(page_table), _ptr(n_slots), _ptr(slot_len),
                                _ptr(mask_mode), _ptr(out), _ptr(workspace), ws_bytes,
                                ctypes.byref(desc), _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_slot_attn")


def slot_attn_staged(q, k_new, v_new, k_cache, v_cache, cache_lens, page_table, n_slots,
                     slot_len, mask_mode, out, desc: AttnDesc,
                     workspace: Optional[torch.Tensor] = None, stream=None) -> None:
    """``zarya_slot_attn_staged``: stage the block's own K/V into the cache
    and attend, in one launch (= stage append + ``zarya_slot_attn``)."""
    for name, t in (("q", q), ("k_new", k_new), ("v_new", v_new), ("k_cache", k_cache),
                    ("v_cache", v_cache), ("out", out)):
        _check_cuda(name, t)
    for name, t in (("cache_lens", cache_lens), ("n_slots", n_slots), ("slot_len", slot_len),
                    ("mask_mode", mask_mode)):
        _check_cuda(name, t, torch.int32)
    if page_table is not None:
        _check_cuda("page_table", page_table, torch.int32)
    ws_bytes = 0
    if workspace is not None:
        _check_cuda("workspace", workspace)
        ws_bytes = workspace.numel() * workspace.element_size()
    st = load().zarya_slot_attn_staged(_ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache),
                                       _ptr(v_cache), _ptr(cache_lens), _ptr(page_table),
                                       _ptr(n_slots), _ptr(slot_len), _ptr(mask_mode), _ptr(out),
                                       _ptr(workspace), ws_bytes, ctypes.byref(desc),
                                       _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_slot_attn_staged")


def slot_attn_noalloc(q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len,
                      mask_mode, out, desc: AttnDesc, stream=None) -> None:
    """``zarya_slot_attn_noalloc``: slot attention for callers that cannot
    allocate device memory when they run it. Its split-KV scratch is a fixed
    16 MiB array inside the library (one per GPU), so no workspace is passed
    and nothing is allocated; plans that need more scratch are rejected.
    Calls that overlap on the GPU share that array and must not be issued."""
    for name, t in (("q", q), ("k_cache", k_cache), ("v_cache", v_cache), ("out", out)):
        _check_cuda(name, t)
    for name, t in (("cache_lens", cache_lens), ("n_slots", n_slots), ("slot_len", slot_len),
                    ("mask_mode", mask_mode)):
        _check_cuda(name, t, torch.int32)
    if page_table is not None:
        _check_cuda("page_table", page_table, torch.int32)
    st = load().zarya_slot_attn_noalloc(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(cache_lens),
                                        _ptr(page_table), _ptr(n_slots), _ptr(slot_len),
                                        _ptr(mask_mode), _ptr(out), ctypes.byref(desc),
                                        _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_slot_attn_noalloc")


def kv_append(k_new, v_new, accept_len, k_cache, v_cache, cache_lens, page_table,
              desc: AttnDesc, commit: bool = True, stream=None) -> None:
    """``zarya_kv_append``: copy accepted rows into the cache (Sec. 5.2 step 7)."""
    for name, t in (("k_new", k_new), ("v_new", v_new), ("k_cache", k_cache),
                    ("v_cache", v_cache)):
        _check_cuda(name, t)
    _check_cuda("accept_len", accept_len, torch.int32)
    _check_cuda("cache_lens", cache_lens, torch.int32)
    if page_table is not None:
        _check_cuda("page_table", page_table, torch.int32)
    st = load().zarya_kv_append(_ptr(k_new), _ptr(v_new), _ptr(accept_len), _ptr(k_cache),
                                _ptr(v_cache), _ptr(cache_lens), _ptr(page_table),
                                APPEND_COMMIT if commit else APPEND_STAGE, ctypes.byref(desc),
                                _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_kv_append")


def kv_append_commit_to(k_new, v_new, accept_len, k_cache, v_cache, cache_lens, new_lens,
                        page_table, desc: AttnDesc, stream=None) -> None:
    """``zarya_kv_append_commit_to``: the commit with new_lens = cache_lens + accept_len
    written to a second array (cache_lens is only read)."""
    for name, t in (("k_new", k_new), ("v_new", v_new), ("k_cache", k_cache),
                    ("v_cache", v_cache)):
        _check_cuda(name, t)
    _check_cuda("accept_len", accept_len, torch.int32)
    _check_cuda("cache_lens", cache_lens, torch.int32)
    _check_cuda("new_lens", new_lens, torch.int32)
    if page_table is not None:
        _check_cuda("page_table", page_table, torch.int32)
    st = load().zarya_kv_append_commit_to(_ptr(k_new), _ptr(v_new), _ptr(accept_len),
                                          _ptr(k_cache), _ptr(v_cache), _ptr(cache_lens),
                                          _ptr(new_lens), _ptr(page_table), ctypes.byref(desc),
                                          _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_kv_append_commit_to")


def kv_commit_staged(accept_len, cache_lens, new_lens, desc: AttnDesc, stream=None) -> None:
    """``zarya_kv_commit_staged``: the commit of a block already staged in the
    cache, new_lens = cache_lens + accept_len (Sec. 5.2 step 7)."""
    _check_cuda("accept_len", accept_len, torch.int32)
    _check_cuda("cache_lens", cache_lens, torch.int32)
    _check_cuda("new_lens", new_lens, torch.int32)
    st = load().zarya_kv_commit_staged(_ptr(accept_len), _ptr(cache_lens), _ptr(new_lens),
                                       ctypes.byref(desc), _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_kv_commit_staged")


def sample_rows(logits, tokens, prob, desc: SampleDesc, stream=None) -> None:
    """``zarya_sample_rows``: the draw and its probability for every row in
    desc.row_offsets (Sec. 5.1 step 3, Sec. 5.2 steps 3-4)."""
    _check_logits(logits, desc)
    _check_cuda("tokens", tokens, torch.int32)
    _check_cuda("prob", prob, torch.float32)
    st = load().zarya_sample_rows(_ptr(logits), _ptr(tokens), _ptr(prob), ctypes.byref(desc),
                                  _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_sample_rows")


def repetition_penalty(logits, hist_offsets, hist_tokens, penalty: float, desc: SampleDesc,
                       stream=None) -> None:
    """``zarya_repetition_penalty``: in place, the logits of every token in a
    row's sequence history multiplied by ``penalty`` when negative, divided by
    it otherwise (Sec. 5.1 step 3, Table 2)."""
    _check_logits(logits, desc)
    _check_cuda("hist_offsets", hist_offsets, torch.int32)
    _check_cuda("hist_tokens", hist_tokens, torch.int32)
    st = load().zarya_repetition_penalty(_ptr(logits), _ptr(hist_offsets), _ptr(hist_tokens),
                                         hist_tokens.numel(), float(penalty), ctypes.byref(desc),
                                         _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_repetition_penalty")


def top_p(logits, top_p: float, desc: SampleDesc, stream=None) -> None:
    """``zarya_top_p``: in place, the logits outside each row's nucleus (the
    smallest most-probable set reaching ``top_p`` under softmax(x / T))
    become -inf (Sec. 5.1 step 3, Table 2)."""
    _check_logits(logits, desc)
    st = load().zarya_top_p(_ptr(logits), float(top_p), ctypes.byref(desc), _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_top_p")


def mode_a_budget(n_masked, T: int, alpha0: float, seed: int, offset: int, counts, n_steps,
                  stream=None) -> None:
    """``zarya_mode_a_budget``: per-step reveal counts of Mode A (Sec. 5.1
    step 1) into counts [B, max_steps] and n_steps [B]."""
    _check_cuda("n_masked", n_masked, torch.int32)
    _check_cuda("counts", counts, torch.int32)
    _check_cuda("n_steps", n_steps, torch.int32)
    B = n_masked.shape[0]
    if counts.dim() != 2 or counts.shape[0] != B:
        raise ValueError("counts must be [B, max_steps]")
    st = load().zarya_mode_a_budget(_ptr(n_masked), B, int(T), float(alpha0),
                                    int(seed) & (2 ** 64 - 1), int(offset) & (2 ** 64 - 1),
                                    counts.shape[1], _ptr(counts), _ptr(n_steps),
                                    _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_mode_a_budget")


def reorder(tokens, is_masked, lens, perm, tokens_out, n_unmasked, order_key=None,
            stream=None) -> None:
    """``zarya_reorder``: unmasked positions first, then masked ones (in order,
    or by ``order_key``); Sec. 5.1 step 2 / Sec. 5.2 step 1."""
    _check_cuda("tokens", tokens, torch.int32)
    _check_cuda("is_masked", is_masked, torch.uint8)
    _check_cuda("lens", lens, torch.int32)
    _check_cuda("perm", perm, torch.int32)
    _check_cuda("tokens_out", tokens_out, torch.int32)
    _check_cuda("n_unmasked", n_unmasked, torch.int32)
    if order_key is not None:
        _check_cuda("order_key", order_key, torch.int32)   # uint32 bits in an int32 tensor
    B, L = tokens.shape
    for name, t in (("is_masked", is_masked), ("perm", perm), ("tokens_out", tokens_out)):
        if tuple(t.shape) != (B, L):
            raise ValueError(f"{name} must be [{B}, {L}]")
    st = load().zarya_reorder(_ptr(tokens), _ptr(is_masked), _ptr(order_key), _ptr(lens), B, L,
                              _ptr(perm), _ptr(tokens_out), _ptr(n_unmasked), _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_reorder")


def restore(tokens, perm, lens, tokens_out, stream=None) -> None:
    """``zarya_restore``: back to the original order (Sec. 5.1 step 4 / Sec. 5.2
    step 8)."""
    _check_cuda("tokens", tokens, torch.int32)
    _check_cuda("perm", perm, torch.int32)
    _check_cuda("lens", lens, torch.int32)
    _check_cuda("tokens_out", tokens_out, torch.int32)
    B, L = tokens.shape
    st = load().zarya_restore(_ptr(tokens), _ptr(perm), _ptr(lens), B, L, _ptr(tokens_out),
                              _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_restore")


def copy(dst: torch.Tensor, src: torch.Tensor, stream=None) -> None:
    """``zarya_copy``: dst <- src (the same number of bytes) by a kernel; each
    tensor lives on the device or in pinned host memory, at least one on the
    device."""
    for name, t in (("src", src), ("dst", dst)):
        if not isinstance(t, torch.Tensor) or not (t.is_cuda or t.is_pinned()):
            raise TypeError(f"{name} must be a CUDA tensor or a pinned host tensor")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
    nbytes = src.numel() * src.element_size()
    if dst.numel() * dst.element_size() != nbytes:
        raise ValueError("src and dst differ in size")
    st = load().zarya_copy(_ptr(src), _ptr(dst), nbytes, _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_copy")


def make_sample_desc(*, batch: int, vocab: int, dtype: int, max_slots: int, total_rows: int,
                     row_stride: int, temperature: float, slot_threshold: float,
                     token_threshold: float, seed: int, offset: int,
                     row_offsets: torch.Tensor) -> SampleDesc:
    """Fill a ``zarya_sample_desc``; ``row_offsets`` (int32 [B + 1]) must stay alive."""
    _check_cuda("row_offsets", row_offsets, torch.int32)
    d = SampleDesc()
    d.batch, d.vocab, d.dtype = int(batch), int(vocab), int(dtype)
    d.max_slots, d.total_rows, d.reserved = int(max_slots), int(total_rows), 0
    d.row_stride = int(row_stride)
    d.temperature = float(temperature)
    d.slot_threshold = float(slot_threshold)
    d.token_threshold = float(token_threshold)
    d.reserved2 = 0
    d.seed = int(seed) & (2 ** 64 - 1)
    d.offset = int(offset) & (2 ** 64 - 1)
    d.row_offsets = row_offsets.data_ptr()
    return d


def _check_logits(logits, desc: SampleDesc):
    if not isinstance(logits, torch.Tensor) or not logits.is_cuda:
        raise TypeError("logits must be a CUDA tensor")
    want = torch.bfloat16 if desc.dtype == BF16 else torch.float32
    if logits.dtype != want:
        raise TypeError(f"logits must be {want}, got {logits.dtype}")
    if logits.dim() != 2 or logits.stride(1) != 1 or logits.stride(0) != desc.row_stride:
        raise ValueError("logits must be [rows, V] with row stride desc.row_stride")
    if logits.shape[0] < desc.total_rows or logits.shape[1] != desc.vocab:
        raise ValueError("logits shape does not match the descriptor")


def draft_select(logits, n_slots, slot_len, draft_tokens, draft_prob, slot_conf, slot_selected,
                 n_selected, verify_row_offsets, verify_src_rows, verify_tokens,
                 desc: SampleDesc, stream=None) -> None:
    """``zarya_draft_select``: draws, slot confidences, slot selection and the
    verification layout (Sec. 5.2 steps 3-5)."""
    _check_logits(logits, desc)
    for name, t in (("n_slots", n_slots), ("slot_len", slot_len), ("draft_tokens", draft_tokens),
                    ("n_selected", n_selected), ("verify_row_offsets", verify_row_offsets),
                    ("verify_src_rows", verify_src_rows), ("verify_tokens", verify_tokens)):
        _check_cuda(name, t, torch.int32)
    _check_cuda("draft_prob", draft_prob, torch.float32)
    _check_cuda("slot_conf", slot_conf, torch.float32)
    _check_cuda("slot_selected", slot_selected, torch.uint8)
    st = load().zarya_draft_select(_ptr(logits), _ptr(n_slots), _ptr(slot_len), _ptr(draft_tokens),
                                   _ptr(draft_prob), _ptr(slot_conf), _ptr(slot_selected),
                                   _ptr(n_selected), _ptr(verify_row_offsets),
                                   _ptr(verify_src_rows), _ptr(verify_tokens), ctypes.byref(desc),
                                   _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_draft_select")


def verify_accept(logits, tokens, n_slots, slot_len, token_prob, slot_accept, accept_len,
                  desc: SampleDesc, stream=None) -> None:
    """``zarya_verify_accept``: token probabilities and accepted prefixes of the
    verification block (Sec. 5.2 step 6)."""
    _check_logits(logits, desc)
    for name, t in (("tokens", tokens), ("n_slots", n_slots), ("slot_len", slot_len),
                    ("slot_accept", slot_accept), ("accept_len", accept_len)):
        _check_cuda(name, t, torch.int32)
    _check_cuda("token_prob", token_prob, torch.float32)
    st = load().zarya_verify_accept(_ptr(logits), _ptr(tokens), _ptr(n_slots), _ptr(slot_len),
                                    _ptr(token_prob), _ptr(slot_accept), _ptr(accept_len),
                                    ctypes.byref(desc), _stream(stream))
    if st != OK:
        raise ZaryaError(st, "zarya_verify_accept")


def check_device_error(stream=None) -> int:
    """Synchronise and return (and clear) the device error word (0 = none)."""
    code = ctypes.c_int32(0)
    st = load().zarya_check_device_error(_stream(stream), ctypes.byref(code))
    if st not in (OK, ERR_DEVICE_FAULT):
        raise ZaryaError(st, "zarya_check_device_error")
    return int(code.value)
