"""Device-resident state of one slot-decoding attention layer.

``DeviceBatch`` holds, on one GPU, everything a Mode B step (Sec. 5.2) of
one layer touches: the KV cache (contiguous or paged), the committed prefix
lengths, the block layout (slots x slot length per sequence, mask mode, row
offsets), the block's queries and keys/values, the accepted lengths, the
output and the library workspace. Its three methods are the three calls of
a step, all of which run in the library's kernels:

  stage()   zarya_kv_append(STAGE): block K/V -> cache positions P_b..
  attend()  zarya_slot_attn: out <- attention of the block over prefix+block
  commit()  zarya_kv_append(COMMIT): accepted rows -> cache, P_b += accepted
  commit_staged()  zarya_kv_commit_staged: P_b += accepted, for a block
            already staged (its accepted rows are in place)
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import numpy as np
import torch

from . import _binding as zb


@dataclass
class DeviceBatch:
    q: torch.Tensor
    k_cache: torch.Tensor
    v_cache: torch.Tensor
    k_new: torch.Tensor
    v_new: torch.Tensor
    out: torch.Tensor
    cache_lens: torch.Tensor
    n_slots: torch.Tensor
    slot_len: torch.Tensor
    mask_mode: torch.Tensor
    accept_len: torch.Tensor
    stage_len: torch.Tensor
    q_row_offsets: torch.Tensor
    page_table: Optional[torch.Tensor]
    desc: zb.AttnDesc
    workspace: Optional[torch.Tensor]

    def stage(self, stream=None) -> None:
        zb.kv_append(self.k_new, self.v_new, self.stage_len, self.k_cache, self.v_cache,
                     self.cache_lens, self.page_table, self.desc, commit=False, stream=stream)

    def attend(self, stream=None) -> None:
        zb.slot_attn(self.q, self.k_cache, self.v_cache, self.cache_lens, self.page_table,
                     self.n_slots, self.slot_len, self.mask_mode, self.out, self.desc,
                     self.workspace, stream=stream)

    def stage_and_attend(self, stream=None) -> None:
        """``stage`` then ``attend`` in one launch (zarya_slot_attn_staged)."""
        zb.slot_attn_staged(self.q, self.k_new, self.v_new, self.k_cache, self.v_cache,
                            self.cache_lens, self.page_table, self.n_slots, self.slot_len,
                            self.mask_mode, self.out, self.desc, self.workspace, stream=stream)

    def commit(self, stream=None, new_lens=None) -> None:
        """Append the accepted rows and advance the lengths: in place, or into
        ``new_lens`` (leaving ``cache_lens`` as it was) when given."""
        if new_lens is None:
            zb.kv_append(self.k_new, self.v_new, self.accept_len, self.k_cache, self.v_cache,
                         self.cache_lens, self.page_table, self.desc, commit=True, stream=stream)
        else:
            zb.kv_append_commit_to(self.k_new, self.v_new, self.accept_len, self.k_cache,
                                   self.v_cache, self.cache_lens, new_lens, self.page_table,
                                   self.desc, stream=stream)

    def commit_staged(self, stream=None, new_lens=None) -> None:
        """The commit after ``stage_and_attend`` (or ``stage``) of this block:
        its accepted rows are already in the cache, so only the lengths
        advance (in place, or into ``new_lens``)."""
        zb.kv_commit_staged(self.accept_len, self.cache_lens,
                            self.cache_lens if new_lens is None else new_lens, self.desc,
                            stream=stream)


def _i32(a, device) -> torch.Tensor:
    return torch.as_tensor(np.ascontiguousarray(a, dtype=np.int32)).to(device)


def upload(w, device="cuda", kv_splits: int = 0, mask_mode=None,
           caches: Optional[tuple] = None) -> DeviceBatch:
    """Copy a host workload (``workloads.Workload``) to ``device``.

    ``caches`` may pass already-resident (k_cache, v_cache) tensors to reuse.
    """
    dev = torch.device(device)
    mm = w.mask_mode if mask_mode is None else np.full(w.B, mask_mode, dtype=np.int32)
    dtype_code = zb.BF16 if w.dtype == "bf16" else zb.FP32
    offs = _i32(w.q_row_offsets, dev)
    R = w.R
    max_kv = int((w.cache_lens.astype(np.int64) + R).max())
    if caches is None:
        k_cache = w.k_cache.to(dev)
        v_cache = w.v_cache.to(dev)
    else:
        k_cache, v_cache = caches
    desc = zb.make_desc(batch=w.B, n_q_heads=w.Hq, n_kv_heads=w.Hkv, head_dim=w.D,
                        dtype=dtype_code, page_size=w.page_size, cache_capacity=w.capacity,
                        n_pages=w.n_pages, max_rows=w.max_rows, total_rows=w.rows,
                        q_row_offsets=offs, max_kv_len=max_kv, kv_splits=kv_splits,
                        scale=w.scale)
    ws_bytes = zb.workspace_size(desc)
    workspace = torch.zeros(ws_bytes, dtype=torch.uint8, device=dev) if ws_bytes else None
    return DeviceBatch(
        q=w.q.to(dev), k_cache=k_cache, v_cache=v_cache, k_new=w.k_new.to(dev),
        v_new=w.v_new.to(dev), out=torch.zeros_like(w.q, device=dev),
        cache_lens=_i32(w.cache_lens, dev), n_slots=_i32(w.n_slots, dev),
        slot_len=_i32(w.slot_len, dev), mask_mode=_i32(mm, dev),
        accept_len=_i32(w.accept_len, dev), stage_len=_i32(R, dev), q_row_offsets=offs,
        page_table=None if w.page_table is None else _i32(w.page_table, dev), desc=desc,
        workspace=workspace)


@dataclass
class SamplingBatch:
    """Device-resident state of slot selection and token acceptance
    (Sec. 5.2 steps 3-6) for one block: the draft logits and the
    verification logits, the block layout, and the outputs of both calls.

      draft()   zarya_draft_select: draws, confidences, selected slots and
                the verification layout (verify_row_offsets, verify_tokens)
      verify()  zarya_verify_accept over the verification logits, in the
                layout ``verify_offsets`` (the draft's own layout, or a given
                one) with tokens ``verify_tokens_in``: token probabilities,
                per-slot accepted prefixes and accept_len
    """
    draft_logits: torch.Tensor
    verify_logits: torch.Tensor
    n_slots: torch.Tensor
    slot_len: torch.Tensor
    row_offsets: torch.Tensor
    draft_tokens: torch.Tensor
    draft_prob: torch.Tensor
    slot_conf: torch.Tensor
    slot_selected: torch.Tensor
    n_selected: torch.Tensor
    verify_row_offsets: torch.Tensor
    verify_src_rows: torch.Tensor
    verify_tokens: torch.Tensor
    n_verify: torch.Tensor
    verify_offsets: torch.Tensor
    verify_tokens_in: torch.Tensor
    token_prob: torch.Tensor
    slot_accept: torch.Tensor
    accept_len: torch.Tensor
    draft_desc: zb.SampleDesc
    verify_desc: zb.SampleDesc

    def draft(self, stream=None) -> None:
        zb.draft_select(self.draft_logits, self.n_slots, self.slot_len, self.draft_tokens,
                        self.draft_prob, self.slot_conf, self.slot_selected, self.n_selected,
                        self.verify_row_offsets, self.verify_src_rows, self.verify_tokens,
                        self.draft_desc, stream=stream)

    def verify(self, stream=None) -> None:
        zb.verify_accept(self.verify_logits, self.verify_tokens_in, self.n_verify,
                         self.slot_len, self.token_prob, self.slot_accept, self.accept_len,
                         self.verify_desc, stream=stream)


def _padded_rows(x: torch.Tensor, rows: int, stride: int, device) -> torch.Tensor:
    """[rows, V] view, with row stride ``stride``, of a zero-filled buffer
    holding ``x`` in its first rows."""
    V = x.shape[1]
    if stride == V and x.shape[0] == rows:
        return x.to(device).contiguous()
    buf = torch.zeros((rows, stride), dtype=x.dtype, device=device)
    buf[: x.shape[0], :V] = x.to(device)
    return buf[:, :V]


def upload_sampling(w, device="cuda", *, temperature: float = 0.0,
                    slot_threshold: Optional[float] = None,
                    token_threshold: Optional[float] = None, seed: int = 0, offset: int = 0,
                    chain: bool = False) -> SamplingBatch:
    """Put a ``workloads.SamplingWorkload`` on ``device``. With ``chain`` the
    verification call reads the draft's own outputs (n_selected,
    verify_row_offsets, verify_tokens), as in a decoding step; otherwise it
    reads the workload's verification block (n_verify, verify_offsets,
    verify_tokens)."""
    from . import workloads as wl

    slot_threshold = wl.SLOT_THRESHOLD if slot_threshold is None else slot_threshold
    token_threshold = wl.TOKEN_THRESHOLD if token_threshold is None else token_threshold
    dtype = zb.BF16 if w.dtype == "bf16" else zb.FP32
    B, rows = w.B, w.rows
    vrows_buf = max(rows, 1)
    # rows padded to a multiple of 16 bytes (the library's alignment rule)
    epv = 8 if w.dtype == "bf16" else 4
    stride = (w.V + epv - 1) // epv * epv
    dl = _padded_rows(w.draft_logits, rows, stride, device)
    vl = _padded_rows(w.verify_logits, vrows_buf, stride, device)
    ms = w.max_slots
    i32 = lambda a: _i32(a, device)  # noqa: E731
    row_offsets = i32(w.row_offsets)
    verify_row_offsets = torch.zeros(B + 1, dtype=torch.int32, device=device)
    verify_tokens = torch.full((rows,), -1, dtype=torch.int32, device=device)
    n_selected = torch.zeros(B, dtype=torch.int32, device=device)
    if chain:
        n_verify, verify_offsets, verify_tokens_in = n_selected, verify_row_offsets, verify_tokens
    else:
        n_verify = i32(w.n_verify)
        verify_offsets = i32(w.verify_offsets)
        vt = np.full(vrows_buf, -1, dtype=np.int32)
        vt[: w.verify_rows] = w.verify_tokens
        verify_tokens_in = i32(vt)
    common = dict(batch=B, vocab=w.V, dtype=dtype, max_slots=ms, row_stride=stride,
                  temperature=temperature, slot_threshold=slot_threshold,
                  token_threshold=token_threshold, seed=seed, offset=offset)
    draft_desc = zb.make_sample_desc(total_rows=rows, row_offsets=row_offsets, **common)
    verify_desc = zb.make_sample_desc(total_rows=vrows_buf, row_offsets=verify_offsets, **common)
    f32 = dict(dtype=torch.float32, device=device)
    return SamplingBatch(
        draft_logits=dl, verify_logits=vl, n_slots=i32(w.n_slots), slot_len=i32(w.slot_len),
        row_offsets=row_offsets,
        draft_tokens=torch.full((rows,), -1, dtype=torch.int32, device=device),
        draft_prob=torch.full((rows,), float("nan"), **f32),
        slot_conf=torch.zeros((B, ms), **f32),
        slot_selected=torch.zeros((B, ms), dtype=torch.uint8, device=device),
        n_selected=n_selected, verify_row_offsets=verify_row_offsets,
        verify_src_rows=torch.full((rows,), -1, dtype=torch.int32, device=device),
        verify_tokens=verify_tokens, n_verify=n_verify, verify_offsets=verify_offsets,
        verify_tokens_in=verify_tokens_in,
        token_prob=torch.full((vrows_buf,), float("nan"), **f32),
        slot_accept=torch.zeros((B, ms), dtype=torch.int32, device=device),
        accept_len=torch.zeros(B, dtype=torch.int32, device=device),
        draft_desc=draft_desc, verify_desc=verify_desc)
