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
