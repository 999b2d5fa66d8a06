"""Shared helpers of the GPU tests (comparison rules and oracle runs)."""
import numpy as np
import torch


def tolerance_ok(got, ref, dtype):
    """Parity rule: bf16 outputs max|err| <= 1e-2 and max|err| / max|ref| <=
    2e-2 against the fp64 oracle; fp32 outputs max|err| <= 1e-5."""
    g = got.detach().double().cpu().numpy() if isinstance(got, torch.Tensor) else got
    err = float(np.max(np.abs(g - ref))) if ref.size else 0.0
    scale = float(np.max(np.abs(ref))) if ref.size else 1.0
    if dtype == "fp32":
        return err <= 1e-5, err, scale
    return (err <= 1e-2 and err <= 2e-2 * scale), err, scale


def oracle_staged(oracle, w):
    """The oracle's caches after staging every block row (Sec. 5.2: the
    block's keys sit after the prefix while it attends)."""
    kc, vc, _ = oracle.kv_append(w.k_new, w.v_new, w.R, w.k_cache, w.v_cache, w.cache_lens,
                                 w.page_table, w.q_row_offsets, page_size=w.page_size,
                                 commit=False)
    return kc, vc


def oracle_full(oracle, w, kc, vc, mask_mode=None):
    mm = w.mask_mode if mask_mode is None else np.full(w.B, mask_mode, dtype=np.int32)
    return oracle.slot_attn(w.q, kc, vc, w.cache_lens, w.page_table, w.n_slots, w.slot_len, mm,
                            w.q_row_offsets, scale=w.scale, page_size=w.page_size,
                            capacity=w.capacity, n_pages=w.n_pages if w.page_size else -1)


def oracle_rows(oracle, w, kc, vc, sel, mask_mode=None):
    mm = w.mask_mode if mask_mode is None else np.full(w.B, mask_mode, dtype=np.int32)
    return oracle.slot_attn_rows(w.q, kc, vc, w.cache_lens, w.page_table, w.n_slots,
                                 w.slot_len, mm, w.q_row_offsets, sel=sel, scale=w.scale,
                                 page_size=w.page_size, capacity=w.capacity,
                                 n_pages=w.n_pages if w.page_size else -1)


def sample_rows(w, n, seed):
    """(b, h, r) triples: every sequence's first and last row at the first
    and last head, plus random ones."""
    rng = np.random.default_rng(seed)
    sel = []
    R = w.R
    for b in range(w.B):
        for h in (0, w.Hq - 1):
            sel.append((b, h, 0))
            sel.append((b, h, int(R[b]) - 1))
    while len(sel) < n:
        b = int(rng.integers(0, w.B))
        sel.append((b, int(rng.integers(0, w.Hq)), int(rng.integers(0, R[b]))))
    return np.asarray(sel, dtype=np.int64)


def gather_rows(out, w, sel):
    offs = w.q_row_offsets
    idx_rows = torch.as_tensor([int(offs[b]) + int(r) for b, _, r in sel])
    idx_heads = torch.as_tensor([int(h) for _, h, _ in sel])
    o = out.detach().cpu()
    return o[idx_rows, idx_heads].double().numpy()
