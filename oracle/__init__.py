"""CPU oracle for Zarya slot attention and KV append (fp64, plain and slow).

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package. It shares no
code with the CUDA library and never imports it.

The package holds these formulations, each written from the paper:

* ``slot_attn`` / ``slot_attn_rows``: the C implementation in
  ``slot_attn_oracle.c`` (masked softmax attention written out by its
  definition, fp64, OpenMP over (sequence, head)).
* ``slot_attn_dense``: a numpy brute force that materialises the dense mask of
  the whole reordered sequence (prefix then block) and applies it to a full
  score matrix; used to pin the C code on tiny shapes.
* ``kv_append``: the cache update with accepted tokens (Sec. 5.2 step 7) as a
  plain row copy in numpy.
* ``oracle.sampling``: slot selection and token acceptance (Sec. 5.2 steps
  3-6): draws, Gumbel-max sampling, slot confidences, the selection rule and
  the accepted prefixes, in numpy fp64.
* ``oracle.mode_a``: Mode A's mask-budget plan and per-step draws (Sec. 5.1
  steps 1 and 3).
* ``oracle.reorder``: reordering and restoration (Sec. 5.1 steps 2 and 4,
  Sec. 5.2 steps 1 and 8).
* ``oracle.penalty`` and ``oracle.nucleus``: the repetition penalty and top_p
  truncation the per-step draws honour (Sec. 5.1 step 3, Table 2).

Mask modes (Sec. 5.2):
  0  block-bidirectional (draft pass, step 3): block rows see the whole prefix
     and the whole block;
  1  slot-causal (verification pass, step 6): block row r sees the prefix and
     block rows 0..r, i.e. plain causal attention over the reordered sequence.
  2  slot-independent (step 6 for several selected slots at once, each
     verified on its own): block row r = s*L + j sees the prefix and rows
     s*L .. r of its own slot.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_SRC = os.path.join(_HERE, "slot_attn_oracle.c")

MODE_BIDIR_BLOCK = 0
MODE_SLOT_CAUSAL = 1
MODE_SLOT_INDEPENDENT = 2

_F64, _F32, _BF16 = 0, 1, 2


def build(force: bool = False) -> str:
    """Compile the C oracle with gcc + OpenMP into ``oracle/liboracle.so``."""
    import hashlib

    cmd_flags = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp"]
    with open(_SRC, "rb") as f:
        digest = hashlib.sha256(" ".join(cmd_flags).encode() + b"\0" + f.read()).hexdigest()
    stamp = _LIB_PATH + ".sha256"
    if not force and os.path.exists(_LIB_PATH) and os.path.exists(stamp):
        with open(stamp) as f:
            if f.read().strip() == digest:
                return _LIB_PATH
    tmp = _LIB_PATH + ".tmp%d" % os.getpid()
    subprocess.run(cmd_flags + ["-o", tmp, _SRC, "-lm"], check=True)
    os.replace(tmp, _LIB_PATH)
    with open(stamp + ".tmp", "w") as f:
        f.write(digest + "\n")
    os.replace(stamp + ".tmp", stamp)
    return _LIB_PATH


_lib = None


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        p = ctypes.c_void_p
        i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        common = [p, p, p, ctypes.c_int, p, p, i32, i32, i32, i64, p, p, p, p, i32, i32, i32,
                  i32, f64]
        lib.oracle_slot_attn.argtypes = common + [p, i32]
        lib.oracle_slot_attn.restype = ctypes.c_int
        lib.oracle_slot_attn_rows.argtypes = common + [p, i64, p, i32]
        lib.oracle_slot_attn_rows.restype = ctypes.c_int
        lib.oracle_max_threads.argtypes = []
        lib.oracle_max_threads.restype = ctypes.c_int
        _lib = lib
    return _lib


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def _as_numpy(x):
    """numpy view of a numpy array or CPU torch tensor; bf16 -> raw uint16."""
    if isinstance(x, np.ndarray):
        return x
    import torch  # only for CPU tensors handed in by tests

    if isinstance(x, torch.Tensor):
        x = x.detach()
        if x.is_cuda:
            raise ValueError("oracle takes host arrays only")
        if x.dtype == torch.bfloat16:
            return x.contiguous().view(torch.int16).numpy().view(np.uint16)
        return x.contiguous().numpy()
    return np.asarray(x)


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float64:
        return _F64
    if a.dtype == np.float32:
        return _F32
    if a.dtype == np.uint16:
        return _BF16
    raise TypeError(f"unsupported element type {a.dtype}")


def _i32(a, n=None):
    a = np.ascontiguousarray(_as_numpy(a), dtype=np.int32)
    if n is not None and a.size != n:
        raise ValueError("length mismatch")
    return a


def _prep(q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len, mask_mode,
          q_row_offsets):
    q = np.ascontiguousarray(_as_numpy(q))
    k = np.ascontiguousarray(_as_numpy(k_cache))
    v = np.ascontiguousarray(_as_numpy(v_cache))
    dt = _dtype_code(q)
    if _dtype_code(k) != dt or _dtype_code(v) != dt:
        raise TypeError("q, k and v must share one element type")
    B = int(np.asarray(_as_numpy(cache_lens)).size)
    lens = _i32(cache_lens, B)
    ns = _i32(n_slots, B)
    sl = _i32(slot_len, B)
    mm = _i32(mask_mode, B)
    if q_row_offsets is None:
        R = ns.astype(np.int64) * sl
        q_row_offsets = np.concatenate([[0], np.cumsum(R)])
    offs = np.ascontiguousarray(_as_numpy(q_row_offsets), dtype=np.int64)
    pt = None if page_table is None else _i32(page_table)
    return q, k, v, dt, lens, ns, sl, mm, offs, pt, B


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def slot_attn(q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len, mask_mode,
              q_row_offsets=None, *, scale: float, page_size: int = 0, capacity: int = 0,
              n_pages: int = -1, threads: int = 0) -> np.ndarray:
    """Full fp64 output ``[rows, Hq, D]`` of slot attention (Sec. 5.2 steps 3/6).

    ``q``: ``[rows, Hq, D]``; caches ``[B, capacity, Hkv, D]`` (``page_size`` 0)
    or ``[n_pages, page_size, Hkv, D]`` with ``page_table [B, max_pages]``.
    The block's own keys must already sit at cache positions ``P_b ..``.
    """
    q, k, v, dt, lens, ns, sl, mm, offs, pt, B = _prep(
        q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len, mask_mode, q_row_offsets)
    rows, Hq, D = q.shape
    Hkv = k.shape[-2]
    max_pages = 0 if pt is None else pt.shape[-1]
    out = np.zeros((rows, Hq, D), dtype=np.float64)
    rc = _load().oracle_slot_attn(
        _ptr(q), _ptr(k), _ptr(v), dt, _ptr(lens), _ptr(pt), max_pages, page_size, capacity,
        n_pages, _ptr(ns), _ptr(sl), _ptr(mm), _ptr(offs), B, Hq, Hkv, D, float(scale),
        _ptr(out), threads)
    if rc != 0:
        raise ValueError("oracle_slot_attn rejected its arguments")
    return out


def slot_attn_rows(q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len, mask_mode,
                   q_row_offsets=None, *, sel, scale: float, page_size: int = 0,
                   capacity: int = 0, n_pages: int = -1, threads: int = 0) -> np.ndarray:
    """fp64 outputs ``[n_sel, D]`` for the selected ``(b, h, r)`` triples only."""
    q, k, v, dt, lens, ns, sl, mm, offs, pt, B = _prep(
        q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len, mask_mode, q_row_offsets)
    rows, Hq, D = q.shape
    Hkv = k.shape[-2]
    max_pages = 0 if pt is None else pt.shape[-1]
    sel = np.ascontiguousarray(np.asarray(sel, dtype=np.int64).reshape(-1, 3))
    out = np.zeros((sel.shape[0], D), dtype=np.float64)
    rc = _load().oracle_slot_attn_rows(
        _ptr(q), _ptr(k), _ptr(v), dt, _ptr(lens), _ptr(pt), max_pages, page_size, capacity,
        n_pages, _ptr(ns), _ptr(sl), _ptr(mm), _ptr(offs), B, Hq, Hkv, D, float(scale),
        _ptr(sel), sel.shape[0], _ptr(out), threads)
    if rc != 0:
        raise ValueError("oracle_slot_attn_rows rejected its arguments")
    return out


# --------------------------------------------------------------------------
# numpy brute force (dense mask over the whole reordered sequence)

def _to_f64(a: np.ndarray) -> np.ndarray:
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def gather_sequence(cache, b: int, n_tokens: int, page_table=None, page_size: int = 0):
    """Logical tokens ``0 .. n_tokens-1`` of sequence ``b`` as ``[n, Hkv, D]``."""
    cache = _as_numpy(cache)
    if page_size == 0:
        return cache[b, :n_tokens]
    pt = _as_numpy(page_table)
    t = np.arange(n_tokens)
    return cache[pt[b, t // page_size], t % page_size]


def slot_attn_dense(q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len, mask_mode,
                    q_row_offsets=None, *, scale: float, page_size: int = 0) -> np.ndarray:
    """Brute force: per sequence, build the square mask of the reordered
    sequence [prefix ; block] (all-ones for mode 0's block rows, lower
    triangular for mode 1, block-diagonal lower triangular over the slots for
    mode 2), take the block's rows, and apply it to the full score matrix.
    fp64 throughout."""
    q = _as_numpy(q)
    lens = np.asarray(_as_numpy(cache_lens), dtype=np.int64)
    ns = np.asarray(_as_numpy(n_slots), dtype=np.int64)
    sl = np.asarray(_as_numpy(slot_len), dtype=np.int64)
    mm = np.asarray(_as_numpy(mask_mode), dtype=np.int64)
    B = lens.size
    if q_row_offsets is None:
        q_row_offsets = np.concatenate([[0], np.cumsum(ns * sl)])
    offs = np.asarray(_as_numpy(q_row_offsets), dtype=np.int64)
    rows, Hq, D = q.shape
    out = np.zeros((rows, Hq, D), dtype=np.float64)
    for b in range(B):
        P, R = int(lens[b]), int(ns[b] * sl[b])
        n = P + R
        K = _to_f64(gather_sequence(k_cache, b, n, page_table, page_size))  # [n, Hkv, D]
        V = _to_f64(gather_sequence(v_cache, b, n, page_table, page_size))
        Hkv = K.shape[1]
        g = Hq // Hkv
        K = np.repeat(K, g, axis=1)  # query head h reads kv head h // g
        V = np.repeat(V, g, axis=1)
        Q = _to_f64(q[offs[b]:offs[b] + R])  # [R, Hq, D]
        if mm[b] == MODE_SLOT_CAUSAL:
            full = np.tril(np.ones((n, n), dtype=bool))
        elif mm[b] == MODE_BIDIR_BLOCK:
            full = np.ones((n, n), dtype=bool)
        elif mm[b] == MODE_SLOT_INDEPENDENT:
            full = np.tril(np.ones((n, n), dtype=bool))
            L = int(sl[b])
            slot = np.arange(R) // L            # slot of each block position
            same = slot[:, None] == slot[None, :]
            full[P:, P:] &= same                # no key of another slot
        else:
            raise ValueError("bad mask mode")
        mask = full[P:P + R]  # block rows of the reordered sequence
        for h in range(Hq):
            s = scale * (Q[:, h, :] @ K[:, h, :].T)  # [R, n]
            s = np.where(mask, s, -np.inf)
            s = s - s.max(axis=1, keepdims=True)
            w = np.exp(s)
            w = w / w.sum(axis=1, keepdims=True)
            out[offs[b]:offs[b] + R, h, :] = w @ V[:, h, :]
    return out


# --------------------------------------------------------------------------
# KV append (Sec. 5.2 step 7)

def kv_append(k_new, v_new, accept_len, k_cache, v_cache, cache_lens, page_table=None,
              q_row_offsets=None, *, page_size: int = 0, commit: bool = True):
    """Copy rows ``q_row_offsets[b] + i`` (i < accept_len[b]) of ``k_new`` /
    ``v_new`` (``[rows, Hkv, D]``) to cache positions ``cache_lens[b] + i``.
    With ``commit`` the lengths advance by ``accept_len``; without it (staging
    the block's keys before its own attention pass) they stay. Returns new
    ``(k_cache, v_cache, cache_lens)``; the inputs are not modified. Values are
    moved bit for bit."""
    kc = np.array(_as_numpy(k_cache), copy=True)
    vc = np.array(_as_numpy(v_cache), copy=True)
    kn = _as_numpy(k_new)
    vn = _as_numpy(v_new)
    lens = np.array(_as_numpy(cache_lens), dtype=np.int64, copy=True)
    acc = np.asarray(_as_numpy(accept_len), dtype=np.int64)
    B = lens.size
    if q_row_offsets is None:
        q_row_offsets = np.concatenate([[0], np.cumsum(acc)])
    offs = np.asarray(_as_numpy(q_row_offsets), dtype=np.int64)
    pt = None if page_table is None else _as_numpy(page_table)
    for b in range(B):
        for i in range(int(acc[b])):
            t = int(lens[b]) + i
            src = int(offs[b]) + i
            if page_size == 0:
                kc[b, t] = kn[src]
                vc[b, t] = vn[src]
            else:
                page = int(pt[b, t // page_size])
                kc[page, t % page_size] = kn[src]
                vc[page, t % page_size] = vn[src]
    if commit:
        lens = lens + acc
    return kc, vc, lens.astype(np.int32)
