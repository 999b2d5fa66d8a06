"""Seeded synthetic inputs for the slot-attention workloads.

This module only draws numbers and lays them out; it holds none of the
attention or append arithmetic, so both the CUDA path and the CPU oracle can
consume what it makes without sharing code.

Recipe (same for every workload; integers first, in this order, then floats):
  rng = numpy.random.default_rng(seed)
  1. prefix lengths P_b   (fixed, uniform integer, or floor(exp(U(ln lo, ln hi))))
  2. slot lengths L_b     (fixed or uniform choice from a set); S_b slots each
  3. mask modes           (fixed, or uniform choice of {0, 1} per sequence)
  4. accepted lengths     (uniform integer in [lo, hi] clipped to R_b, or
                           uniform in [0, R_b])
  5. page permutation     (paged caches: a random permutation of all pages)
  6. Q, prefix K, prefix V, block K, block V ~ N(0, 1) drawn as float32 and
     rounded to the storage type (bf16 round-to-nearest-even, or fp32).
Cache positions at or beyond P_b hold a poison value (NaN) so that any read
past the valid keys shows up in the output.

Shapes follow the paper's model sizes (Table 1: 16/8 and 32/8 query/KV heads)
and its Mode B block structure (Sec. 5.2: S slots x L tokens per block).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, replace
from typing import Optional

import numpy as np
import torch

MODE_BIDIR_BLOCK = 0
MODE_SLOT_CAUSAL = 1

# name -> parameters. "both" modes means the workload is run once per mode.
SPECS = {
    # B1, 4/2 heads, D64, fp32, P=128 contiguous, 2 slots x 4 tokens, append 3.
    "tiny_fp32": dict(seed=0, B=1, Hq=4, Hkv=2, D=64, dtype="fp32", page_size=0,
                      prefix=("fixed", 128), n_slots=2, slot_len=("fixed", 4),
                      mode=("both",), accept=("fixed", 3)),
    # B8, 16/8 heads, D128, bf16, P=2048 contiguous, 4 x 8, slot-causal.
    "decode_small": dict(seed=1, B=8, Hq=16, Hkv=8, D=128, dtype="bf16", page_size=0,
                         prefix=("fixed", 2048), n_slots=4, slot_len=("fixed", 8),
                         mode=("fixed", MODE_SLOT_CAUSAL), accept=("upto_R",)),
    # B32, 32/8 heads, D128, bf16, P ~ U[512, 8192] contiguous, 8 x 16, bidirectional.
    "ragged_mid": dict(seed=2, B=32, Hq=32, Hkv=8, D=128, dtype="bf16", page_size=0,
                       prefix=("uniform", 512, 8192), n_slots=8, slot_len=("fixed", 16),
                       mode=("fixed", MODE_BIDIR_BLOCK), accept=("upto_R",)),
    # B4, 32/8 heads, D128, bf16, P=32768 contiguous, 16 x 32, both modes, accept U[0,512].
    "long_ctx": dict(seed=3, B=4, Hq=32, Hkv=8, D=128, dtype="bf16", page_size=0,
                     prefix=("fixed", 32768), n_slots=16, slot_len=("fixed", 32),
                     mode=("both",), accept=("uniform", 0, 512)),
    # B64, 32/8 heads, D128, bf16, paged (16-token pages, random permutation),
    # P log-uniform in [1024, 16384], L in {4, 8, 16, 32}, 8 slots, random mode.
    "serving_mix": dict(seed=4, B=64, Hq=32, Hkv=8, D=128, dtype="bf16", page_size=16,
                        prefix=("loguniform", 1024, 16384), n_slots=8,
                        slot_len=("choice", (4, 8, 16, 32)), mode=("random",),
                        accept=("upto_R",)),
}

# Reduced versions the oracle finishes in seconds; they keep every structural
# feature (GQA ratio, head dim, slot shapes, ragged tails, paging, modes).
SMALL = {
    "tiny_fp32": {},
    "decode_small": dict(B=3, prefix=("fixed", 300)),
    "ragged_mid": dict(B=4, prefix=("uniform", 37, 700)),
    "long_ctx": dict(B=1, prefix=("fixed", 1100)),
    "serving_mix": dict(B=6, prefix=("loguniform", 20, 900)),
}

ORDER = ["tiny_fp32", "decode_small", "ragged_mid", "long_ctx", "serving_mix"]


@dataclass
class Workload:
    name: str
    B: int
    Hq: int
    Hkv: int
    D: int
    dtype: str                  # "bf16" | "fp32"
    page_size: int              # 0 = contiguous cache
    capacity: int               # tokens per sequence (contiguous) / pages*page_size (paged)
    n_pages: int                # paged only (0 otherwise)
    cache_lens: np.ndarray      # int32 [B]   committed prefix P_b
    n_slots: np.ndarray         # int32 [B]
    slot_len: np.ndarray        # int32 [B]
    mask_mode: np.ndarray       # int32 [B]
    accept_len: np.ndarray      # int32 [B]
    q_row_offsets: np.ndarray   # int32 [B+1] exclusive prefix sum of R_b
    page_table: Optional[np.ndarray]  # int32 [B, max_pages] or None
    q: torch.Tensor             # [rows, Hq, D]
    k_cache: torch.Tensor       # [B, capacity, Hkv, D] or [n_pages, page_size, Hkv, D]
    v_cache: torch.Tensor
    k_new: torch.Tensor         # [rows, Hkv, D] block keys (staged before attention)
    v_new: torch.Tensor
    scale: float
    both_modes: bool = False

    @property
    def rows(self) -> int:
        return int(self.q_row_offsets[-1])

    @property
    def R(self) -> np.ndarray:
        return self.n_slots.astype(np.int64) * self.slot_len

    @property
    def max_rows(self) -> int:
        return int(self.R.max())

    @property
    def max_pages(self) -> int:
        return 0 if self.page_table is None else int(self.page_table.shape[1])

    def with_mode(self, mode: int) -> "Workload":
        return replace(self, mask_mode=np.full(self.B, mode, dtype=np.int32))


def _torch_dtype(name: str):
    return {"bf16": torch.bfloat16, "fp32": torch.float32}[name]


def _normal(rng, shape, dtype) -> torch.Tensor:
    a = rng.standard_normal(size=shape, dtype=np.float32)
    return torch.from_numpy(a).to(_torch_dtype(dtype))


def make(name: str, small: bool = False, seed: Optional[int] = None, **override) -> Workload:
    """Build workload ``name`` (see SPECS), optionally reduced (SMALL)."""
    spec = dict(SPECS[name])
    if small:
        spec.update(SMALL[name])
    spec.update(override)
    if seed is not None:
        spec["seed"] = seed
    rng = np.random.default_rng(spec["seed"])
    B, Hq, Hkv, D = spec["B"], spec["Hq"], spec["Hkv"], spec["D"]
    dtype, page_size, S = spec["dtype"], spec["page_size"], spec["n_slots"]

    # 1. prefix lengths
    kind = spec["prefix"]
    if kind[0] == "fixed":
        P = np.full(B, kind[1], dtype=np.int64)
    elif kind[0] == "uniform":
        P = rng.integers(kind[1], kind[2] + 1, size=B)
    elif kind[0] == "loguniform":
        P = np.floor(np.exp(rng.uniform(math.log(kind[1]), math.log(kind[2]), size=B)))
        P = np.clip(P.astype(np.int64), kind[1], kind[2])
    else:
        raise ValueError(kind)
    # 2. slot lengths
    kind = spec["slot_len"]
    if kind[0] == "fixed":
        L = np.full(B, kind[1], dtype=np.int64)
    else:
        L = rng.choice(np.asarray(kind[1], dtype=np.int64), size=B)
    n_slots = np.full(B, S, dtype=np.int64)
    R = n_slots * L
    # 3. mask modes
    kind = spec["mode"]
    both = kind[0] == "both"
    if kind[0] == "fixed":
        mode = np.full(B, kind[1], dtype=np.int64)
    elif kind[0] == "random":
        mode = rng.integers(0, 2, size=B)
    else:
        mode = np.full(B, MODE_SLOT_CAUSAL, dtype=np.int64)
    # 4. accepted lengths
    kind = spec["accept"]
    if kind[0] == "fixed":
        acc = np.minimum(np.full(B, kind[1], dtype=np.int64), R)
    elif kind[0] == "uniform":
        acc = np.minimum(rng.integers(kind[1], kind[2] + 1, size=B), R)
    else:
        acc = rng.integers(0, R + 1)
    offs = np.concatenate([[0], np.cumsum(R)]).astype(np.int64)
    rows = int(offs[-1])

    # 5. pages
    poison = float("nan")
    tdt = _torch_dtype(dtype)
    if page_size:
        pages_per_seq = (P + R + page_size - 1) // page_size
        n_pages = int(pages_per_seq.sum())
        perm = rng.permutation(n_pages).astype(np.int64)
        max_pages = int(pages_per_seq.max())
        page_table = np.full((B, max_pages), -1, dtype=np.int32)
        start = 0
        for b in range(B):
            page_table[b, :pages_per_seq[b]] = perm[start:start + pages_per_seq[b]]
            start += pages_per_seq[b]
        capacity = max_pages * page_size
        k_cache = torch.full((n_pages, page_size, Hkv, D), poison, dtype=tdt)
        v_cache = torch.full((n_pages, page_size, Hkv, D), poison, dtype=tdt)
    else:
        n_pages = 0
        page_table = None
        capacity = int((P + R).max())
        capacity = (capacity + 63) // 64 * 64
        k_cache = torch.full((B, capacity, Hkv, D), poison, dtype=tdt)
        v_cache = torch.full((B, capacity, Hkv, D), poison, dtype=tdt)

    # 6. values
    q = _normal(rng, (rows, Hq, D), dtype)
    for b in range(B):
        pb = int(P[b])
        kb = _normal(rng, (pb, Hkv, D), dtype)
        vb = _normal(rng, (pb, Hkv, D), dtype)
        if page_size:
            npg = (pb + page_size - 1) // page_size
            if npg:
                pad = npg * page_size - pb
                kfull = torch.cat([kb, torch.full((pad, Hkv, D), poison, dtype=tdt)])
                vfull = torch.cat([vb, torch.full((pad, Hkv, D), poison, dtype=tdt)])
                idx = torch.from_numpy(page_table[b, :npg].astype(np.int64))
                k_cache[idx] = kfull.view(npg, page_size, Hkv, D)
                v_cache[idx] = vfull.view(npg, page_size, Hkv, D)
        else:
            k_cache[b, :pb] = kb
            v_cache[b, :pb] = vb
    k_new = _normal(rng, (rows, Hkv, D), dtype)
    v_new = _normal(rng, (rows, Hkv, D), dtype)

    i32 = lambda a: np.ascontiguousarray(a, dtype=np.int32)  # noqa: E731
    return Workload(
        name=name + ("_small" if small else ""), B=B, Hq=Hq, Hkv=Hkv, D=D, dtype=dtype,
        page_size=page_size, capacity=capacity, n_pages=n_pages, cache_lens=i32(P),
        n_slots=i32(n_slots), slot_len=i32(L), mask_mode=i32(mode), accept_len=i32(acc),
        q_row_offsets=i32(offs), page_table=page_table, q=q, k_cache=k_cache,
        v_cache=v_cache, k_new=k_new, v_new=v_new, scale=1.0 / math.sqrt(D),
        both_modes=both)


# --------------------------------------------------------------------------
# Logits for slot selection and token acceptance (Sec. 5.2 steps 3-6).
#
# Recipe (rng = numpy.random.default_rng(seed); integers and peak draws first,
# in this order, then the base logits):
#   1. slot lengths L_b (fixed or uniform choice from a set); S_b slots each
#   2. verified slots n_b ~ uniform integer in [1, S_b] (the slot count of the
#      verification block, whose rows are packed densely)
#   3. per draft row: a peak with probability 0.7 at a uniform token, of
#      height ~ U(10, 22)
#   4. per verification row: its token, uniform in [0, V); a peak at that
#      token with probability 0.8, of height ~ U(8, 20), else at a uniform token
#   5. base logits ~ N(0, 2^2), drawn with torch.randn from a generator seeded
#      with ``seed`` on the target device, in float32; peaks are added, then
#      the values are rounded to the storage type (bf16 rounding makes ties
#      of the row maximum common in rows without a peak).
# With V = 151936 a row's softmax mass off the peak is about V e^2 ~ e^13.9,
# so peak heights in [10, 22] give first-token confidences from ~0.02 to
# ~1: both sides of the thresholds 0.9 / 0.4 occur.
# The vocabulary size is that of the Qwen3 backbone Zarya builds on.

QWEN3_VOCAB = 151936

SAMPLE_SPECS = {
    # small case for parity against the oracle: ragged V (not a multiple of 8)
    "select_tiny": dict(seed=20, B=3, V=20011, dtype="fp32", n_slots=3,
                        slot_len=("choice", (2, 3, 5))),
    # the decode_small block (B8, 4 slots x 8 tokens) over the full vocabulary
    "select_decode_small": dict(seed=21, B=8, V=QWEN3_VOCAB, dtype="bf16", n_slots=4,
                                slot_len=("fixed", 8)),
    # the serving_mix blocks (B64, 8 slots, L in {4, 8, 16, 32})
    "select_serving_mix": dict(seed=22, B=64, V=QWEN3_VOCAB, dtype="bf16", n_slots=8,
                               slot_len=("choice", (4, 8, 16, 32))),
    # the long_ctx blocks (B4, 16 slots x 32 tokens)
    "select_long_ctx": dict(seed=23, B=4, V=QWEN3_VOCAB, dtype="bf16", n_slots=16,
                            slot_len=("fixed", 32)),
}

SLOT_THRESHOLD = 0.9    # Sec. 6 evaluation settings
TOKEN_THRESHOLD = 0.4


@dataclass
class SamplingWorkload:
    name: str
    B: int
    V: int
    dtype: str
    n_slots: np.ndarray         # int32 [B]   S_b of the draft block
    slot_len: np.ndarray        # int32 [B]   L_b
    row_offsets: np.ndarray     # int32 [B+1] draft layout (running sum of S_b L_b)
    draft_logits: torch.Tensor  # [rows, V]
    n_verify: np.ndarray        # int32 [B]   slots in the verification block
    verify_offsets: np.ndarray  # int32 [B+1] running sum of n_b L_b
    verify_tokens: np.ndarray   # int32 [verify rows]
    verify_logits: torch.Tensor  # [verify rows, V]

    @property
    def rows(self) -> int:
        return int(self.row_offsets[-1])

    @property
    def verify_rows(self) -> int:
        return int(self.verify_offsets[-1])

    @property
    def max_slots(self) -> int:
        return int(self.n_slots.max())


def make_sampling(name: str, device="cpu", seed: Optional[int] = None,
                  **override) -> SamplingWorkload:
    """Build sampling workload ``name`` (SAMPLE_SPECS) with its logits on ``device``."""
    spec = dict(SAMPLE_SPECS[name])
    spec.update(override)
    if seed is not None:
        spec["seed"] = seed
    rng = np.random.default_rng(spec["seed"])
    B, V, S = spec["B"], spec["V"], spec["n_slots"]
    kind = spec["slot_len"]
    if kind[0] == "fixed":
        L = np.full(B, kind[1], dtype=np.int64)
    else:
        L = rng.choice(np.asarray(kind[1], dtype=np.int64), size=B)
    n_slots = np.full(B, S, dtype=np.int64)
    n_ver = rng.integers(1, n_slots + 1)
    offs = np.concatenate([[0], np.cumsum(n_slots * L)]).astype(np.int64)
    voffs = np.concatenate([[0], np.cumsum(n_ver * L)]).astype(np.int64)
    rows, vrows = int(offs[-1]), int(voffs[-1])
    d_peak = rng.random(rows) < 0.7
    d_tok = rng.integers(0, V, size=rows)
    d_h = rng.uniform(10.0, 22.0, size=rows)
    v_tok = rng.integers(0, V, size=vrows)
    v_on = rng.random(vrows) < 0.8
    v_other = rng.integers(0, V, size=vrows)
    v_h = rng.uniform(8.0, 20.0, size=vrows)

    gen = torch.Generator(device=device)
    gen.manual_seed(int(spec["seed"]))
    tdt = _torch_dtype(spec["dtype"])

    def logits(n, peak_rows, peak_tok, peak_h):
        x = torch.randn((n, V), generator=gen, device=device, dtype=torch.float32) * 2.0
        if len(peak_rows):
            r = torch.as_tensor(peak_rows, dtype=torch.int64, device=device)
            t = torch.as_tensor(peak_tok, dtype=torch.int64, device=device)
            h = torch.as_tensor(peak_h, dtype=torch.float32, device=device)
            x[r, t] += h
        return x.to(tdt)

    pr = np.nonzero(d_peak)[0]
    draft = logits(rows, pr, d_tok[pr], d_h[pr])
    vt = np.where(v_on, v_tok, v_other)
    verify = logits(vrows, np.arange(vrows), vt, v_h)
    i32 = lambda a: np.ascontiguousarray(a, dtype=np.int32)  # noqa: E731
    return SamplingWorkload(name=name, B=B, V=V, dtype=spec["dtype"], n_slots=i32(n_slots),
                            slot_len=i32(L), row_offsets=i32(offs), draft_logits=draft,
                            n_verify=i32(n_ver), verify_offsets=i32(voffs),
                            verify_tokens=i32(v_tok), verify_logits=verify)


# --------------------------------------------------------------------------
# Token rows for reordering / restoration (Sec. 5.1 steps 2/4, Sec. 5.2
# steps 1/8). Recipe (rng = numpy.random.default_rng(seed), in this order):
# sequence lengths ~ U{lo..max_len}; per sequence a mask fraction ~ U(0.1,
# 0.9) and per position a Bernoulli draw with it (masked positions scattered,
# as in Mode A's first-hitting sampling or fill-in-the-middle prompts);
# token ids ~ U{0..V-1}; order keys ~ U{0..2^32-1} (Mode A's token shuffling).
# max_len 2048 is the models' context length (Table 1).

REORDER_SPECS = {
    "reorder_small": dict(seed=30, B=4, max_len=300, lo=1),
    "reorder_serving": dict(seed=31, B=64, max_len=2048, lo=512),
}


@dataclass
class ReorderWorkload:
    name: str
    B: int
    max_len: int
    lens: np.ndarray        # int32 [B]
    tokens: np.ndarray      # int32 [B, max_len]
    is_masked: np.ndarray   # uint8 [B, max_len]
    order_key: np.ndarray   # uint32 [B, max_len]


def make_reorder(name: str, seed: Optional[int] = None) -> ReorderWorkload:
    spec = dict(REORDER_SPECS[name])
    if seed is not None:
        spec["seed"] = seed
    rng = np.random.default_rng(spec["seed"])
    B, L = spec["B"], spec["max_len"]
    lens = rng.integers(spec["lo"], L + 1, size=B).astype(np.int32)
    frac = rng.uniform(0.1, 0.9, size=(B, 1))
    mask = (rng.random((B, L)) < frac).astype(np.uint8)
    tokens = rng.integers(0, QWEN3_VOCAB, size=(B, L)).astype(np.int32)
    key = rng.integers(0, 2 ** 32, size=(B, L), dtype=np.uint64).astype(np.uint32)
    return ReorderWorkload(name=name, B=B, max_len=L, lens=lens, tokens=tokens,
                           is_masked=mask, order_key=key)
