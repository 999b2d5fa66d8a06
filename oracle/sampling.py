"""CPU oracle for Zarya's Mode B slot selection and token acceptance.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this module. It shares no
code with the CUDA library and never imports it. Arithmetic is fp64 unless a
step below says otherwise.

What it computes (Sec. 5.2, Mode B, steps 3-6):

* Step 3, draft pass: every row of the block (S slots x L tokens per
  sequence, rows in slot order) draws a token from its logits, and the
  confidence of a slot is the probability of the token drawn at its first
  row.
* Step 4: with temperature T > 0 the draw is Gumbel-max sampling, the argmax
  over the vocabulary of x / T + g with g standard Gumbel noise (Gumbel 1935;
  the categorical sampler of masked diffusion models); with T = 0 it is the
  plain argmax of x. A row's probability is softmax(x / T) at the drawn token
  (softmax(x) when T = 0).
* Step 5: the slots whose confidence exceeds ``slot_threshold`` are selected;
  if none does, the single most confident slot is, so that one slot always
  goes on to verification.
* Step 6: the selected slots, concatenated in slot order, are verified. A
  verification row's probability is softmax(x / T) of its verification logits
  at the token drafted for it; a token is accepted while its probability
  exceeds ``token_threshold``. Per selected slot this gives its accepted
  prefix; over the concatenation, the accepted prefix length ``accept_len`` is
  what step 7 appends to the KV cache.

Readings where the paper is silent:

* Ties (equal logits, equal scores, equal confidences) go to the lowest index.
* "Exceeding" a threshold is strict (>).
* Verification logits come aligned: row k holds the distribution for the
  token at verification position k (any shift by one position of a causal
  model is done by whoever produces the logits).
* Gumbel noise is drawn from Philox4x32-10 (Salmon, Moraes, Dror, Shaw,
  "Parallel random numbers: as easy as 1, 2, 3", SC'11), keyed by the 64-bit
  seed and countered by (vocabulary index / 4, logits row, 64-bit offset);
  word (vocabulary index mod 4) of the output block gives the 32-bit draw w.
  It becomes u = fl32(fl32(w) * 2^-32 + 2^-33) in (0, 1] (float32 rounding,
  so both implementations start from the same u), then E = -log1p(-u) (a
  standard exponential variate) and g = -log(E) (a standard Gumbel variate),
  both in fp64 here.
"""
from __future__ import annotations

import numpy as np

# Philox4x32 round multipliers and Weyl key increments (Salmon et al., SC'11).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
PHILOX_ROUNDS = 10

_MASK32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(counter, key):
    """Philox4x32 with 10 rounds. ``counter`` is four uint32 values or
    arrays (broadcast together), ``key`` two. Each round multiplies counter
    words 0 and 2 by the two round constants into 64-bit products, and the
    new counter is (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2), hi(M0*c0) ^ c3 ^ k1,
    lo(M0*c0)); the key advances by the Weyl increments between rounds.
    Returns four uint32 arrays."""
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & _MASK32 for c in counter)
    k0, k1 = (np.asarray(k, dtype=np.uint64) & _MASK32 for k in key)
    m0, m1 = np.uint64(PHILOX_M0), np.uint64(PHILOX_M1)
    for rnd in range(PHILOX_ROUNDS):
        if rnd > 0:
            k0 = (k0 + np.uint64(PHILOX_W0)) & _MASK32
            k1 = (k1 + np.uint64(PHILOX_W1)) & _MASK32
        p0 = c0 * m0          # < 2^64: both factors < 2^32
        p1 = c2 * m1
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return tuple(c.astype(np.uint32) for c in (c0, c1, c2, c3))


def philox_words(seed: int, offset: int, row: int, n: int) -> np.ndarray:
    """The 32-bit draws w for vocabulary indices 0..n-1 of logits row ``row``:
    counter (v // 4, row, offset low word, offset high word), key (seed low
    word, seed high word), output word v % 4."""
    seed, offset = int(seed), int(offset)
    blocks = (n + 3) // 4
    ctr = (np.arange(blocks, dtype=np.uint64), np.uint64(row),
           np.uint64(offset & 0xFFFFFFFF), np.uint64((offset >> 32) & 0xFFFFFFFF))
    key = (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    out = philox4x32_10(ctr, key)
    w = np.empty(blocks * 4, dtype=np.uint32)
    for j in range(4):
        w[j::4] = out[j]
    return w[:n]


def uniform_from_words(w) -> np.ndarray:
    """u = fl32(fl32(w) * 2^-32 + 2^-33), evaluated in float32: in (0, 1]."""
    wf = np.asarray(w, dtype=np.uint32).astype(np.float32)
    return wf * np.float32(2.0 ** -32) + np.float32(2.0 ** -33)


def gumbel_from_uniform(u) -> np.ndarray:
    """g = -log(E) with E = -log1p(-u) exponential: standard Gumbel (fp64).
    u = 1 gives E = inf and g = -inf."""
    u = np.asarray(u, dtype=np.float64)
    with np.errstate(divide="ignore"):
        e = -np.log1p(-u)
        return -np.log(e)


def gumbel_noise(seed: int, offset: int, row: int, n: int) -> np.ndarray:
    """Gumbel noise for vocabulary indices 0..n-1 of logits row ``row``."""
    return gumbel_from_uniform(uniform_from_words(philox_words(seed, offset, row, n)))


def _f64(x) -> np.ndarray:
    return np.asarray(x, dtype=np.float64)


def row_probability(x, token: int, temperature: float) -> float:
    """softmax(x / T)[token] (T = 0 reads as T = 1), fp64, max-subtracted."""
    t = float(temperature) if temperature > 0 else 1.0
    y = _f64(x) / t
    m = y.max()
    return float(np.exp(y[token] - m) / np.exp(y - m).sum())


def draw_token(x, temperature: float, seed: int, offset: int, row: int) -> int:
    """Step 3 / step 4 draw for one row: argmax of x / T + g (T > 0) or of x
    (T = 0); the first maximum wins."""
    x = _f64(x)
    if temperature > 0:
        z = x / float(temperature) + gumbel_noise(seed, offset, row, x.size)
    else:
        z = x
    best = 0
    for v in range(1, z.size):   # first maximum: strict comparison
        if z[v] > z[best]:
            best = v
    return best


def _draw_token_fast(x, temperature, seed, offset, row):
    """Same draw as ``draw_token``, vectorised (np.argmax returns the first
    maximum). Used on full-size rows."""
    x = _f64(x)
    if temperature > 0:
        x = x / float(temperature) + gumbel_noise(seed, offset, row, x.size)
    return int(np.argmax(x))


def select_slots(conf, slot_threshold: float) -> np.ndarray:
    """Step 5: boolean mask of the selected slots. ``conf`` > threshold, or
    else only the most confident (first) slot."""
    conf = _f64(conf)
    sel = conf > float(slot_threshold)
    if conf.size and not sel.any():
        best = 0
        for s in range(1, conf.size):
            if conf[s] > conf[best]:
                best = s
        sel[best] = True
    return sel


def accept_prefix(token_prob, n_selected: int, slot_len: int, token_threshold: float):
    """Step 6 acceptance over the concatenation of ``n_selected`` slots of
    ``slot_len`` verification rows: returns (per-slot accepted prefix
    lengths, accepted prefix length of the whole concatenation)."""
    p = _f64(token_prob)[: n_selected * slot_len]
    passed = p > float(token_threshold)
    slot_acc = np.zeros(n_selected, dtype=np.int32)
    for k in range(n_selected):
        n = 0
        while n < slot_len and passed[k * slot_len + n]:
            n += 1
        slot_acc[k] = n
    total = 0
    while total < n_selected * slot_len and passed[total]:
        total += 1
    return slot_acc, int(total)


def _offsets(row_offsets, n_slots, slot_len):
    ns = np.asarray(n_slots, dtype=np.int64)
    sl = np.asarray(slot_len, dtype=np.int64)
    if row_offsets is None:
        row_offsets = np.concatenate([[0], np.cumsum(ns * sl)])
    return np.asarray(row_offsets, dtype=np.int64), ns, sl


def draft_select(logits, n_slots, slot_len, *, temperature: float, slot_threshold: float,
                 seed: int = 0, offset: int = 0, row_offsets=None, max_slots=None,
                 rows=None, fast: bool = False):
    """Steps 3-5 for a batch. ``logits`` is [total_rows, V] (read as fp64;
    bf16 callers pass the values widened to float32). Sequence b's block is
    rows row_offsets[b] .. row_offsets[b] + S_b L_b - 1 (default offsets: the
    running sum of S_b L_b), slot s in its rows s L_b .. s L_b + L_b - 1.

    Returns a dict with
      draft_tokens [total_rows] int32 and draft_prob [total_rows] float64
        (-1 / NaN on rows outside every block),
      slot_conf [B, max_slots] (0 past S_b), slot_selected [B, max_slots] uint8,
      n_selected [B] int32,
      verify_row_offsets [B + 1] int64: the verification block's layout, the
        running sum of n_selected_b L_b (its rows are packed densely),
      verify_src_rows [total_rows] int32: for verification row
        verify_row_offsets[b] + k, the global draft row it verifies (the
        selected slots' rows in slot order); -1 from verify_row_offsets[B] on,
      verify_tokens [total_rows] int32: the tokens drafted at those rows, -1 after.
    ``rows``, if given, restricts the per-row draw to those global rows (the
    other entries stay -1 / NaN and selection is skipped): for sampled checks
    of full-size workloads."""
    x = np.asarray(logits)
    offs, ns, sl = _offsets(row_offsets, n_slots, slot_len)
    B = ns.size
    total = int(x.shape[0])
    if max_slots is None:
        max_slots = int(ns.max()) if B else 0
    draw = _draw_token_fast if fast else draw_token
    tokens = np.full(total, -1, dtype=np.int32)
    prob = np.full(total, np.nan)
    active = np.zeros(total, dtype=bool)
    for b in range(B):
        active[offs[b]: offs[b] + ns[b] * sl[b]] = True
    todo = range(total) if rows is None else [int(r) for r in rows]
    for g in todo:
        if not active[g]:
            continue
        row = _f64(x[g])
        tok = draw(row, temperature, seed, offset, g)
        tokens[g] = tok
        prob[g] = row_probability(row, tok, temperature)
    out = dict(draft_tokens=tokens, draft_prob=prob)
    if rows is not None:
        return out
    conf = np.zeros((B, max_slots))
    sel = np.zeros((B, max_slots), dtype=np.uint8)
    n_sel = np.zeros(B, dtype=np.int32)
    voffs = np.zeros(B + 1, dtype=np.int64)
    src = np.full(total, -1, dtype=np.int32)
    vtok = np.full(total, -1, dtype=np.int32)
    for b in range(B):
        S, L, o = int(ns[b]), int(sl[b]), int(offs[b])
        c = np.array([prob[o + s * L] for s in range(S)])
        conf[b, :S] = c
        mask = select_slots(c, slot_threshold)
        sel[b, :S] = mask
        n_sel[b] = int(mask.sum())
        voffs[b + 1] = voffs[b] + n_sel[b] * L
        k = int(voffs[b])
        for s in range(S):
            if mask[s]:
                for j in range(L):
                    src[k] = o + s * L + j
                    vtok[k] = tokens[o + s * L + j]
                    k += 1
    out.update(slot_conf=conf, slot_selected=sel, n_selected=n_sel, verify_row_offsets=voffs,
               verify_src_rows=src, verify_tokens=vtok)
    return out


def verify_accept(logits, tokens, n_slots, slot_len, *, temperature: float,
                  token_threshold: float, row_offsets=None, max_slots=None, rows=None):
    """Step 6 for a batch. ``n_slots[b]`` is the number of slots verified for
    sequence b (n_selected of the draft) and its verification rows are
    row_offsets[b] .. row_offsets[b] + n_slots[b] L_b - 1 of ``logits``
    (default: packed densely), row k carrying token ``tokens[row]``.

    Returns token_prob [total_rows] (NaN outside every block),
    slot_accept [B, max_slots] int32 (0 past n_slots[b]), accept_len [B] int32.
    ``rows`` restricts the per-row probabilities as in ``draft_select``."""
    x = np.asarray(logits)
    offs, ns, sl = _offsets(row_offsets, n_slots, slot_len)
    tok = np.asarray(tokens, dtype=np.int64)
    B = ns.size
    total = int(x.shape[0])
    if max_slots is None:
        max_slots = int(ns.max()) if B else 0
    active = np.zeros(total, dtype=bool)
    for b in range(B):
        active[offs[b]: offs[b] + ns[b] * sl[b]] = True
    prob = np.full(total, np.nan)
    todo = range(total) if rows is None else [int(r) for r in rows]
    for g in todo:
        if active[g]:
            prob[g] = row_probability(x[g], int(tok[g]), temperature)
    if rows is not None:
        return dict(token_prob=prob)
    slot_acc = np.zeros((B, max_slots), dtype=np.int32)
    acc = np.zeros(B, dtype=np.int32)
    for b in range(B):
        n, L, o = int(ns[b]), int(sl[b]), int(offs[b])
        sa, a = accept_prefix(prob[o: o + n * L], n, L, token_threshold)
        slot_acc[b, :n] = sa
        acc[b] = a
    return dict(token_prob=prob, slot_accept=slot_acc, accept_len=acc)
