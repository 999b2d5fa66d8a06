"""CPU oracle for the repetition penalty of Zarya's per-step draws.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this module. It shares no
code with the CUDA library and never imports it.

What it computes: Sec. 5.1 step 3 says the per-step draws honour the usual
sampling parameters (temperature, top_p, repetition_penalty), and Table 2
lists them for both inference modes. The paper names the parameter only.

Reading (the penalised sampling of Keskar et al., "CTRL", 2019, in the form
a generate() call applies it): for every logits row of a sequence and every
distinct token that occurs in that sequence's history, a negative logit is
multiplied by the penalty and any other logit divided by it, so a penalty
above 1 always makes the token less likely. A token that occurs several
times is penalised once. The arithmetic is one float32 product or quotient
(the precision the logits come in), and bf16 logits are rounded back to bf16
to nearest even, so the result is a single correctly rounded operation that
both sides can reproduce bit for bit.
"""
from __future__ import annotations

import numpy as np


def bf16_round(x) -> np.ndarray:
    """float32 values rounded to the nearest bfloat16 (ties to even), as
    float32. Finite inputs only (the rounding of the 32-bit pattern: add
    0x7FFF plus the lowest kept bit, drop the low 16 bits)."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (b + 0x7FFF + ((b >> 16) & 1)) >> 16
    return (r.astype(np.uint32) << 16).view(np.float32)


def repetition_penalty(logits, row_offsets, hist_offsets, hist_tokens, penalty: float,
                       dtype: str = "fp32"):
    """The penalised copy of ``logits`` [rows, V] and whether a history token
    fell outside [0, V) (such tokens are skipped). Rows of sequence b are
    row_offsets[b] .. row_offsets[b + 1] - 1; its history is
    hist_tokens[hist_offsets[b] .. hist_offsets[b + 1] - 1]. Rows of no
    sequence are returned unchanged."""
    x = np.array(logits, dtype=np.float32, copy=True)
    V = x.shape[1]
    p = np.float32(penalty)
    bad = False
    B = len(row_offsets) - 1
    for b in range(B):
        hist = [int(t) for t in hist_tokens[int(hist_offsets[b]):int(hist_offsets[b + 1])]]
        bad = bad or any(t < 0 or t >= V for t in hist)
        toks = sorted({t for t in hist if 0 <= t < V})
        if not toks:
            continue
        for g in range(int(row_offsets[b]), int(row_offsets[b + 1])):
            v = x[g, toks]
            y = np.where(v < 0, v * p, v / p).astype(np.float32)
            x[g, toks] = bf16_round(y) if dtype == "bf16" else y
    return x, bad
