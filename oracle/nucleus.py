"""CPU oracle for top_p (nucleus) truncation of Zarya's per-step draws.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this module. It shares no
code with the CUDA library and never imports it. Arithmetic is fp64.

What it computes: Sec. 5.1 step 3 says the per-step draws honour the usual
sampling parameters (temperature, top_p, repetition_penalty), and Table 2
lists them for both inference modes. The paper names the parameter only.

Reading (nucleus sampling, Holtzman et al., "The curious case of neural text
degeneration", 2020): over a row's distribution p = softmax(x / T) (softmax(x)
at T = 0, as for the row probabilities of ``oracle.sampling``), keep the
smallest set of most probable tokens whose total probability reaches top_p;
tokens whose probability equals that of the least probable kept token are
all kept (a tie at the boundary is never split), so the kept set is
{v : x_v >= x*} for one logit value x*. top_p >= 1 keeps every token. The
draw is the draw of ``oracle.sampling`` restricted to the kept set (the same
per-token Gumbel noise, so a token keeps its noise whether or not others are
cut), and a token's probability is renormalised over the kept set (0 for a
token outside it).
"""
from __future__ import annotations

import numpy as np

from . import sampling as smp


def _probs(x, temperature: float) -> np.ndarray:
    t = float(temperature) if temperature > 0 else 1.0
    y = np.asarray(x, dtype=np.float64) / t
    e = np.exp(y - y.max())
    return e / e.sum()


def kept_threshold(x, temperature: float, top_p: float) -> float:
    """x*: the smallest logit of the kept set (-inf when every token is kept)."""
    x = np.asarray(x, dtype=np.float64)
    if top_p >= 1.0:
        return -np.inf
    p = _probs(x, temperature)
    order = np.argsort(-x, kind="stable")
    mass = 0.0
    k = 0
    while k < x.size:
        # take every token with the next logit value at once (ties stay together)
        v = x[order[k]]
        j = k
        while j < x.size and x[order[j]] == v:
            mass += p[order[j]]
            j += 1
        if mass >= top_p:
            return float(v)
        k = j
    return -np.inf


def kept_mask(x, temperature: float, top_p: float) -> np.ndarray:
    return np.asarray(x, dtype=np.float64) >= kept_threshold(x, temperature, top_p)


def draw_token(x, temperature: float, top_p: float, seed: int, offset: int, row: int) -> int:
    """The draw of ``oracle.sampling.draw_token`` over the kept set only."""
    x = np.asarray(x, dtype=np.float64)
    keep = kept_mask(x, temperature, top_p)
    if temperature > 0:
        z = x / float(temperature) + smp.gumbel_noise(seed, offset, row, x.size)
    else:
        z = x
    best = int(np.flatnonzero(keep)[0])
    for v in range(z.size):   # first maximum among the kept tokens
        if keep[v] and z[v] > z[best]:
            best = v
    return best


def row_probability(x, token: int, temperature: float, top_p: float) -> float:
    """The renormalised probability of ``token`` over the kept set."""
    keep = kept_mask(x, temperature, top_p)
    if not keep[token]:
        return 0.0
    p = _probs(x, temperature)
    return float(p[token] / p[keep].sum())
