"""CPU oracle for the reordering and restoration of Zarya's inference modes.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this module. It shares no
code with the CUDA library and never imports it.

What it computes:

* Reordering (Sec. 5.1 step 2, Sec. 5.2 step 1): a sequence's positions are
  rearranged so that every unmasked (visible) token comes before every masked
  one. Within each group the original order is kept, except that the masked
  group may be put in a given order instead (the token shuffling of Mode A,
  Table 2: ``diffusion_shuffle``), by ascending key with ties broken by
  position. The result is the permutation perm (reordered index ->
  original position); the reordered tokens are tokens[perm], and perm itself
  is the position-id vector of the reordered sequence (a token keeps its
  original position for positional encoding; the order only decides what
  each token can attend to under the causal mask, Sec. 3.1 and Sec. 5.1).
* Restoration (Sec. 5.1 step 4, Sec. 5.2 step 8): the reordered sequence is
  put back in the original order, out[perm[i]] = x[i].

Readings where the paper is silent: the permutation convention (reordered
index -> original position), the stable order within each group, the
key order of the shuffled masked group (keys are inputs: the random numbers
the method draws are passed in), and positions at or past a sequence's
length being left out (perm -1, tokens untouched).
"""
from __future__ import annotations

import numpy as np


def reorder_one(is_masked, key=None):
    """Permutation of one sequence: unmasked positions in order, then masked
    positions in order (or by (key, position) when ``key`` is given)."""
    m = [bool(x) for x in np.asarray(is_masked)]
    n = len(m)
    visible = [i for i in range(n) if not m[i]]
    masked = [i for i in range(n) if m[i]]
    if key is not None:
        k = [int(x) for x in np.asarray(key)]
        masked = sorted(masked, key=lambda i: (k[i], i))
    return visible + masked


def reorder(tokens, is_masked, lens, order_key=None):
    """Batch reordering over ``[B, max_len]`` arrays; sequence b uses its
    first lens[b] positions. Returns (perm, tokens_out, n_unmasked) with
    perm / tokens_out ``[B, max_len]`` int32 (-1 / the input past lens[b])
    and n_unmasked ``[B]`` int32."""
    tok = np.asarray(tokens)
    msk = np.asarray(is_masked)
    B, max_len = tok.shape
    perm = np.full((B, max_len), -1, dtype=np.int32)
    out = np.array(tok, dtype=np.int32, copy=True)
    nvis = np.zeros(B, dtype=np.int32)
    for b in range(B):
        n = int(lens[b])
        key = None if order_key is None else np.asarray(order_key)[b, :n]
        p = reorder_one(msk[b, :n], key)
        perm[b, :n] = p
        out[b, :n] = [tok[b, i] for i in p]
        nvis[b] = sum(1 for i in range(n) if not msk[b, i])
    return perm, out, nvis


def restore(tokens, perm, lens):
    """Inverse of the reordering: out[b, perm[b, i]] = tokens[b, i] for
    i < lens[b]; positions past lens[b] keep the input's values."""
    tok = np.asarray(tokens)
    pm = np.asarray(perm)
    out = np.array(tok, dtype=np.int32, copy=True)
    for b in range(tok.shape[0]):
        for i in range(int(lens[b])):
            out[b, int(pm[b, i])] = tok[b, i]
    return out
