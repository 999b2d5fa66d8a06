"""zarya_repetition_penalty against the oracle (oracle/penalty.py): bit for
bit on fp32 and bf16 rows, padded strides, empty and repeated histories,
rows of no sequence, the device checks, and a draw taken after the penalty."""
import numpy as np
import pytest
import torch

from oracle import penalty as pen
from oracle import sampling as smp

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def zb():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_19868_gb300 import build
    from paper_2609_19868_gb300 import _binding as zb

    build.build()
    zb.load()
    zb.check_device_error()
    return zb


def _i32(a):
    return torch.as_tensor(np.asarray(a, dtype=np.int32)).cuda()


def _case(zb, x, dtype, row_offsets, hist_offsets, hist, penalty):
    """Run the penalty on a padded copy of x [rows, V] (float32 values, bf16
    representable when dtype is bf16); returns the result as float32 values,
    the padding past the vocabulary, the error code, and (the logits view, the
    row offsets, the descriptor) for a call that follows."""
    rows, V = x.shape
    epv = 8 if dtype == torch.bfloat16 else 4
    stride = (V + epv - 1) // epv * epv + epv     # one spare vector of padding
    buf = torch.full((rows, stride), float("nan"), dtype=dtype, device="cuda")
    buf[:, :V] = torch.as_tensor(x).to(dtype).cuda()
    logits = buf.as_strided((rows, V), (stride, 1))
    ro, ho = _i32(row_offsets), _i32(hist_offsets)
    ht = _i32(hist if len(hist) else [0])[:len(hist)]
    d = zb.make_sample_desc(batch=len(row_offsets) - 1, vocab=V,
                            dtype=zb.BF16 if dtype == torch.bfloat16 else zb.FP32, max_slots=1,
                            total_rows=rows, row_stride=stride, temperature=0.0,
                            slot_threshold=0.9, token_threshold=0.4, seed=0, offset=0,
                            row_offsets=ro)
    zb.repetition_penalty(logits, ho, ht, penalty, d)
    torch.cuda.synchronize()
    err = zb.check_device_error()
    pad = buf[:, V:].float().cpu()
    return logits.float().cpu().numpy(), pad, err, (logits, ro, d)


def _inputs(rng, B, V, dtype, rows_per_seq=(0, 4), hist_len=(0, 300)):
    n_rows = rng.integers(rows_per_seq[0], rows_per_seq[1] + 1, size=B)
    row_offsets = np.concatenate([[0], np.cumsum(n_rows)]).astype(np.int32)
    rows = int(row_offsets[-1]) + 2                     # two rows of no sequence
    x = rng.normal(scale=3.0, size=(rows, V)).astype(np.float32)
    x[rng.random(size=x.shape) < 0.01] = 0.0
    x[rng.random(size=x.shape) < 0.01] = -0.0
    x[rng.random(size=x.shape) < 0.002] = -np.inf
    if dtype == torch.bfloat16:
        x = np.where(np.isfinite(x), pen.bf16_round(np.where(np.isfinite(x), x, 0.0)), x)
    n_hist = rng.integers(hist_len[0], hist_len[1] + 1, size=B)
    n_hist[0] = 0                                       # an empty history
    hist_offsets = np.concatenate([[0], np.cumsum(n_hist)]).astype(np.int32)
    hist = rng.integers(0, V, size=int(hist_offsets[-1])).astype(np.int32)
    if len(hist) > 8:
        hist[1::7] = hist[0]                            # repeated tokens
    return x.astype(np.float32), row_offsets, hist_offsets, hist


def _bits_equal(got, want):
    g, w = np.asarray(got, np.float32), np.asarray(want, np.float32)
    nan = np.isnan(w)
    return np.array_equal(np.isnan(g), nan) and np.array_equal(g.view(np.uint32)[~nan],
                                                                 w.view(np.uint32)[~nan])


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V,penalty", [(37, 1.3), (1031, 0.7), (151936, 1.15)])
def test_matches_oracle_bit_for_bit(zb, dtype, V, penalty):
    rng = np.random.default_rng(V)
    x, ro, ho, hist = _inputs(rng, 6, V, dtype)
    got, pad, err, _ = _case(zb, x, dtype, ro, ho, hist, penalty)
    want, bad = pen.repetition_penalty(x, ro, ho, hist, penalty,
                                       dtype="bf16" if dtype == torch.bfloat16 else "fp32")
    assert err == 0 and not bad
    assert _bits_equal(got, want)
    assert torch.isnan(pad).all()                       # nothing written past the vocabulary


def test_out_of_range_tokens_are_flagged_and_skipped(zb):
    x = np.arange(1, 9, dtype=np.float32).reshape(1, 8)
    got, _, err, _ = _case(zb, x, torch.float32, [0, 1], [0, 4], [2, 8, -1, 5], 2.0)
    want, bad = pen.repetition_penalty(x, [0, 1], [0, 4], [2, 8, -1, 5], 2.0)
    assert bad and err == 7                             # ZARYA_DEVERR_TOKEN
    assert _bits_equal(got, want)                       # tokens 2 and 5 still penalised


def test_history_range_past_the_tokens_is_refused(zb):
    x = np.ones((2, 16), dtype=np.float32)
    # sequence 1's range ends past the 3 history tokens: its row stays as it is
    got, _, err, _ = _case(zb, x, torch.float32, [0, 1, 2], [0, 1, 5], [3, 4, 5], 2.0)
    assert err == 2                                     # ZARYA_DEVERR_ROWS
    assert got[0, 3] == 0.5 and (np.delete(got[0], 3) == 1.0).all()
    assert (got[1] == 1.0).all()


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_draw_after_the_penalty_matches_the_oracle(zb, dtype):
    rng = np.random.default_rng(5)
    B, S, L, V = 3, 2, 4, 4099
    x = rng.normal(scale=2.0, size=(B * S * L, V)).astype(np.float32)
    # each row's top logit is in its sequence's history, so the penalty moves the argmax
    top = x.argmax(axis=1)
    x[np.arange(len(x)), top] = 9.0
    if dtype == torch.bfloat16:
        x = pen.bf16_round(x)
    ro = np.arange(0, B * S * L + 1, S * L, dtype=np.int32)
    hist = np.concatenate([top[b * S * L:(b + 1) * S * L] for b in range(B)]).astype(np.int32)
    ho = ro.copy()
    got, _, err, (logits, ro_dev, d) = _case(zb, x, dtype, ro, ho, hist, 4.0)
    want, _ = pen.repetition_penalty(x, ro, ho, hist, 4.0,
                                     dtype="bf16" if dtype == torch.bfloat16 else "fp32")
    assert err == 0 and _bits_equal(got, want)
    rows = B * S * L
    d.max_slots = S
    dev_i32 = lambda n, v: torch.full((n,), v, dtype=torch.int32, device="cuda")  # noqa: E731
    tok = dev_i32(rows, -7)
    prob = torch.full((rows,), -7.0, device="cuda")
    conf = torch.full((B, S), -7.0, device="cuda")
    sel = torch.zeros((B, S), dtype=torch.uint8, device="cuda")
    zb.draft_select(logits, dev_i32(B, S), dev_i32(B, L), tok, prob, conf, sel, dev_i32(B, -7),
                    dev_i32(B + 1, -7), dev_i32(rows, -7), dev_i32(rows, -7), d)
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    ref = smp.draft_select(want, [S] * B, [L] * B, temperature=0.0, slot_threshold=0.9)
    assert np.array_equal(tok.cpu().numpy(), ref["draft_tokens"])
    assert not np.array_equal(ref["draft_tokens"], top)   # the penalty moved the draws
