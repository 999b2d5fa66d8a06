"""zarya_top_p against the oracle (oracle/nucleus.py): the kept set of every
row on fp32 and bf16 rows (heavy ties in bf16), several temperatures and top_p
values, rows of no sequence, and draws taken after the truncation. The GPU
sums masses in fixed point from fp32 exponentials, so a kept set may differ
from the exact one only in one logit value whose boundary mass is within
2e-6 of top_p; every difference is checked to be such a case."""
import numpy as np
import pytest
import torch

from oracle import nucleus as nuc
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


def _run(zb, x, dtype, row_offsets, T, top_p, max_slots=1):
    rows, V = x.shape
    epv = 8 if dtype == torch.bfloat16 else 4
    stride = (V + epv - 1) // epv * epv
    buf = torch.full((rows, stride), float("nan"), dtype=dtype, device="cuda")
    buf[:, :V] = torch.as_tensor(x).to(dtype).cuda()
    logits = buf.as_strided((rows, V), (stride, 1))
    ro = _i32(row_offsets)
    d = zb.make_sample_desc(batch=len(row_offsets) - 1, vocab=V,
                            dtype=zb.BF16 if dtype == torch.bfloat16 else zb.FP32,
                            max_slots=max_slots, total_rows=rows, row_stride=stride,
                            temperature=T, slot_threshold=0.9, token_threshold=0.4, seed=7,
                            offset=1, row_offsets=ro)
    zb.top_p(logits, top_p, d)
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    return logits, ro, d


# The kernel's masses are fp32 exponentials of fp32 arguments summed in 2^-40
# fixed point: relative to the exact masses they are off by less than 1e-6 (the
# argument's rounding dominates), so the boundary value x* can come out one
# distinct value off only when the exact cumulative mass at that boundary lies
# within this margin of top_p.
BOUNDARY_MARGIN = 2e-6


def _kept_ok(x_row, gpu_kept, T, top_p):
    """The GPU's kept set (over the finite logits) equals the oracle's, or
    differs in one distinct logit value whose boundary mass (the exact mass
    of the tokens at or above it, or strictly above it) lies within
    BOUNDARY_MARGIN of top_p."""
    fin = np.isfinite(x_row)
    want = nuc.kept_mask(x_row, T, top_p)
    if np.array_equal(gpu_kept[fin], want[fin]):
        return True
    diff = np.unique(x_row[fin & (gpu_kept != want)])
    if len(diff) != 1:
        return False
    p = nuc._probs(x_row, T)
    v = diff[0]
    return min(abs(p[x_row >= v].sum() - top_p), abs(p[x_row > v].sum() - top_p)) <= BOUNDARY_MARGIN


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V", [37, 4099, 151936])
def test_kept_sets_match_the_oracle(zb, dtype, V):
    rng = np.random.default_rng(V)
    grid = [(T, p) for T in (0.0, 0.6, 1.0, 1.9) for p in (0.05, 0.5, 0.9, 0.99)]
    if V > 100000:   # the oracle walks up to the whole row in Python: a few cases suffice
        grid = [(0.0, 0.5), (1.0, 0.99), (0.6, 0.05)]
    for T, top_p in grid:
        rows = 5
        scale = float(rng.choice([0.5, 2.0, 4.0]))
        x = rng.normal(scale=scale, size=(rows, V)).astype(np.float32)
        x[0, : V // 3] = -np.inf                      # a row with tokens already cut
        if dtype == torch.bfloat16:
            x = np.where(np.isfinite(x), pen.bf16_round(np.where(np.isfinite(x), x, 0.0)), x)
        ro = [0, 2, 4]                                # row 4 belongs to no sequence
        logits, _, _ = _run(zb, x, dtype, ro, T, top_p)
        got = logits.float().cpu().numpy()
        for g in range(4):
            kept = np.isfinite(got[g])
            assert np.array_equal(got[g][kept], x[g][kept])      # kept logits unchanged
            assert (got[g][~kept] == -np.inf).all()               # the rest cut
            assert kept.any()
            assert _kept_ok(x[g].astype(np.float64), kept, T, top_p), (T, top_p, g)
        assert np.array_equal(got[4], x[4])           # a row of no sequence: untouched


@pytest.mark.parametrize("T", [0.0, 0.8])
def test_draws_after_top_p_stay_in_the_nucleus(zb, T):
    rng = np.random.default_rng(11)
    B, S, L, V = 2, 2, 4, 2053
    rows = B * S * L
    x = rng.normal(scale=2.0, size=(rows, V)).astype(np.float32)
    ro = np.arange(0, rows + 1, S * L, dtype=np.int32)
    logits, ro_dev, d = _run(zb, x, torch.float32, ro, T, 0.6, max_slots=S)
    kept_gpu = np.isfinite(logits.float().cpu().numpy())
    dev_i32 = lambda n, v: torch.full((n,), v, dtype=torch.int32, device="cuda")  # noqa: E731
    tok = dev_i32(rows, -7)
    prob = torch.full((rows,), -7.0, device="cuda")
    zb.draft_select(logits, dev_i32(B, S), dev_i32(B, L), tok, prob,
                    torch.zeros((B, S), device="cuda"),
                    torch.zeros((B, S), dtype=torch.uint8, device="cuda"), dev_i32(B, -7),
                    dev_i32(B + 1, -7), dev_i32(rows, -7), dev_i32(rows, -7), d)
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    tok, prob = tok.cpu().numpy(), prob.cpu().numpy()
    g_noise = lambda g: smp.gumbel_noise(7, 1, g, V)      # noqa: E731
    for g in range(rows):
        xg = x[g].astype(np.float64)
        assert kept_gpu[g][tok[g]]                                      # inside the nucleus
        want = nuc.draw_token(xg, T, 0.6, 7, 1, g)
        if tok[g] != want:   # only a near-tie of two kept scores may differ
            z = xg / T + g_noise(g) if T > 0 else xg
            assert abs(z[tok[g]] - z[want]) < 1e-4 * (1 + abs(z[want]))
        p_ref = nuc.row_probability(xg, int(tok[g]), T, 0.6)
        assert abs(prob[g] - p_ref) < 1e-5 + 1e-4 * p_ref


def _shaped_rows(rng, V):
    """Rows whose masses sit in one mass bin, in every bin, or at its edges."""
    flat = np.full(V, 1.25, dtype=np.float32)                        # every token equal
    plateau = np.full(V, -3.0, dtype=np.float32)                      # a plateau and a few peaks
    plateau[rng.choice(V, 7, replace=False)] = rng.uniform(2.0, 6.0, 7).astype(np.float32)
    wide = np.linspace(-90.0, 10.0, V).astype(np.float32)             # masses in every bin and below
    rng.shuffle(wide)
    single = np.full(V, -np.inf, dtype=np.float32)                    # one finite logit
    single[V // 2] = 0.5
    steps = np.repeat(np.arange(-40.0, 0.0, 2.0), V // 20 + 1)[:V].astype(np.float32)  # bin edges
    return np.stack([flat, plateau, wide, single, steps])


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("T", [0.05, 1.0, 25.0])
def test_kept_sets_at_mass_bin_extremes(zb, dtype, T):
    rng = np.random.default_rng(17)
    V = 4099
    x = _shaped_rows(rng, V)
    if dtype == torch.bfloat16:
        x = np.where(np.isfinite(x), pen.bf16_round(np.where(np.isfinite(x), x, 0.0)), x)
    for top_p in (0.3, 0.9, 0.999):
        rows = x.shape[0]
        logits, _, _ = _run(zb, x, dtype, [0, rows], T, top_p)
        got = logits.float().cpu().numpy()
        for g in range(rows):
            kept = np.isfinite(got[g])
            assert np.array_equal(got[g][kept], x[g][kept])
            assert (got[g][~kept] == -np.inf).all()
            assert kept.any()
            assert _kept_ok(x[g].astype(np.float64), kept, T, top_p), (T, top_p, g)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_kept_sets_when_a_mass_bin_outgrows_shared_memory(zb, dtype):
    """Rows whose boundary bin holds tens of thousands of distinct values (more
    than the kernel gathers in shared memory): the descent then runs over the
    row itself."""
    rng = np.random.default_rng(23)
    V = 60000
    band = rng.uniform(0.0, 0.5, V).astype(np.float32)          # one mass octave at T = 1
    mixed = rng.uniform(-1.0, 1.0, V).astype(np.float32)
    mixed[rng.choice(V, 50, replace=False)] = 3.0
    x = np.stack([band, mixed])
    if dtype == torch.bfloat16:
        x = pen.bf16_round(x)
    for T, top_p in ((1.0, 0.5), (1.0, 0.97), (3.0, 0.8)):
        logits, _, _ = _run(zb, x, dtype, [0, 2], T, top_p)
        got = logits.float().cpu().numpy()
        for g in range(2):
            kept = np.isfinite(got[g])
            assert np.array_equal(got[g][kept], x[g][kept])
            assert (got[g][~kept] == -np.inf).all()
            assert _kept_ok(x[g].astype(np.float64), kept, T, top_p), (T, top_p, g)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_signed_zeros_at_the_boundary_are_kept_together(zb, dtype):
    """x* = 0 with +0.0 and -0.0 logits both present: the kept set is
    {x >= x*}, so both zeros stay (they are equal values)."""
    V = 64
    x = np.full(V, -6.0, dtype=np.float32)
    x[:4] = 1.0
    x[4:14] = 0.0
    x[14:24] = -0.0
    rows = np.stack([x, x[::-1].copy()])
    for top_p in (0.5, 0.8):
        logits, _, _ = _run(zb, rows, dtype, [0, 2], 1.0, top_p)
        got = logits.float().cpu().numpy()
        for g in range(2):
            kept = np.isfinite(got[g])
            zeros = rows[g] == 0.0
            assert kept[zeros].all() or not kept[zeros].any(), "the zeros split"
            assert _kept_ok(rows[g].astype(np.float64), kept, 1.0, top_p), (top_p, g)


# The kernel's stage 2 counts the tokens of every key of the boundary bin and
# scans the counts when the bin spans at most this many logit values (bf16 or
# fp32), and otherwise descends over the bin's keys by digits.
HIST_KEYS = 4096


def _bin_keys(x_row, T, top_p, dtype=torch.bfloat16):
    """How many representable logit values (bf16 or fp32) the boundary mass
    bin (one octave of probability below the row maximum's, counted in whole
    octaves) spans."""
    xs = nuc.kept_threshold(x_row, T, top_p)
    m = float(np.max(x_row))
    w = float(T) * np.log(2.0)
    j = np.floor((m - xs) / w)
    lo, hi = m - (j + 1) * w, m - j * w
    if dtype == torch.bfloat16:
        allv = (np.arange(65536, dtype=np.uint32) << 16).view(np.float32)
        allv = allv[np.isfinite(allv)]
        return int(np.count_nonzero((allv > lo) & (allv <= hi)))

    def key(v):   # order-preserving key of an fp32 value
        b = int(np.array([v], dtype=np.float32).view(np.uint32)[0])
        return b ^ 0xFFFFFFFF if b & 0x80000000 else b | 0x80000000

    lo32, hi32 = np.float32(lo), np.float32(hi)
    if lo32 <= lo:   # the smallest fp32 value above lo
        lo32 = np.nextafter(lo32, np.float32(np.inf))
    if hi32 > hi:
        hi32 = np.nextafter(hi32, np.float32(-np.inf))
    return key(hi32) - key(lo32) + 1


@pytest.mark.parametrize("T", [0.3, 1.0])
def test_kept_sets_on_both_stage2_paths_with_heavy_ties(zb, T):
    """bf16 rows of the decode vocabulary whose boundary bin is narrow (the
    key counts: one key holding nearly every token and two adjacent keys
    interleaved, both overflowing the gathered segments, and a normal spread)
    or crosses zero (tens of thousands of keys: the digit descent)."""
    rng = np.random.default_rng(29)
    V = 151936
    peaks = rng.choice(V, 40, replace=False)
    one_key = np.full(V, 1.25, dtype=np.float32)
    one_key[peaks] = 4.0
    two_keys = np.where(rng.random(V) < 0.5, 1.5, 1.5078125).astype(np.float32)
    two_keys[peaks] = 4.0
    spread = rng.normal(size=V).astype(np.float32)
    near_zero = rng.uniform(-0.3, 0.3, V).astype(np.float32)
    near_zero[peaks[:5]] = 0.4
    x = pen.bf16_round(np.stack([one_key, two_keys, spread, near_zero]))
    for top_p in (0.3, 0.9, 0.999):
        logits, _, _ = _run(zb, x, torch.bfloat16, [0, 4], T, top_p)
        got = logits.float().cpu().numpy()
        for g in range(4):
            xg = x[g].astype(np.float64)
            keys = _bin_keys(xg, T, top_p)
            if g == 3 and T == 1.0 and top_p < 0.99:
                assert keys > HIST_KEYS, keys          # the digit descent
            elif g < 3:
                assert keys < HIST_KEYS // 2, keys     # the key counts
            kept = np.isfinite(got[g])
            assert np.array_equal(got[g][kept], x[g][kept])
            assert (got[g][~kept] == -np.inf).all()
            assert _kept_ok(xg, kept, T, top_p), (T, top_p, g)


def test_kept_sets_on_the_key_counts_with_fp32_logits(zb):
    """fp32 rows far from zero, where one octave of probability spans a few
    hundred fp32 values: the key counts with 32-bit keys (a spread, a plateau
    with peaks), beside a row near zero that takes the digit descent."""
    rng = np.random.default_rng(31)
    V = 20000
    spread = (20000.0 + rng.normal(scale=2.0, size=V)).astype(np.float32)
    plateau = np.full(V, 20000.0, dtype=np.float32)
    plateau[rng.choice(V, 30, replace=False)] = 20003.0
    near_zero = rng.normal(scale=0.5, size=V).astype(np.float32)
    x = np.stack([spread, plateau, near_zero])
    for T, top_p in ((1.0, 0.5), (1.0, 0.9), (0.7, 0.99)):
        logits, _, _ = _run(zb, x, torch.float32, [0, 3], T, top_p)
        got = logits.cpu().numpy()
        for g in range(3):
            xg = x[g].astype(np.float64)
            keys = _bin_keys(xg, T, top_p, torch.float32)
            if g < 2:
                assert keys < HIST_KEYS // 2, keys     # the key counts
            else:
                assert keys > HIST_KEYS, keys          # the digit descent
            kept = np.isfinite(got[g])
            assert np.array_equal(got[g][kept], x[g][kept])
            assert (got[g][~kept] == -np.inf).all()
            assert _kept_ok(xg, kept, T, top_p), (T, top_p, g)
