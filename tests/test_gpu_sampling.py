"""GPU parity of slot selection and token acceptance (Sec. 5.2 steps 3-6):
zarya_draft_select and zarya_verify_accept against the CPU oracle
(oracle/sampling.py) on the same seeded logits.

What is compared, and how:
  * draws at T = 0: bit-exact (both sides take the first maximum of the same
    values);
  * draws at T > 0: bit-exact except where the oracle's fp64 scores
    x / T + g of the two candidates lie within the kernel's fp32 rounding of
    each other; there the kernel's token must be one of those near-ties;
  * probabilities: |p_gpu - p| <= 1e-6 + 1e-4 p (fp32 sums over the
    vocabulary, fp32 exponentials of 2^-22 relative error);
  * decisions taken from probabilities (selection, acceptance): bit-exact
    when the oracle's rule is applied to the kernel's own fp32
    probabilities, and equal to the oracle's end-to-end decisions except
    where a probability lies within tolerance of a threshold or a tie;
  * layouts and lists (verify_row_offsets, verify_src_rows, verify_tokens,
    slot_accept, accept_len): bit-exact.
"""
import numpy as np
import pytest
import torch

from oracle import sampling as smp
from paper_2609_19868_gb300 import _binding as zb
from paper_2609_19868_gb300 import session
from paper_2609_19868_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

P_ATOL, P_RTOL = 1e-6, 1e-4


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2609_19868_gb300 import build

    build.build()
    zb.load()
    assert zb.check_device_error() == 0


def _host_f32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy()


def _p_close(p_gpu, p_ref):
    p_gpu = np.asarray(p_gpu, dtype=np.float64)
    p_ref = np.asarray(p_ref, dtype=np.float64)
    return np.abs(p_gpu - p_ref) <= P_ATOL + P_RTOL * np.abs(p_ref)


def _score_tol(z):
    # fp32 x * (1/T) + g with g from log1pf / __logf: a few ulp of |z| plus
    # the log's absolute error
    return 4e-5 + 2e-6 * np.abs(z)


def _check_draws(x_host, rows, tokens_gpu, T, seed, offset):
    """Tokens at ``rows`` against the oracle; returns the number of near-tie
    rows where the kernel chose another (valid) token."""
    near = 0
    for g in rows:
        x = x_host[g].astype(np.float64)
        tg = int(tokens_gpu[g])
        assert 0 <= tg < x.size, (g, tg)
        if T > 0:
            z = x / T + smp.gumbel_noise(seed, offset, g, x.size)
        else:
            z = x
        to = smp._draw_token_fast(x_host[g], T, seed, offset, g)
        if tg == to:
            continue
        if T == 0:
            raise AssertionError(f"row {g}: gpu {tg} vs oracle {to}")
        assert z[to] - z[tg] <= _score_tol(z[to]), (g, tg, to, z[to], z[tg])
        near += 1
    return near


def _run_tiny(dtype, T, seed=7, offset=3, slot_threshold=0.9):
    w = wl.make_sampling("select_tiny", dtype=dtype)
    sb = session.upload_sampling(w, "cuda", temperature=T, seed=seed, offset=offset,
                                 slot_threshold=slot_threshold)
    sb.draft()
    sb.verify()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    return w, sb


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("T", [0.0, 0.7, 1.0, 1.8])
def test_draft_select_matches_oracle(dtype, T):
    w, sb = _run_tiny(dtype, T)
    x = _host_f32(w.draft_logits)
    ref = smp.draft_select(x, w.n_slots, w.slot_len, temperature=T, slot_threshold=0.9, seed=7,
                           offset=3, max_slots=w.max_slots)
    tok = sb.draft_tokens.cpu().numpy()
    prob = sb.draft_prob.cpu().numpy()
    near = _check_draws(x, range(w.rows), tok, T, 7, 3)
    assert near <= max(1, w.rows // 50)
    same = tok == ref["draft_tokens"]
    # probabilities of the same tokens: oracle's fp64 value
    assert _p_close(prob[same], ref["draft_prob"][same]).all()
    for g in np.nonzero(~same)[0]:
        assert _p_close(prob[g], smp.row_probability(x[g], int(tok[g]), T))
    # slot confidences are the first rows' probabilities, exactly
    conf = sb.slot_conf.cpu().numpy()
    sel = sb.slot_selected.cpu().numpy()
    nsel = sb.n_selected.cpu().numpy()
    for b in range(w.B):
        S, L, o = int(w.n_slots[b]), int(w.slot_len[b]), int(w.row_offsets[b])
        c = prob[o + np.arange(S) * L]
        assert np.array_equal(conf[b, :S], c)
        assert (conf[b, S:] == 0).all() and (sel[b, S:] == 0).all()
        rule = smp.select_slots(c.astype(np.float64), np.float32(0.9))
        assert np.array_equal(sel[b, :S].astype(bool), rule)
        assert nsel[b] == rule.sum()
        # end to end: equal unless a confidence sits at the threshold / a tie
        near_thr = np.abs(ref["slot_conf"][b, :S] - 0.9) <= P_ATOL + P_RTOL
        if not near_thr.any() and same[o + np.arange(S) * L].all():
            assert np.array_equal(sel[b, :S], ref["slot_selected"][b, :S])
    _check_layout(w, sb)


def _check_layout(w, sb):
    """verify_row_offsets / src rows / tokens follow from the kernel's own
    selection by the oracle's rule (slot order, dense packing)."""
    sel = sb.slot_selected.cpu().numpy()
    nsel = sb.n_selected.cpu().numpy()
    tok = sb.draft_tokens.cpu().numpy()
    voffs = sb.verify_row_offsets.cpu().numpy()
    src = sb.verify_src_rows.cpu().numpy()
    vtok = sb.verify_tokens.cpu().numpy()
    expect_offs = np.concatenate([[0], np.cumsum(nsel.astype(np.int64) * w.slot_len)])
    assert np.array_equal(voffs, expect_offs)
    expect_src = []
    for b in range(w.B):
        S, L, o = int(w.n_slots[b]), int(w.slot_len[b]), int(w.row_offsets[b])
        for s in range(S):
            if sel[b, s]:
                expect_src += list(range(o + s * L, o + s * L + L))
    n = len(expect_src)
    assert np.array_equal(src[:n], expect_src)
    assert (src[n:] == -1).all()
    assert np.array_equal(vtok[:n], tok[expect_src])
    assert (vtok[n:] == -1).all()


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("T", [0.0, 1.0, 0.6])
def test_verify_accept_matches_oracle(dtype, T):
    w, sb = _run_tiny(dtype, T)
    x = _host_f32(w.verify_logits)
    ref = smp.verify_accept(x, w.verify_tokens, w.n_verify, w.slot_len, temperature=T,
                            token_threshold=0.4, max_slots=w.max_slots)
    n = w.verify_rows
    prob = sb.token_prob.cpu().numpy()
    assert _p_close(prob[:n], ref["token_prob"][:n]).all()
    assert np.isnan(prob[n:]).all()          # rows past the layout are not written
    sa = sb.slot_accept.cpu().numpy()
    acc = sb.accept_len.cpu().numpy()
    for b in range(w.B):
        k, L, o = int(w.n_verify[b]), int(w.slot_len[b]), int(w.verify_offsets[b])
        rule_sa, rule_acc = smp.accept_prefix(prob[o:o + k * L].astype(np.float64), k, L,
                                              np.float32(0.4))
        assert np.array_equal(sa[b, :k], rule_sa)
        assert (sa[b, k:] == 0).all()
        assert acc[b] == rule_acc
        if not (np.abs(ref["token_prob"][o:o + k * L] - 0.4) <= P_ATOL + P_RTOL).any():
            assert np.array_equal(sa[b], ref["slot_accept"][b])
            assert acc[b] == ref["accept_len"][b]


def test_chained_step_matches_oracle():
    """draft -> verification layout -> acceptance on the draft's own outputs
    (verification logits taken from the workload's rows)."""
    w = wl.make_sampling("select_tiny", dtype="bf16")
    sb = session.upload_sampling(w, "cuda", temperature=0.0, slot_threshold=0.5, chain=True)
    sb.draft()
    sb.verify()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    d = smp.draft_select(_host_f32(w.draft_logits), w.n_slots, w.slot_len, temperature=0.0,
                         slot_threshold=0.5, max_slots=w.max_slots)
    nsel = sb.n_selected.cpu().numpy()
    if not np.array_equal(nsel, d["n_selected"]):
        pytest.skip("a confidence at the threshold decided differently (checked elsewhere)")
    assert np.array_equal(sb.verify_row_offsets.cpu().numpy(), d["verify_row_offsets"])
    assert np.array_equal(sb.verify_tokens.cpu().numpy(), d["verify_tokens"])
    vx = _host_f32(sb.verify_logits)
    v = smp.verify_accept(vx, d["verify_tokens"], d["n_selected"], w.slot_len, temperature=0.0,
                          token_threshold=0.4, row_offsets=d["verify_row_offsets"],
                          max_slots=w.max_slots)
    nv = int(d["verify_row_offsets"][-1])
    assert _p_close(sb.token_prob.cpu().numpy()[:nv], v["token_prob"][:nv]).all()


def _direct(x, n_slots, slot_len, T=0.0, row_stride=None, slot_threshold=0.9, seed=0, offset=0,
            dtype=torch.float32):
    """Run zarya_draft_select on a hand-built [rows, V] block."""
    x = torch.as_tensor(x, dtype=torch.float32)
    rows, V = x.shape
    epv = 8 if dtype == torch.bfloat16 else 4    # rows padded to 16 bytes by default
    stride = row_stride or (V + epv - 1) // epv * epv
    buf = torch.full((rows, stride), float("nan"), dtype=dtype, device="cuda")
    buf[:, :V] = x.to(dtype).cuda()
    logits = buf[:, :V] if stride == V else buf.as_strided((rows, V), (stride, 1))
    n_slots = np.asarray(n_slots)
    slot_len = np.asarray(slot_len)
    offs = np.concatenate([[0], np.cumsum(n_slots * slot_len)]).astype(np.int32)
    B, ms = len(n_slots), int(n_slots.max())
    dev = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int32)).cuda()  # noqa: E731
    ro = dev(offs)
    d = zb.make_sample_desc(batch=B, vocab=V, dtype=zb.BF16 if dtype == torch.bfloat16 else
                            zb.FP32, max_slots=ms, total_rows=rows, row_stride=stride,
                            temperature=T, slot_threshold=slot_threshold, token_threshold=0.4,
                            seed=seed, offset=offset, row_offsets=ro)
    out = dict(draft_tokens=torch.full((rows,), -7, dtype=torch.int32, device="cuda"),
               draft_prob=torch.full((rows,), -7.0, device="cuda"),
               slot_conf=torch.full((B, ms), -7.0, device="cuda"),
               slot_selected=torch.full((B, ms), 7, dtype=torch.uint8, device="cuda"),
               n_selected=torch.full((B,), -7, dtype=torch.int32, device="cuda"),
               verify_row_offsets=torch.full((B + 1,), -7, dtype=torch.int32, device="cuda"),
               verify_src_rows=torch.full((rows,), -7, dtype=torch.int32, device="cuda"),
               verify_tokens=torch.full((rows,), -7, dtype=torch.int32, device="cuda"))
    zb.draft_select(logits, dev(n_slots), dev(slot_len), out["draft_tokens"], out["draft_prob"],
                    out["slot_conf"], out["slot_selected"], out["n_selected"],
                    out["verify_row_offsets"], out["verify_src_rows"], out["verify_tokens"], d)
    torch.cuda.synchronize()
    err = zb.check_device_error()
    return {k: v.cpu().numpy() for k, v in out.items()}, err, (logits, ro, d)


@pytest.mark.parametrize("V", [1, 3, 7, 8, 9, 1031, 16384, 16391])
@pytest.mark.parametrize("T", [0.0, 1.0])
def test_vocabulary_sizes_and_ragged_tails(V, T):
    rng = np.random.default_rng(V)
    x = rng.standard_normal((6, V)).astype(np.float32) * 3
    out, err, _ = _direct(x, [2], [3], T=T, seed=11, offset=1)
    assert err == 0
    _check_draws(x, range(6), out["draft_tokens"], T, 11, 1)
    for g in range(6):
        assert _p_close(out["draft_prob"][g],
                        smp.row_probability(x[g], int(out["draft_tokens"][g]), T))


def test_padded_row_stride_is_not_read():
    rng = np.random.default_rng(1)
    V = 1003
    x = rng.standard_normal((4, V)).astype(np.float32)
    out, err, _ = _direct(x, [1, 1], [2, 2], row_stride=1008)    # NaN in the padding
    assert err == 0
    ref = smp.draft_select(x, [1, 1], [2, 2], temperature=0.0, slot_threshold=0.9)
    assert np.array_equal(out["draft_tokens"], ref["draft_tokens"])
    assert _p_close(out["draft_prob"], ref["draft_prob"]).all()


def test_ties_go_to_the_first_index():
    V = 5000
    x = np.zeros((4, V), dtype=np.float32)
    x[1, [4999, 17, 3000]] = 2.0                 # three equal maxima
    x[2, :] = -1.0
    x[2, 4096:] = 0.5                            # first maximum at a vector boundary
    x[3, 4999] = 1.0                             # the maximum in the last element
    out, err, _ = _direct(x, [1, 1], [2, 2])
    assert err == 0
    assert out["draft_tokens"].tolist() == [0, 17, 4096, 4999]
    assert abs(out["draft_prob"][0] - 1 / V) < 1e-9
    for dt in (torch.bfloat16,):
        out2, _, _ = _direct(x, [1, 1], [2, 2], dtype=dt)
        assert out2["draft_tokens"].tolist() == [0, 17, 4096, 4999]


def test_infinite_logits():
    V = 300
    x = np.zeros((3, V), dtype=np.float32)
    x[0, :] = -np.inf
    x[0, 123] = 1.0                               # masked vocabulary, one live token
    x[1, ::2] = -np.inf
    out, err, _ = _direct(x, [3], [1])
    assert err == 0
    assert out["draft_tokens"][0] == 123 and out["draft_prob"][0] == 1.0
    assert out["draft_tokens"][1] == 1
    assert _p_close(out["draft_prob"][1], 1 / 150)
    out, err, _ = _direct(x, [3], [1], T=0.5, seed=3)
    assert err == 0 and out["draft_tokens"][0] == 123
    assert x[1, out["draft_tokens"][1]] == 0.0   # never a masked token


def test_selection_fallback_and_strict_threshold():
    # 3 slots of 1 token each per sequence, V = 40: p = e^a / (e^a + 39)
    V = 40
    heights = {0: [1.0, 3.0, 3.0], 1: [6.0, 1.0, 8.0]}
    x = np.zeros((6, V), dtype=np.float32)
    for b, hs in heights.items():
        for s, a in enumerate(hs):
            x[b * 3 + s, 5 + s] = a
    out, err, _ = _direct(x, [3, 3], [1, 1], slot_threshold=0.9)
    assert err == 0
    # b0: all below 0.9 -> most confident, first of the tie at 3.0 (slot 1)
    # b1: p(6) = .912 and p(8) = .987 above 0.9 -> slots 0 and 2
    assert out["slot_selected"].tolist() == [[0, 1, 0], [1, 0, 1]]
    assert out["n_selected"].tolist() == [1, 2]
    assert out["verify_row_offsets"].tolist() == [0, 1, 3]
    assert out["verify_src_rows"].tolist() == [1, 3, 5, -1, -1, -1]
    assert out["verify_tokens"].tolist() == [6, 5, 7, -1, -1, -1]
    # a threshold equal to a confidence does not select it (strict)
    p = out["draft_prob"][3]
    out2, _, _ = _direct(x, [3, 3], [1, 1], slot_threshold=float(p))
    assert out2["slot_selected"][1].tolist() == [0, 0, 1]


def test_inconsistent_layout_sets_error_and_skips():
    x = np.zeros((6, 64), dtype=np.float32)
    logits = torch.as_tensor(x).cuda()
    B = 2
    dev = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int32)).cuda()  # noqa: E731
    ro = dev([0, 2, 6])                          # sequence 0 claims 2 rows but has 1 x 3
    d = zb.make_sample_desc(batch=B, vocab=64, dtype=zb.FP32, max_slots=2, total_rows=6,
                            row_stride=64, temperature=0.0, slot_threshold=0.9,
                            token_threshold=0.4, seed=0, offset=0, row_offsets=ro)
    o = [torch.zeros(6, dtype=torch.int32, device="cuda"), torch.zeros(6, device="cuda"),
         torch.zeros((B, 2), device="cuda"), torch.zeros((B, 2), dtype=torch.uint8, device="cuda"),
         torch.full((B,), -1, dtype=torch.int32, device="cuda"),
         torch.zeros(B + 1, dtype=torch.int32, device="cuda"),
         torch.zeros(6, dtype=torch.int32, device="cuda"),
         torch.zeros(6, dtype=torch.int32, device="cuda")]
    zb.draft_select(logits, dev([1, 2]), dev([3, 2]), *o, d)
    assert zb.check_device_error() == 2          # ZARYA_DEVERR_ROWS
    assert o[4].cpu().tolist() == [0, 1]
    assert o[5].cpu().tolist() == [0, 0, 2]


def test_verify_rejects_out_of_range_token_and_empty_blocks():
    V = 52
    x = torch.zeros((4, V), device="cuda")
    dev = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int32)).cuda()  # noqa: E731
    ro = dev([0, 0, 4])                          # sequence 0 verifies nothing
    d = zb.make_sample_desc(batch=2, vocab=V, dtype=zb.FP32, max_slots=2, total_rows=4,
                            row_stride=V, temperature=0.0, slot_threshold=0.9,
                            token_threshold=0.01, seed=0, offset=0, row_offsets=ro)
    prob = torch.full((4,), -1.0, device="cuda")
    sa = torch.full((2, 2), -1, dtype=torch.int32, device="cuda")
    acc = torch.full((2,), -1, dtype=torch.int32, device="cuda")
    zb.verify_accept(x, dev([3, 4, V, 6]), dev([0, 2]), dev([5, 2]), prob, sa, acc, d)
    assert zb.check_device_error() == 7          # ZARYA_DEVERR_TOKEN
    p = prob.cpu().numpy()
    assert abs(p[0] - 1 / V) < 1e-7 and p[2] == 0.0
    assert acc.cpu().tolist() == [0, 2]
    assert sa.cpu().tolist() == [[0, 0], [2, 0]]


def test_gumbel_draws_follow_softmax_law():
    """Independent of the oracle: frequencies of kernel draws over many rows
    of the same logits match softmax(x / T)."""
    scipy_stats = pytest.importorskip("scipy.stats")
    V, rows, T = 6, 4096, 0.8
    base = np.array([0.0, 1.0, -0.5, 2.0, 0.3, 1.5], dtype=np.float32)
    x = np.tile(base, (rows, 1))
    counts = np.zeros(V)
    n = 0
    for off in range(3):
        out, err, _ = _direct(x, [rows], [1], T=T, slot_threshold=2.0, seed=5, offset=off)
        assert err == 0
        counts += np.bincount(out["draft_tokens"], minlength=V)
        n += rows
    e = np.exp(base.astype(np.float64) / T)
    p = e / e.sum()
    assert scipy_stats.chisquare(counts, n * p).pvalue > 1e-4


@pytest.mark.parametrize("name", ["select_decode_small", "select_serving_mix"])
@pytest.mark.parametrize("T", [0.0, 1.0])
def test_full_size_sampled_rows(name, T):
    """Full-size workloads: sampled rows against the oracle; every row and
    sequence against properties that hold at any size."""
    w = wl.make_sampling(name, device="cuda")
    sb = session.upload_sampling(w, "cuda", temperature=T, seed=123, offset=9)
    sb.draft()
    sb.verify()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    tok = sb.draft_tokens.cpu().numpy()
    prob = sb.draft_prob.cpu().numpy()
    assert ((tok >= 0) & (tok < w.V)).all()
    assert ((prob > 0) & (prob <= 1.0 + 1e-6)).all()
    rng = np.random.default_rng(0)
    sample = np.unique(np.concatenate([[0, w.rows - 1], rng.integers(0, w.rows, size=10)]))
    x_s = {int(g): w.draft_logits[int(g)].float().cpu().numpy() for g in sample}
    near = 0
    for g, x in x_s.items():
        to = smp._draw_token_fast(x, T, 123, 9, g)
        if tok[g] != to:
            assert T > 0
            z = x.astype(np.float64) / T + smp.gumbel_noise(123, 9, g, x.size)
            assert z[to] - z[tok[g]] <= _score_tol(z[to])
            near += 1
        assert _p_close(prob[g], smp.row_probability(x, int(tok[g]), T))
    assert near <= 1
    if T == 0:
        # every row: the token holds the row maximum and no earlier index does
        xd = w.draft_logits.float()
        mx = xd.max(dim=1).values
        t = sb.draft_tokens.long()
        assert torch.equal(xd.gather(1, t[:, None])[:, 0], mx)
        idx = torch.arange(w.V, device="cuda")[None, :]
        assert not ((xd == mx[:, None]) & (idx < t[:, None])).any()
    _check_layout(w, sb)
    sel = sb.slot_selected.cpu().numpy()
    conf = sb.slot_conf.cpu().numpy()
    for b in range(w.B):
        S = int(w.n_slots[b])
        assert np.array_equal(sel[b, :S].astype(bool),
                              smp.select_slots(conf[b, :S].astype(np.float64), np.float32(0.9)))
    # verification: sampled rows and the rule on every sequence
    vp = sb.token_prob.cpu().numpy()
    vs = np.unique(np.concatenate([[0, w.verify_rows - 1],
                                   rng.integers(0, w.verify_rows, size=8)]))
    for g in vs:
        x = w.verify_logits[int(g)].float().cpu().numpy()
        assert _p_close(vp[g], smp.row_probability(x, int(w.verify_tokens[g]), T))
    acc = sb.accept_len.cpu().numpy()
    for b in range(w.B):
        k, L, o = int(w.n_verify[b]), int(w.slot_len[b]), int(w.verify_offsets[b])
        _, a = smp.accept_prefix(vp[o:o + k * L].astype(np.float64), k, L, np.float32(0.4))
        assert acc[b] == a


def test_calls_capture_into_a_cuda_graph():
    w = wl.make_sampling("select_tiny", dtype="bf16")
    sb = session.upload_sampling(w, "cuda", temperature=1.0, seed=1, offset=2, chain=True)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        sb.draft(s)
        sb.verify(s)
    torch.cuda.synchronize()
    first = (sb.draft_tokens.clone(), sb.accept_len.clone(), sb.token_prob.clone())
    sb.draft_tokens.fill_(-1)
    sb.accept_len.fill_(-1)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        sb.draft(s)
        sb.verify(s)
    g.replay()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert torch.equal(sb.draft_tokens, first[0])
    assert torch.equal(sb.accept_len, first[1])
    assert torch.equal(torch.nan_to_num(sb.token_prob, nan=-1.0),
                       torch.nan_to_num(first[2], nan=-1.0))


@pytest.mark.parametrize("T", [0.0, 0.8])
@pytest.mark.parametrize("rows", [8, 24])
def test_few_full_vocabulary_rows_split_over_a_cluster(T, rows):
    """Few rows of the full vocabulary: every row is split over a cluster of
    CTAs (8 for 8 rows) whose partial maxima, sums and draws merge through
    distributed shared memory; each row against the oracle."""
    V = wl.QWEN3_VOCAB
    rng = np.random.default_rng(rows)
    x = (rng.standard_normal((rows, V)) * 2).astype(np.float32)
    for r in range(0, rows, 3):
        x[r, rng.integers(0, V)] += 15.0
    xb = torch.as_tensor(x).to(torch.bfloat16)
    out, err, _ = _direct(xb.float().numpy(), [rows], [1], T=T, seed=21, offset=4,
                          dtype=torch.bfloat16)
    assert err == 0
    xh = xb.float().numpy()
    near = _check_draws(xh, range(rows), out["draft_tokens"], T, 21, 4)
    assert near <= 1
    for g in range(rows):
        assert _p_close(out["draft_prob"][g],
                        smp.row_probability(xh[g], int(out["draft_tokens"][g]), T))
