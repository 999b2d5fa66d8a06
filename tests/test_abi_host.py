"""CPU checks of the C ABI: the library loads, exports every function that
include/zarya.h declares, and rejects invalid calls on the host (before any
CUDA call, so no GPU is needed)."""
import ctypes

import pytest

from paper_2609_19868_gb300 import _binding as zb


@pytest.fixture(scope="module")
def lib():
    from paper_2609_19868_gb300 import build

    build.build()
    return zb.load()


def _desc(**kw):
    d = zb.AttnDesc()
    base = dict(batch=2, n_q_heads=16, n_kv_heads=8, head_dim=128, dtype=zb.BF16, page_size=0,
                cache_capacity=256, n_pages=0, max_rows=32, total_rows=64, max_kv_len=0,
                kv_splits=0, scale=0.0, q_row_offsets=0x100000)
    base.update(kw)
    for k, v in base.items():
        setattr(d, k, v)
    return d


FAKE = 0x7F0000000000  # never dereferenced: validation fails before any access


def _attn(lib, d, q=FAKE, k=FAKE, v=FAKE, out=FAKE, page_table=None, ws=None, ws_bytes=0):
    vp = ctypes.c_void_p
    return lib.zarya_slot_attn(vp(q), vp(k), vp(v), vp(FAKE), vp(page_table), vp(FAKE), vp(FAKE),
                               vp(FAKE), vp(out), vp(ws), ws_bytes,
                               None if d is None else ctypes.byref(d), None)


def test_exports_every_declared_function(lib):
    names = zb.header_functions()
    assert {"zarya_slot_attn", "zarya_kv_append", "zarya_slot_attn_workspace_size",
            "zarya_check_device_error", "zarya_status_string", "zarya_version"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings_and_version(lib):
    assert zb.status_string(0) == "ok"
    assert zb.status_string(2) == "unsupported configuration"
    assert zb.status_string(99) == "unknown status"
    assert zb.version() >= 100


def test_desc_struct_layout_matches_c():
    # 12 int32 + float, a pointer aligned to 8, then the wait limit and the debug flags
    assert ctypes.sizeof(zb.AttnDesc) == 72
    assert zb.AttnDesc.q_row_offsets.offset == 56
    assert zb.AttnDesc.wait_limit_us.offset == 64
    assert zb.AttnDesc.debug_flags.offset == 68


@pytest.mark.parametrize("bad,status", [
    (dict(batch=0), 1),
    (dict(wait_limit_us=-1), 1),
    (dict(debug_flags=2), 1),
    (dict(n_q_heads=12, n_kv_heads=8), 1),
    (dict(dtype=7), 1),
    (dict(max_rows=0), 1),
    (dict(total_rows=0), 1),
    (dict(cache_capacity=0), 1),
    (dict(page_size=16, cache_capacity=250, n_pages=10), 1),
    (dict(page_size=16, cache_capacity=256, n_pages=0), 1),
    (dict(scale=-1.0), 1),
    (dict(scale=float("nan")), 1),
    (dict(q_row_offsets=0), 1),
    (dict(kv_splits=-2), 1),
    (dict(head_dim=64), 2),                       # bf16 tensor-core path is D = 128
    (dict(n_q_heads=24, n_kv_heads=8), 2),        # group of 3 does not divide 128 rows
    (dict(page_size=8, cache_capacity=256, n_pages=40), 2),
    (dict(dtype=zb.FP32, head_dim=48), 2),
])
def test_attention_rejects_invalid_descriptors(lib, bad, status):
    assert _attn(lib, _desc(**bad)) == status


def test_attention_rejects_null_and_misaligned_pointers(lib):
    assert _attn(lib, None) == 1
    assert _attn(lib, _desc(), q=None) == 1
    assert _attn(lib, _desc(), out=FAKE + 8) == 1
    assert _attn(lib, _desc(), k=FAKE + 2) == 1
    # page table given for a contiguous cache, or missing for a paged one
    assert _attn(lib, _desc(), page_table=FAKE) == 1
    assert _attn(lib, _desc(page_size=16, n_pages=64), page_table=None) == 1


def test_workspace_size_is_zero_for_invalid_or_fp32(lib):
    assert lib.zarya_slot_attn_workspace_size(None) == 0
    assert lib.zarya_slot_attn_workspace_size(ctypes.byref(_desc(batch=0))) == 0
    assert lib.zarya_slot_attn_workspace_size(ctypes.byref(_desc(dtype=zb.FP32, head_dim=64))) == 0


def test_workspace_size_for_forced_splits(lib):
    # 2 sequences x 8 KV heads x 1 M-tile, 10 splits (more than a cluster
    # holds, so they merge through the workspace): partial O + lse + counters
    d = _desc(kv_splits=10, cache_capacity=2048)
    n = 2 * 8 * 1 * 10 * 128
    expect = n * 128 * 4
    expect = (expect + 255) // 256 * 256 + n * 4
    expect = (expect + 255) // 256 * 256 + 16 * 4
    expect = (expect + 255) // 256 * 256
    assert lib.zarya_slot_attn_workspace_size(ctypes.byref(d)) == expect
    # up to 3 splits merge inside a thread-block cluster and need no workspace
    for s in (1, 2, 3):
        d = _desc(kv_splits=s, cache_capacity=2048)
        assert lib.zarya_slot_attn_workspace_size(ctypes.byref(d)) == 0


def test_attention_requires_large_enough_workspace(lib):
    d = _desc(kv_splits=10, cache_capacity=2048)
    need = lib.zarya_slot_attn_workspace_size(ctypes.byref(d))
    assert need > 0
    # validation of the workspace happens after device selection, which needs
    # a GPU; on a CPU-only host the call must still fail cleanly (no crash)
    st = _attn(lib, d, ws=None, ws_bytes=0)
    assert st in (1, 3)


def test_append_rejects_invalid_calls(lib):
    vp = ctypes.c_void_p
    d = _desc()

    def app(flags=1, k_new=FAKE, desc=d, page_table=None, accept=FAKE):
        return lib.zarya_kv_append(vp(k_new), vp(FAKE), vp(accept), vp(FAKE), vp(FAKE), vp(FAKE),
                                   vp(page_table), flags,
                                   None if desc is None else ctypes.byref(desc), None)

    assert app(flags=2) == 1
    assert app(flags=-1) == 1
    assert app(desc=None) == 1
    assert app(k_new=None) == 1
    assert app(accept=None) == 1
    assert app(k_new=FAKE + 4) == 1
    assert app(page_table=FAKE) == 1
    assert app(desc=_desc(n_kv_heads=1, n_q_heads=1, head_dim=4)) == 2  # row not 16-byte multiple


def test_commit_to_rejects_invalid_calls(lib):
    vp = ctypes.c_void_p
    d = _desc()

    def app(new_lens=FAKE, cache_lens=FAKE, desc=d, k_cache=FAKE):
        return lib.zarya_kv_append_commit_to(vp(FAKE), vp(FAKE), vp(FAKE), vp(k_cache), vp(FAKE),
                                             vp(cache_lens), vp(new_lens), vp(None),
                                             None if desc is None else ctypes.byref(desc), None)

    assert app(new_lens=None) == 1
    assert app(cache_lens=None) == 1
    assert app(desc=None) == 1
    assert app(k_cache=FAKE + 8) == 1


def test_commit_staged_rejects_invalid_calls(lib):
    vp = ctypes.c_void_p
    d = _desc()
    assert lib.zarya_kv_commit_staged(vp(None), vp(FAKE), vp(FAKE), ctypes.byref(d), None) == 1
    assert lib.zarya_kv_commit_staged(vp(FAKE), vp(None), vp(FAKE), ctypes.byref(d), None) == 1
    assert lib.zarya_kv_commit_staged(vp(FAKE), vp(FAKE), vp(None), ctypes.byref(d), None) == 1
    assert lib.zarya_kv_commit_staged(vp(FAKE), vp(FAKE), vp(FAKE), None, None) == 1
    assert lib.zarya_kv_commit_staged(vp(FAKE), vp(FAKE), vp(FAKE),
                                      ctypes.byref(_desc(batch=0)), None) == 1


def test_staged_rejects_missing_block_kv(lib):
    vp = ctypes.c_void_p
    d = _desc()
    st = lib.zarya_slot_attn_staged(vp(FAKE), vp(None), vp(FAKE), vp(FAKE), vp(FAKE), vp(FAKE),
                                    vp(None), vp(FAKE), vp(FAKE), vp(FAKE), vp(FAKE), vp(None), 0,
                                    ctypes.byref(d), None)
    assert st == 1
    st = lib.zarya_slot_attn_staged(vp(FAKE), vp(FAKE), vp(FAKE + 8), vp(FAKE), vp(FAKE), vp(FAKE),
                                    vp(None), vp(FAKE), vp(FAKE), vp(FAKE), vp(FAKE), vp(None), 0,
                                    ctypes.byref(d), None)
    assert st == 1


def _sdesc(**kw):
    d = zb.SampleDesc()
    base = dict(batch=2, vocab=1000, dtype=zb.BF16, max_slots=4, total_rows=16, reserved=0,
                row_stride=1000, temperature=0.0, slot_threshold=0.9, token_threshold=0.4,
                reserved2=0, seed=1, offset=0, row_offsets=0x100000)
    base.update(kw)
    for k, v in base.items():
        setattr(d, k, v)
    return d


def test_sample_desc_layout_matches_c():
    assert ctypes.sizeof(zb.SampleDesc) == 72
    assert zb.SampleDesc.row_stride.offset == 24
    assert zb.SampleDesc.seed.offset == 48
    assert zb.SampleDesc.row_offsets.offset == 64


def _draft(lib, d, logits=FAKE, out=FAKE):
    vp = ctypes.c_void_p
    return lib.zarya_draft_select(vp(logits), vp(FAKE), vp(FAKE), vp(out), vp(FAKE), vp(FAKE),
                                  vp(FAKE), vp(FAKE), vp(FAKE), vp(FAKE), vp(FAKE),
                                  None if d is None else ctypes.byref(d), None)


def _verify(lib, d, logits=FAKE, tokens=FAKE):
    vp = ctypes.c_void_p
    return lib.zarya_verify_accept(vp(logits), vp(tokens), vp(FAKE), vp(FAKE), vp(FAKE), vp(FAKE),
                                   vp(FAKE), None if d is None else ctypes.byref(d), None)


@pytest.mark.parametrize("bad", [
    dict(batch=0), dict(vocab=0), dict(max_slots=0), dict(total_rows=0), dict(dtype=5),
    dict(reserved=1), dict(reserved2=3),
    dict(row_stride=999),                         # shorter than the vocabulary
    dict(row_stride=1001),                        # bf16 rows not a multiple of 16 bytes
    dict(dtype=zb.FP32, row_stride=1002),
    dict(temperature=-0.5), dict(temperature=float("inf")), dict(temperature=float("nan")),
    dict(slot_threshold=float("nan")), dict(token_threshold=float("nan")),
    dict(row_offsets=0),
])
def test_sampling_rejects_invalid_descriptors(lib, bad):
    assert _draft(lib, _sdesc(**bad)) == 1
    assert _verify(lib, _sdesc(**bad)) == 1


def test_sampling_rejects_null_and_misaligned_pointers(lib):
    assert _draft(lib, None) == 1
    assert _verify(lib, None) == 1
    assert _draft(lib, _sdesc(), logits=None) == 1
    assert _draft(lib, _sdesc(), out=None) == 1
    assert _draft(lib, _sdesc(), logits=FAKE + 8) == 1
    assert _verify(lib, _sdesc(), tokens=None) == 1
    assert _verify(lib, _sdesc(), logits=FAKE + 4) == 1
    assert _draft(lib, _sdesc(batch=65536, max_slots=65536)) == 2


def test_reorder_restore_reject_invalid_calls(lib):
    vp = ctypes.c_void_p

    def reo(tokens=FAKE, out=FAKE + 64, batch=2, max_len=8, mask=FAKE):
        return lib.zarya_reorder(vp(tokens), vp(mask), vp(None), vp(FAKE), batch, max_len,
                                 vp(FAKE), vp(out), vp(FAKE), None)

    assert reo(tokens=None) == 1
    assert reo(mask=None) == 1
    assert reo(out=None) == 1
    assert reo(out=FAKE) == 1            # in place is refused
    assert reo(batch=0) == 1
    assert reo(max_len=0) == 1
    assert lib.zarya_restore(vp(FAKE), vp(None), vp(FAKE), 2, 8, vp(FAKE + 64), None) == 1
    assert lib.zarya_restore(vp(FAKE), vp(FAKE), vp(FAKE), 2, 8, vp(FAKE), None) == 1
    assert lib.zarya_restore(vp(FAKE), vp(FAKE), vp(FAKE), 0, 8, vp(FAKE + 64), None) == 1


def test_mode_a_budget_and_sample_rows_reject_invalid_calls(lib):
    vp = ctypes.c_void_p

    def bud(n=FAKE, batch=2, T=4, a0=0.25, max_steps=8, counts=FAKE, steps=FAKE):
        return lib.zarya_mode_a_budget(vp(n), batch, T, a0, 1, 0, max_steps, vp(counts),
                                       vp(steps), None)

    assert bud(n=None) == 1
    assert bud(counts=None) == 1
    assert bud(steps=None) == 1
    assert bud(batch=0) == 1
    assert bud(max_steps=0) == 1
    assert bud(T=-1) == 1
    assert bud(a0=1.5) == 1
    assert bud(a0=float("nan")) == 1
    assert lib.zarya_sample_rows(vp(None), vp(FAKE), vp(FAKE), ctypes.byref(_sdesc()), None) == 1
    assert lib.zarya_sample_rows(vp(FAKE), vp(None), vp(FAKE), ctypes.byref(_sdesc()), None) == 1
    assert lib.zarya_sample_rows(vp(FAKE), vp(FAKE), vp(FAKE), None, None) == 1


def test_copy_rejects_invalid_calls_before_any_cuda_call(lib):
    vp = ctypes.c_void_p
    assert lib.zarya_copy(vp(None), vp(FAKE), 64, None) == 1
    assert lib.zarya_copy(vp(FAKE), vp(None), 64, None) == 1
    assert lib.zarya_copy(vp(FAKE + 8), vp(FAKE + 4096), 64, None) == 1    # unaligned source
    assert lib.zarya_copy(vp(FAKE), vp(FAKE + 4100), 64, None) == 1        # unaligned destination
    assert lib.zarya_copy(vp(FAKE), vp(FAKE + 4096), 0, None) == 0         # nothing to move


def test_copy_binding_checks_tensors():
    import torch

    a = torch.zeros(16, dtype=torch.uint8)
    with pytest.raises(TypeError):
        zb.copy(a, a.clone())       # neither pinned nor on a device


def test_repetition_penalty_rejects_invalid_calls(lib):
    vp = ctypes.c_void_p

    def call(logits=FAKE, offs=FAKE + 64, toks=FAKE + 128, n=4, p=1.2, d="ok"):
        desc = _sdesc() if d == "ok" else d
        return lib.zarya_repetition_penalty(vp(logits), vp(offs), vp(toks), n, p,
                                            None if desc is None else ctypes.byref(desc), None)

    assert call(logits=None) == 1
    assert call(logits=FAKE + 8) == 1           # unaligned logits
    assert call(offs=None) == 1
    assert call(toks=None) == 1                 # tokens promised but missing
    assert call(n=-1) == 1
    for p in (0.0, -1.0, float("nan"), float("inf")):
        assert call(p=p) == 1
    assert call(d=None) == 1
    assert call(d=_sdesc(vocab=0)) == 1
    assert call(d=_sdesc(vocab=2_000_000, row_stride=2_000_000)) == 2   # bitmap too large
    # rows closer together than the vocabulary would overlap (and be penalised twice)
    assert call(d=_sdesc(vocab=1000, row_stride=992)) == 1


def test_top_p_rejects_invalid_calls(lib):
    vp = ctypes.c_void_p
    d = _sdesc()
    assert lib.zarya_top_p(vp(None), 0.9, ctypes.byref(d), None) == 1
    assert lib.zarya_top_p(vp(FAKE + 8), 0.9, ctypes.byref(d), None) == 1
    for p in (0.0, -0.5, float("nan")):
        assert lib.zarya_top_p(vp(FAKE), p, ctypes.byref(d), None) == 1
    assert lib.zarya_top_p(vp(FAKE), 0.9, None, None) == 1
    assert lib.zarya_top_p(vp(FAKE), 1.0, ctypes.byref(d), None) == 0   # nothing to cut
    # overlapping rows (stride below the vocabulary) are refused before anything runs
    short = _sdesc(vocab=1000, row_stride=992)
    assert lib.zarya_top_p(vp(FAKE), 0.9, ctypes.byref(short), None) == 1
    # the kernel's 32-bit mass sums hold up to 520,192 tokens a row
    big = _sdesc(vocab=520_200, row_stride=520_200)
    assert lib.zarya_top_p(vp(FAKE), 0.9, ctypes.byref(big), None) == 2


def test_kernel_name_follows_the_plan(lib):
    """The paired kernel is planned for paged caches whose M-tile pairs fill
    the GPU; contiguous caches, a forced key split or few pairs keep the
    single-tile kernel; fp32 has its own; invalid descriptors name none."""
    name = lambda d: lib.zarya_slot_attn_kernel(ctypes.byref(d)).decode()  # noqa: E731
    paged = dict(batch=64, n_q_heads=32, n_kv_heads=8, page_size=16, cache_capacity=16640,
                 n_pages=30000, max_rows=256, total_rows=8192)
    assert name(_desc(**paged)) == "slot_attn_pair_kernel"
    assert name(_desc(**dict(paged, kv_splits=2))) == "slot_attn_tc_kernel"
    assert name(_desc(**dict(paged, batch=2))) == "slot_attn_tc_kernel"
    assert name(_desc(**dict(paged, page_size=0, n_pages=0))) == "slot_attn_tc_kernel"
    assert name(_desc(dtype=zb.FP32, head_dim=64)) == "slot_attn_f32_kernel"
    assert name(_desc(batch=0)) == "none"


def test_dispatch_order_is_planned_for_unsplit_multi_wave_launches(lib):
    """A paired launch (paged cache) taking several waves of CTAs gets a
    longest-first dispatch order: one more kernel and a workspace of one
    int32 per work item; other plans get neither."""
    wsz = lambda d: lib.zarya_slot_attn_workspace_size(ctypes.byref(d))  # noqa: E731
    nl = lambda d: lib.zarya_slot_attn_launches(ctypes.byref(d))  # noqa: E731
    paged = dict(batch=64, n_q_heads=32, n_kv_heads=8, page_size=16, cache_capacity=16640,
                 n_pages=30000, max_rows=256, total_rows=8192)
    d = _desc(**paged)                        # 64 x 4 pairs, x 8 heads: many waves
    assert nl(d) == 2 and wsz(d) == (64 * 4 * 4 + 255) // 256 * 256
    ragged = dict(batch=32, n_q_heads=32, n_kv_heads=8, cache_capacity=8320, max_rows=128,
                  total_rows=4096)
    assert nl(_desc(**ragged)) == 1 and wsz(_desc(**ragged)) == 0   # contiguous: grid order
    assert nl(_desc(**dict(paged, kv_splits=1))) == 1      # forced split: single-tile kernel
    assert nl(_desc(**dict(paged, batch=2))) == 1          # pairs do not fill the GPU
    assert nl(_desc()) == 1 and wsz(_desc()) == 0        # 16 CTAs: one wave
    assert nl(_desc(dtype=zb.FP32, head_dim=64)) == 1
    assert nl(_desc(batch=0)) == 0
