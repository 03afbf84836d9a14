"""CPU tests of the C ABI: the library loads, exports every declared symbol,
and its host logic (validation, sequencing, ring slots, visible segments)
matches the oracle's definition of visibility.  No compute call runs here."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import attention as OA
from oracle import kv_cache as OK

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def fv():
    from paper_2609_36757_gb300 import build
    build.build()
    from paper_2609_36757_gb300 import fastvr
    return fastvr


def _declared_symbols():
    names = set()
    inc = os.path.join(ROOT, "include")
    for fn in os.listdir(inc):
        if fn.endswith(".h"):
            src = open(os.path.join(inc, fn)).read()
            names |= set(re.findall(r"FASTVR_API\s+[\w\s\*]*?\b(fastvr_\w+)\s*\(",
                                    src))
    return names


def test_every_declared_symbol_is_exported(fv):
    names = _declared_symbols()
    assert len(names) >= 11
    lib = ctypes.CDLL(fv.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert names == set(fv.SIGNATURES), "binding and header disagree"


def test_debug_library_exports_the_same_symbols(fv):
    names = _declared_symbols()
    lib = ctypes.CDLL(fv.DEBUG_LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n


def test_append_shift_hook_exists_only_in_the_debug_library(fv):
    cfg, plan = _plan(fv)
    try:
        with pytest.raises(fv.FastVRError) as e:
            fv.fastvr_debug_shift_next_append(plan, 1)
        assert e.value.status == fv.FASTVR_ERR_UNSUPPORTED
        previous = fv.use_library(fv.DEBUG_LIB_PATH)
        try:
            dplan = fv.fastvr_attn_plan(cfg, FAKE, fv.fastvr_kv_cache_bytes(cfg))
            try:
                fv.fastvr_debug_shift_next_append(dplan, 8)  # one slot: k N
                for bad in (-1, 9):
                    with pytest.raises(fv.FastVRError) as e:
                        fv.fastvr_debug_shift_next_append(dplan, bad)
                    assert e.value.status == fv.FASTVR_ERR_INVALID_ARG
            finally:
                fv.fastvr_plan_destroy(dplan)
        finally:
            fv.lib = previous
    finally:
        fv.fastvr_plan_destroy(plan)


def test_status_strings(fv):
    assert fv.fastvr_status_string(fv.FASTVR_OK) == "FASTVR_OK"
    assert fv.fastvr_status_string(fv.FASTVR_ERR_TIMEOUT) == "FASTVR_ERR_TIMEOUT"
    assert fv.fastvr_status_string(fv.FASTVR_ERR_BOUNDS) == "FASTVR_ERR_BOUNDS"
    assert fv.fastvr_status_string(99) == "FASTVR_ERR_UNKNOWN"


def test_cache_bytes_formula(fv):
    # K and V regions, the split-KV workspace (256 parts x 256 rows x
    # (d + 1) floats), the 256-byte control block
    ws = lambda d: 256 * 256 * (d + 1) * 4
    cfg = fv.make_config(2, 3, 128, 10, 3, window_chunks=4)
    slots = 5
    per = 2 * 3 * slots * 3 * 10 * 128 * 2
    assert fv.fastvr_kv_cache_bytes(cfg) == \
        2 * ((per + 255) // 256 * 256) + ws(128) + 256
    cfg = fv.make_config(1, 12, 128, 8160, 2, -1, 15)
    assert fv.fastvr_kv_cache_bytes(cfg) == \
        2 * 12 * 15 * 2 * 8160 * 256 + ws(128) + 256
    cfg = fv.make_config(1, 2, 64, 64, 2, -1, 3)
    assert fv.fastvr_kv_cache_bytes(cfg) == 2 * 2 * 3 * 2 * 64 * 128 + ws(64) + 256


@pytest.mark.parametrize("kw,code", [
    (dict(batch=0), 1), (dict(heads=-1), 1), (dict(tokens_per_frame=0), 1),
    (dict(frames_per_chunk=0), 1), (dict(window_chunks=-2), 1),
    (dict(window_chunks=-1, max_chunks=0), 1), (dict(softmax_scale=-1.0), 1),
    (dict(head_dim=96), 2), (dict(head_dim=256), 2),
])
def test_config_validation(fv, kw, code):
    base = dict(batch=1, heads=2, head_dim=64, tokens_per_frame=4,
                frames_per_chunk=2, window_chunks=1, max_chunks=0,
                softmax_scale=0.0)
    base.update(kw)
    cfg = fv.make_config(**base)
    with pytest.raises(fv.FastVRError) as e:
        fv.fastvr_kv_cache_bytes(cfg)
    assert e.value.status == code


FAKE = 1 << 40  # a 256-aligned address: plan creation is host only


def _plan(fv, **kw):
    base = dict(batch=1, heads=2, head_dim=64, tokens_per_frame=4,
                frames_per_chunk=2, window_chunks=1, max_chunks=0)
    base.update(kw)
    cfg = fv.make_config(**base)
    return cfg, fv.fastvr_attn_plan(cfg, FAKE, fv.fastvr_kv_cache_bytes(cfg))


def test_plan_rejects_small_or_misaligned_buffers(fv):
    cfg = fv.make_config(1, 2, 64, 4, 2, 1, 0)
    need = fv.fastvr_kv_cache_bytes(cfg)
    with pytest.raises(fv.FastVRError) as e:
        fv.fastvr_attn_plan(cfg, FAKE, need - 1)
    assert e.value.status == fv.FASTVR_ERR_CAPACITY
    with pytest.raises(fv.FastVRError) as e:
        fv.fastvr_attn_plan(cfg, FAKE + 16, need)
    assert e.value.status == fv.FASTVR_ERR_INVALID_ARG
    with pytest.raises(fv.FastVRError) as e:
        fv.fastvr_attn_plan(cfg, 0, need)
    assert e.value.status == fv.FASTVR_ERR_INVALID_ARG


def test_sequencing_errors_before_any_device_work(fv):
    cfg, plan = _plan(fv, window_chunks=-1, max_chunks=3)
    try:
        with pytest.raises(fv.FastVRError) as e:  # nothing appended yet
            fv.fastvr_chunk_attn_fwd(plan, FAKE, FAKE, 0, 0)
        assert e.value.status == fv.FASTVR_ERR_SEQUENCE
        with pytest.raises(fv.FastVRError) as e:
            fv.fastvr_plan_visible(plan)
        assert e.value.status == fv.FASTVR_ERR_SEQUENCE
        with pytest.raises(fv.FastVRError) as e:  # frames > k
            fv.fastvr_kv_append(plan, FAKE, FAKE, 3, 0)
        assert e.value.status == fv.FASTVR_ERR_CAPACITY
        with pytest.raises(fv.FastVRError) as e:  # frames < 1
            fv.fastvr_kv_append(plan, FAKE, FAKE, 0, 0)
        assert e.value.status == fv.FASTVR_ERR_INVALID_ARG
        with pytest.raises(fv.FastVRError) as e:  # misaligned input
            fv.fastvr_kv_append(plan, FAKE + 8, FAKE, 2, 0)
        assert e.value.status == fv.FASTVR_ERR_INVALID_ARG
        fv.fastvr_plan_set_state(plan, 3, 2)
        with pytest.raises(fv.FastVRError) as e:  # capacity reached
            fv.fastvr_kv_append(plan, FAKE, FAKE, 2, 0)
        assert e.value.status == fv.FASTVR_ERR_CAPACITY
        fv.fastvr_plan_set_state(plan, 2, 1)
        with pytest.raises(fv.FastVRError) as e:  # after a ragged final chunk
            fv.fastvr_kv_append(plan, FAKE, FAKE, 2, 0)
        assert e.value.status == fv.FASTVR_ERR_SEQUENCE
        with pytest.raises(fv.FastVRError):
            fv.fastvr_plan_set_state(plan, 4, 2)  # beyond capacity
        with pytest.raises(fv.FastVRError):
            fv.fastvr_plan_set_state(plan, 1, 3)  # more frames than k
        fv.fastvr_plan_reset(plan)
        assert fv.fastvr_plan_get_state(plan) == (0, 0)
    finally:
        fv.fastvr_plan_destroy(plan)


def test_device_calls_fail_without_a_gpu(fv):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    _, plan = _plan(fv)
    try:
        with pytest.raises(fv.FastVRError) as e:
            fv.fastvr_kv_append(plan, FAKE, FAKE, 2, 0)
        assert e.value.status in (fv.FASTVR_ERR_CUDA, fv.FASTVR_ERR_UNSUPPORTED)
        assert fv.fastvr_plan_get_state(plan) == (0, 0)  # no state change
    finally:
        fv.fastvr_plan_destroy(plan)


def _oracle_visible_tokens(W, max_chunks, k, N, chunks, last_frames):
    """Cache token indices the newest chunk must read, from the oracle's
    definitions: visible chunks (Eq. 1 with window W) placed by the ring
    layout (chunk c' in slot c' mod S)."""
    S = OK.num_slots(W, max_chunks)
    c = chunks - 1
    toks = set()
    for cc in OA.visible_chunks(c, W):
        f = last_frames if cc == c else k
        base = (cc % S) * k * N
        toks |= set(range(base, base + f * N))
    return toks


@pytest.mark.parametrize("W,max_chunks,k,N", [
    (-1, 6, 2, 5), (0, 0, 3, 4), (1, 0, 3, 4), (4, 0, 3, 7), (2, 0, 1, 3)])
def test_visible_segments_match_oracle(fv, W, max_chunks, k, N):
    cfg, plan = _plan(fv, window_chunks=W, max_chunks=max_chunks,
                      frames_per_chunk=k, tokens_per_frame=N)
    try:
        limit = max_chunks if W < 0 else 13
        for chunks in range(1, limit + 1):
            for last in range(1, k + 1):
                fv.fastvr_plan_set_state(plan, chunks, last)
                segs, total = fv.fastvr_plan_visible(plan)
                assert 1 <= len(segs) <= 2
                got = set()
                for s, n in segs:
                    assert n > 0
                    got |= set(range(s, s + n))
                want = _oracle_visible_tokens(W, max_chunks, k, N, chunks, last)
                assert got == want
                assert total == len(want)
                if W >= 0:  # the cache holds at most (W+1) k N tokens
                    assert total <= (W + 1) * k * N
    finally:
        fv.fastvr_plan_destroy(plan)


def test_visible_counts_match_oracle_pair_counts(fv):
    # per-chunk visible keys x chunk tokens == the oracle's visible pairs
    frames = [3] * 9 + [1]
    N, W = 5, 4
    cfg, plan = _plan(fv, window_chunks=W, frames_per_chunk=3,
                      tokens_per_frame=N)
    try:
        want = OA.visible_pairs_per_chunk(frames, N, W)
        for c, f in enumerate(frames):
            fv.fastvr_plan_set_state(plan, c + 1, f)
            _, lk = fv.fastvr_plan_visible(plan)
            assert f * N * lk == want[c]
    finally:
        fv.fastvr_plan_destroy(plan)


def test_static_entry_rejects_bad_arguments_before_any_device_work(fv):
    cfg = fv.make_config(1, 2, 128, 64, 2, -1, 4)
    ok_seg = [(0, 128)]
    cases = [
        dict(q=0), dict(q_frames=0), dict(cache_tokens=0),
        dict(segments=[(0, 64)] * 3), dict(segments=[(0, 0)]),
        dict(segments=[(200, 100)]), dict(segments=[(-1, 10)]),
        dict(q=FAKE + 8), dict(out=FAKE + 4), dict(k=FAKE + 2),
        dict(v=FAKE + 8), dict(lse=FAKE + 2),
        # q_frames * N past 2^30 - 1 (32-bit token indexing in the kernels)
        dict(q_frames=1 << 24),
        # a segment ending past 2^30 - 1, even inside a huge cache
        dict(segments=[((1 << 30) - 64, 128)], cache_tokens=1 << 40),
        dict(segments=[(0, 128), ((1 << 31), 128)], cache_tokens=1 << 40),
        dict(cfg=fv.make_config(1, 2, 128, 64, 2, -1, 4, float("inf"))),
        dict(cfg=fv.make_config(1, 2, 128, 64, 2, -1, 4, float("nan"))),
        dict(cfg=fv.make_config(1, 2, 128, 64, 2, -1, 4, -1.0)),
    ]
    for kw in cases:
        a = dict(cfg=cfg, q=FAKE, q_frames=1, k=FAKE, v=FAKE,
                 cache_tokens=256, segments=ok_seg, out=FAKE, lse=0)
        a.update(kw)
        with pytest.raises(fv.FastVRError) as e:
            fv.fastvr_chunk_attn_fwd_static(a["cfg"], a["q"], a["q_frames"],
                                            a["k"], a["v"], a["cache_tokens"],
                                            a["segments"], a["out"], a["lse"],
                                            0)
        assert e.value.status == fv.FASTVR_ERR_INVALID_ARG, kw
    bad_d = fv.make_config(1, 2, 96, 64, 2, -1, 4)
    with pytest.raises(fv.FastVRError) as e:
        fv.fastvr_chunk_attn_fwd_static(bad_d, FAKE, 1, FAKE, FAKE, 256, ok_seg,
                                        FAKE, 0, 0)
    assert e.value.status == fv.FASTVR_ERR_UNSUPPORTED
