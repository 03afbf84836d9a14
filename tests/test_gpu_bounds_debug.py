"""The debug library (libfastvr_attn_debug.so, built with FASTVR_BOUNDS_CHECK)
checks every computed global-memory index of the append and attention
kernels before the access.  On correct inputs it reports nothing and gives
the release library's outputs bit for bit; a deliberately shifted append
destination is caught (FASTVR_ERR_BOUNDS), the stray writes skipped."""
import gc

import pytest
import torch

from paper_2609_36757_gb300 import workloads as WL

pytestmark = pytest.mark.gpu

CASES = [
    # several query tiles with a ragged tail, key tiles of two segments
    WL.custom("N300-k2", batch=1, heads=2, head_dim=128, tokens_per_frame=300,
              frames_per_chunk=2, num_chunks=4, seed=21),
    # units cut into many key ranges: workspace writes and the merge kernel
    WL.custom("split-many", batch=1, heads=1, head_dim=128,
              tokens_per_frame=256, frames_per_chunk=2, num_chunks=8, seed=28),
    # d = 64, a ring that wraps, a ragged last chunk
    WL.custom("d64-N130-W2", batch=1, heads=4, head_dim=64,
              tokens_per_frame=130, frames_per_chunk=2, num_chunks=5,
              window_chunks=2, last_chunk_frames=1, seed=23),
]


def _stream(FV, w):
    att = FV.StreamingAttention(FV.config_from_workload(w))
    outs = []
    for _, q, k, v in WL.chunk_stream(w):
        att.append(k.cuda(), v.cuda())
        o, lse = att.forward(q.cuda(), want_lse=True)
        outs.append((o.cpu(), lse.cpu()))
    status = att.status()
    del att
    gc.collect()
    return outs, status


@pytest.mark.parametrize("w", CASES, ids=lambda w: w.name)
def test_debug_library_runs_clean_and_matches_release(w):
    from paper_2609_36757_gb300 import fastvr as FV
    ref, status = _stream(FV, w)
    assert status == FV.FASTVR_OK
    previous = FV.use_library(FV.DEBUG_LIB_PATH)
    try:
        got, status = _stream(FV, w)
    finally:
        FV.lib = previous
    assert status == FV.FASTVR_OK
    for (o_ref, l_ref), (o, l) in zip(ref, got):
        assert torch.equal(o_ref, o) and torch.equal(l_ref, l)


def test_debug_library_catches_a_shifted_append():
    from paper_2609_36757_gb300 import fastvr as FV
    # W = 1: a ring of two slots of k N = 128 tokens.  The second chunk goes to
    # the last slot; shifted by 64 tokens, its last 64 tokens per head would
    # land past the head's cache (for the last head, past the K region, still
    # inside the plan's buffer).
    w = WL.custom("shift", batch=1, heads=2, head_dim=64, tokens_per_frame=64,
                  frames_per_chunk=2, num_chunks=2, window_chunks=1, seed=31)
    chunks = list(WL.chunk_stream(w))
    previous = FV.use_library(FV.DEBUG_LIB_PATH)
    try:
        att = FV.StreamingAttention(FV.config_from_workload(w))
        _, _, k0, v0 = chunks[0]
        att.append(k0.cuda(), v0.cuda())
        assert att.status() == FV.FASTVR_OK
        FV.fastvr_debug_shift_next_append(att.plan, 64)
        _, _, k1, v1 = chunks[1]
        att.append(k1.cuda(), v1.cuda())
        assert att.status() == FV.FASTVR_ERR_BOUNDS
        assert att.status() == FV.FASTVR_OK  # the word is cleared when read
        del att
        gc.collect()
    finally:
        FV.lib = previous
