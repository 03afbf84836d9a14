"""Checkpoint/resume of a stream: its whole state is the cache buffer plus
the plan's counters (chunks appended, frames of the newest chunk).  A stream
interrupted after some chunks, saved to host memory and restored into a new
plan and buffer, must continue exactly as the uninterrupted stream does."""
import pytest
import torch

from paper_2609_36757_gb300 import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("w,stop", [
    (WL.custom("resume-ring", batch=1, heads=2, head_dim=128,
               tokens_per_frame=200, frames_per_chunk=2, num_chunks=7,
               window_chunks=2, last_chunk_frames=1, seed=81), 4),
    (WL.custom("resume-unbounded", batch=2, heads=3, head_dim=64,
               tokens_per_frame=97, frames_per_chunk=3, num_chunks=5,
               seed=82), 2),
], ids=lambda x: getattr(x, "name", str(x)))
def test_resumed_stream_is_bit_identical(w, stop):
    from paper_2609_36757_gb300 import fastvr as FV
    cfg = FV.config_from_workload(w)
    chunks = list(WL.chunk_stream(w))

    ref = FV.StreamingAttention(cfg)
    ref_out = []
    for _, q, k, v in chunks:
        ref.append(k.cuda(), v.cuda())
        ref_out.append(ref.forward(q.cuda(), want_lse=True))

    first = FV.StreamingAttention(cfg)
    for _, q, k, v in chunks[:stop]:
        first.append(k.cuda(), v.cuda())
        first.forward(q.cuda())
    torch.cuda.synchronize()
    saved_cache = first.cache.cpu()          # checkpoint: bytes + counters
    saved_state = first.state()
    del first

    resumed = FV.StreamingAttention(cfg)
    resumed.cache.copy_(saved_cache)
    resumed.set_state(*saved_state)
    for c, q, k, v in chunks[stop:]:
        resumed.append(k.cuda(), v.cuda())
        o, lse = resumed.forward(q.cuda(), want_lse=True)
        ro, rl = ref_out[c]
        assert torch.equal(o, ro), f"output differs at chunk {c}"
        assert torch.equal(lse, rl), f"lse differs at chunk {c}"
    assert resumed.state() == ref.state()
    assert resumed.status() == FV.FASTVR_OK
