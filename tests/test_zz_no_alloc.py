"""The allocation-free attention entry point (fastvr_chunk_attn_fwd_static).

It serves callers that cannot allocate device memory: engines that own all
device memory through their own pool and keep K and V in their own buffers,
and real-time pipelines that forbid cudaMalloc/cudaFree after start-up.  Its
split-KV scratch is a fixed device array inside the library instead of the
workspace region of a plan's cache buffer.  Here it is called through the C
ABI, twice in a row per chunk, on K/V that live in a plan's cache, and each
output must match the plan entry point's output on the same inputs within
the tolerances the parity tests use.  The device's free memory must not move
across a call, some chunk of each case must be split along the keys (so the
static scratch is really used), and no timeout may be recorded.  The file is
collected last so that a run that stops at its first failure has already run
every other test."""
import pytest
import torch

from paper_2609_36757_gb300 import workloads as WL
from parity_helpers import Err, to64

pytestmark = pytest.mark.gpu


CASES = [
    # 156 query units on 152 SMs: the last units are split along the keys
    WL.custom("480p-shape", batch=1, heads=12, head_dim=128,
              tokens_per_frame=1590, frames_per_chunk=2, num_chunks=3, seed=51),
    # d = 64, ring window with two visible segments, ragged last chunk
    WL.custom("d64-ring", batch=1, heads=1, head_dim=64, tokens_per_frame=200,
              frames_per_chunk=3, num_chunks=7, window_chunks=2,
              last_chunk_frames=1, seed=52),
]


def _region_bytes(w, slots):
    per = w.batch * w.heads * slots * w.frames_per_chunk * \
        w.tokens_per_frame * w.head_dim * 2
    return (per + 255) // 256 * 256


@pytest.mark.parametrize("w", CASES, ids=lambda w: w.name)
def test_static_scratch_entry_matches_plan_entry_on_two_calls(w):
    from paper_2609_36757_gb300 import fastvr as FV
    cfg = FV.config_from_workload(w)
    att = FV.StreamingAttention(cfg)
    slots = w.window_chunks + 1 if w.window_chunks >= 0 else w.max_chunks
    cache_tokens = slots * w.frames_per_chunk * w.tokens_per_frame
    k_ptr = att.cache.data_ptr()
    v_ptr = k_ptr + _region_bytes(w, slots)
    stream = torch.cuda.current_stream().cuda_stream
    splits = 0
    for c, q, k, v in WL.chunk_stream(w):
        att.append(k.cuda(), v.cuda())
        qd = q.cuda()
        before = att.launch_count()
        ref_o, ref_l = att.forward(qd, want_lse=True)
        # two launches: some units were cut along the keys, so the partial
        # results went through the scratch (the same split in both paths)
        splits += att.launch_count() - before == 2
        segments, _ = att.visible()
        frames = q.shape[1] // w.tokens_per_frame
        prev = None
        for call in range(2):
            o = torch.full_like(qd, float("nan"))
            lse = torch.full_like(ref_l, float("nan"))
            torch.cuda.synchronize()
            free_before = torch.cuda.mem_get_info()[0]
            FV.fastvr_chunk_attn_fwd_static(
                cfg, qd.data_ptr(), frames, k_ptr, v_ptr, cache_tokens,
                segments, o.data_ptr(), lse.data_ptr(), stream)
            torch.cuda.synchronize()
            if call == 1:
                # the device's free memory is unchanged by a call (the first
                # call on a device may load the library's kernels)
                assert torch.cuda.mem_get_info()[0] == free_before
            err = Err()
            err.add(to64(o.cpu()), to64(ref_o.cpu()), lse.cpu().numpy(),
                    ref_l.cpu().double().numpy())
            err.check()
            if prev is not None:
                assert torch.equal(o, prev), f"calls differ at chunk {c}"
            prev = o
    assert att.status() == FV.FASTVR_OK
    assert FV.fastvr_get_device_status() == FV.FASTVR_OK
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert splits > 0, f"no chunk of {w.name} was split on {sms} SMs"
