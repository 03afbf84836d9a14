"""GPU parity: the library's kernels (through the C ABI) against the CPU
oracle on the same seeded bf16 inputs."""
import numpy as np
import pytest
import torch

from oracle import attention as OA
from oracle import kv_cache as OK
from paper_2609_36757_gb300 import workloads as WL
from parity_helpers import Err, run_stream, to64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def FV():
    from paper_2609_36757_gb300 import fastvr
    return fastvr


# ------------------------------------------------------------- KV append
@pytest.mark.parametrize("w", [
    WL.custom("ring", batch=2, heads=3, head_dim=64, tokens_per_frame=5,
              frames_per_chunk=2, num_chunks=6, window_chunks=1,
              last_chunk_frames=1, seed=11),
    WL.custom("unbounded", batch=1, heads=12, head_dim=128,
              tokens_per_frame=1590, frames_per_chunk=2, num_chunks=4,
              seed=12),
    WL.custom("w0", batch=1, heads=2, head_dim=128, tokens_per_frame=77,
              frames_per_chunk=3, num_chunks=4, window_chunks=0,
              last_chunk_frames=2, seed=13),
], ids=lambda w: w.name)
def test_kv_append_is_bit_exact(FV, w):
    att = FV.StreamingAttention(FV.config_from_workload(w))
    att.cache.fill_(0x5A)
    ref = OK.RingCache(w.batch, w.heads, w.head_dim, w.tokens_per_frame,
                       w.frames_per_chunk, w.window_chunks, w.max_chunks,
                       fill=0x5A5A)
    region = ref.k.size * 2
    for c, q, k, v in WL.chunk_stream(w):
        att.append(k.cuda(), v.cuda())
        ref.append(k.view(torch.int16).numpy().view(np.uint16),
                   v.view(torch.int16).numpy().view(np.uint16))
        torch.cuda.synchronize()
        raw = att.cache.cpu().numpy()
        got_k = raw[:region].view(np.uint16).reshape(ref.k.shape)
        got_v = raw[region:2 * region].view(np.uint16).reshape(ref.v.shape)
        assert np.array_equal(got_k, ref.k), f"K differs after chunk {c}"
        assert np.array_equal(got_v, ref.v), f"V differs after chunk {c}"


# ------------------------------------------------- small streams, every element
SMALL = [
    # several 128-row Q tiles with a ragged tail, several key tiles per segment
    WL.custom("N300-k2", batch=1, heads=2, head_dim=128, tokens_per_frame=300,
              frames_per_chunk=2, num_chunks=4, seed=21),
    WL.custom("N97-k3-W1", batch=2, heads=3, head_dim=128, tokens_per_frame=97,
              frames_per_chunk=3, num_chunks=6, window_chunks=1,
              last_chunk_frames=2, seed=22),
    WL.custom("d64-N130-W2", batch=1, heads=4, head_dim=64,
              tokens_per_frame=130, frames_per_chunk=2, num_chunks=5,
              window_chunks=2, last_chunk_frames=1, seed=23),
    WL.custom("W0", batch=1, heads=2, head_dim=128, tokens_per_frame=200,
              frames_per_chunk=1, num_chunks=4, window_chunks=0, seed=24),
    WL.custom("N1-k1", batch=1, heads=2, head_dim=64, tokens_per_frame=1,
              frames_per_chunk=1, num_chunks=9, seed=25),
    WL.custom("peaked", batch=1, heads=2, head_dim=128, tokens_per_frame=250,
              frames_per_chunk=2, num_chunks=3, seed=26, peaked=True),
    WL.custom("ring-wrap", batch=1, heads=2, head_dim=128, tokens_per_frame=64,
              frames_per_chunk=2, num_chunks=9, window_chunks=3,
              last_chunk_frames=1, seed=27),
    # few query units, long key ranges: the units are cut into many key
    # ranges whose partial results are merged
    WL.custom("split-many", batch=1, heads=1, head_dim=128,
              tokens_per_frame=256, frames_per_chunk=2, num_chunks=8, seed=28),
    WL.custom("split-d64-ragged", batch=1, heads=1, head_dim=64,
              tokens_per_frame=200, frames_per_chunk=3, num_chunks=7,
              window_chunks=5, last_chunk_frames=1, seed=29),
]


@pytest.mark.parametrize("w", SMALL, ids=lambda w: w.name)
def test_small_stream_every_element(w):
    err = run_stream(w)
    err.check()


def _random_streams(n: int, seed: int):
    """Seeded random small streams: head dim, frame size (ragged against the
    128-row tiles, down to one token), chunk size, window and a ragged last
    chunk drawn at random; small enough for the oracle to check every
    element."""
    rng = np.random.default_rng(seed)
    out = []
    for i in range(n):
        k = int(rng.integers(1, 4))
        out.append(WL.custom(
            f"rand{i}", batch=int(rng.integers(1, 3)),
            heads=int(rng.integers(1, 4)),
            head_dim=int(rng.choice([64, 128])),
            tokens_per_frame=int(rng.integers(1, 260)),
            frames_per_chunk=k, num_chunks=int(rng.integers(2, 6)),
            window_chunks=int(rng.choice([-1, 0, 1, 2])),
            last_chunk_frames=int(rng.integers(0, k)), seed=300 + i))
    return out


RANDOM = _random_streams(12, 2609)


@pytest.mark.parametrize("w", RANDOM, ids=lambda w: w.name)
def test_random_small_stream_every_element(w):
    err = run_stream(w)
    err.check()


@pytest.mark.parametrize("w", SMALL[:3], ids=lambda w: w.name)
def test_streamed_gpu_equals_oneshot_oracle(FV, w):
    att = FV.StreamingAttention(FV.config_from_workload(w))
    qs, ks, vs, outs, lses = [], [], [], [], []
    for c, q, k, v in WL.chunk_stream(w):
        att.append(k.cuda(), v.cuda())
        o, l = att.forward(q.cuda(), want_lse=True)
        qs.append(q), ks.append(k), vs.append(v)
        outs.append(o.cpu()), lses.append(l.cpu())
    ref_o, ref_l = OA.blockcausal_attention(
        to64(torch.cat(qs, 1)), to64(torch.cat(ks, 1)), to64(torch.cat(vs, 1)),
        w.tokens_per_frame, w.frames_per_chunk, w.window_chunks,
        w.softmax_scale)
    err = Err()
    err.add(to64(torch.cat(outs, 1)), ref_o, torch.cat(lses, 2).numpy(), ref_l)
    err.check()


# ---------------------------------------- closed form: uniform attention
# With Q = 0 every visible score is 0, so P is exactly 1 on the visible keys
# of Eq. 1: O_i is the mean of V over them and the log-sum-exp is the log of
# their count, for the streamed and the one-shot path alike (no oracle).
# O = (sum of V) / n accumulates in fp32 and is rounded to bf16 once, so
# 1e-3 absolute covers it with room; the LSE is exact to fp32 rounding.
UNIFORM = [SMALL[0], SMALL[1], SMALL[2], SMALL[6]]


@pytest.mark.parametrize("w", UNIFORM, ids=lambda w: w.name)
def test_uniform_attention_closed_form(FV, w):
    att = FV.StreamingAttention(FV.config_from_workload(w))
    vs, qs, ks, vts, want_all = [], [], [], [], []
    for c, q, k, v in WL.chunk_stream(w):
        zq = torch.zeros_like(q)
        att.append(k.cuda(), v.cuda())
        o, lse = att.forward(zq.cuda(), want_lse=True)
        vs.append(to64(v))
        lo = 0 if w.window_chunks < 0 else max(0, c - w.window_chunks)
        vis = np.concatenate(vs[lo:c + 1], axis=1)           # [B, Lk, H, d]
        want = np.broadcast_to(vis.mean(axis=1, keepdims=True), q.shape)
        assert np.abs(to64(o.cpu()) - want).max() <= 1e-3, c
        assert np.abs(lse.cpu().double().numpy() - np.log(vis.shape[1])).max() <= 1e-5, c
        qs.append(zq), ks.append(k), vts.append(v), want_all.append(want)
    o1 = FV.blockcausal_attention(FV.config_from_workload(w),
                                  torch.cat(qs, 1).cuda(), torch.cat(ks, 1).cuda(),
                                  torch.cat(vts, 1).cuda())
    assert np.abs(to64(o1.cpu()) - np.concatenate(want_all, axis=1)).max() <= 1e-3


def test_forward_is_deterministic_and_repeatable(FV):
    w = SMALL[1]
    att = FV.StreamingAttention(FV.config_from_workload(w))
    for c, q, k, v in WL.chunk_stream(w):
        att.append(k.cuda(), v.cuda())
        qd = q.cuda()
        o1 = att.forward(qd)
        o2 = att.forward(qd)
        assert torch.equal(o1, o2)


def test_errors_on_the_gpu_path(FV):
    w = SMALL[1]
    att = FV.StreamingAttention(FV.config_from_workload(w))
    q = torch.zeros(w.chunk_shape(0), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(FV.FastVRError) as e:
        att.forward(q)
    assert e.value.status == FV.FASTVR_ERR_SEQUENCE
    att.append(q, q)
    ragged = q[:, :w.tokens_per_frame].contiguous()
    att.append(ragged, ragged)
    with pytest.raises(FV.FastVRError) as e:
        att.append(q, q)
    assert e.value.status == FV.FASTVR_ERR_SEQUENCE
    assert att.status() == FV.FASTVR_OK


# ------------------------------------------------------- the five workloads
def test_workload_tiny_every_element():
    run_stream(WL.TINY).check()


def test_workload_480p_every_element():
    run_stream(WL.W480P).check()


def test_workload_720p_peaked_sampled_rows():
    run_stream(WL.W720P_PEAKED, rows_per_chunk=256).check()


# Configs 3-5: 256 sampled rows per chunk (plus every frame's first and last
# row and the ragged tail), every chunk, every head; rows are independent, so
# each sampled row is exact.
def test_workload_1080p_sampled_rows():
    run_stream(WL.W1080P, rows_per_chunk=256).check()


def test_workload_1080p_windowed_sampled_rows():
    run_stream(WL.W1080P_WINDOWED, rows_per_chunk=256).check()


def test_paper_window_eq1_k3_w1_sampled_rows():
    # Eq. 1 as printed: each chunk sees itself and one predecessor, k = 3
    w = WL.custom("eq1-k3-W1", batch=1, heads=4, head_dim=128,
                  tokens_per_frame=8160, frames_per_chunk=3, num_chunks=5,
                  window_chunks=1, last_chunk_frames=2, seed=31)
    run_stream(w, rows_per_chunk=256).check()


# ------------------------------------------- the paper's own inference shape
def test_paper_tiles_32x32_sampled_rows():
    # k = 3, W = 1, six overlapping 64 x 64 latent tiles batched on B
    run_stream(WL.PAPER_TILES_32, rows_per_chunk=256).check()


def test_paper_tiles_64x64_sampled_rows():
    run_stream(WL.PAPER_TILES_64, rows_per_chunk=256).check()


# ------------------------------------ dependencies on the previous work
# The library's kernels start with programmatic dependent launch and wait
# for the preceding kernel before touching its data.  These streams feed
# every call from work queued just before it, with no synchronisation in
# between: (a) torch kernels on the same stream that produce q, k and v, and
# (b) pinned-host copies on a side stream that the compute stream waits for
# through events (the pattern of an end-to-end pipeline).
def test_inputs_from_kernels_queued_just_before():
    w = SMALL[1]
    from paper_2609_36757_gb300 import fastvr as FV
    att = FV.StreamingAttention(FV.config_from_workload(w))
    outs = []
    qs, ks, vs = [], [], []
    for c, q, k, v in WL.chunk_stream(w):
        qd, kd, vd = (x.cuda() for x in (q, k, v))
        torch.cuda.synchronize()
        # each input is rewritten by an elementwise kernel right before use
        k2, v2, q2 = kd * 1.0, vd * 1.0, qd * 1.0
        att.append(k2, v2)
        o = att.forward(q2)
        outs.append(o)
        qs.append(q), ks.append(k), vs.append(v)
    torch.cuda.synchronize()
    ref_o, _ = OA.blockcausal_attention(
        to64(torch.cat(qs, 1)), to64(torch.cat(ks, 1)), to64(torch.cat(vs, 1)),
        w.tokens_per_frame, w.frames_per_chunk, w.window_chunks,
        w.softmax_scale)
    err = Err()
    err.add(to64(torch.cat([o.cpu() for o in outs], 1)), ref_o)
    err.check()
    assert att.status() == FV.FASTVR_OK


def test_inputs_from_side_stream_copies():
    w = SMALL[0]
    from paper_2609_36757_gb300 import fastvr as FV
    att = FV.StreamingAttention(FV.config_from_workload(w))
    compute = torch.cuda.current_stream()
    side = torch.cuda.Stream()
    host = [(q.pin_memory(), k.pin_memory(), v.pin_memory())
            for _, q, k, v in WL.chunk_stream(w)]
    outs = []
    for q, k, v in host:
        with torch.cuda.stream(side):
            qd, kd, vd = (x.to("cuda", non_blocking=True) for x in (q, k, v))
            ready = torch.cuda.Event()
            ready.record(side)
        compute.wait_event(ready)
        for x in (qd, kd, vd):
            x.record_stream(compute)
        att.append(kd, vd)
        outs.append(att.forward(qd))
    torch.cuda.synchronize()
    ref_o, _ = OA.blockcausal_attention(
        to64(torch.cat([h[0] for h in host], 1)),
        to64(torch.cat([h[1] for h in host], 1)),
        to64(torch.cat([h[2] for h in host], 1)),
        w.tokens_per_frame, w.frames_per_chunk, w.window_chunks,
        w.softmax_scale)
    err = Err()
    err.add(to64(torch.cat([o.cpu() for o in outs], 1)), ref_o)
    err.check()
    assert att.status() == FV.FASTVR_OK
