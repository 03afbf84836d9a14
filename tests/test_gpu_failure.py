"""Failure detection on the GPU without a fault or a hang: every wait inside
the attention kernels is bounded; a test hook makes one wait run out (a
barrier nothing arrives on) and the host must read FASTVR_ERR_TIMEOUT, after
which the same context (and plan) keep producing correct results.  The
streamed path reports through its plan, the calls without a plan (one-shot
forward, backward) through the device status word."""
import time

import pytest

from paper_2609_36757_gb300 import workloads as WL
from parity_helpers import Err, to64
from oracle import attention as OA

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_survives():
    from paper_2609_36757_gb300 import fastvr as FV
    w = WL.custom("stall", batch=1, heads=2, head_dim=128,
                  tokens_per_frame=200, frames_per_chunk=2, num_chunks=2,
                  seed=41)
    att = FV.StreamingAttention(FV.config_from_workload(w))
    (_, q, k, v), = [next(WL.chunk_stream(w))]
    att.append(k.cuda(), v.cuda())
    FV.fastvr_debug_inject_stall(att.plan, 1, 20_000_000)  # 20 ms per wait
    t0 = time.perf_counter()
    att.forward(q.cuda())
    status = att.status()
    elapsed = time.perf_counter() - t0
    assert status == FV.FASTVR_ERR_TIMEOUT
    assert elapsed < 5.0
    assert att.status() == FV.FASTVR_OK  # reading the status clears it

    FV.fastvr_debug_inject_stall(att.plan, 0, 0)
    o, lse = att.forward(q.cuda(), want_lse=True)
    assert att.status() == FV.FASTVR_OK
    ref_o, ref_l = OA.chunk_attention(to64(q), to64(k), to64(v),
                                      w.softmax_scale)
    err = Err()
    err.add(to64(o.cpu()), ref_o, lse.cpu().numpy(), ref_l)
    err.check()


def _noplan_case():
    import torch
    w = WL.custom("stall-noplan", batch=1, heads=2, head_dim=128,
                  tokens_per_frame=200, frames_per_chunk=2, num_chunks=3,
                  window_chunks=1, seed=42)
    qs, ks, vs = [], [], []
    for _, q, k, v in WL.chunk_stream(w):
        qs.append(q), ks.append(k), vs.append(v)
    return w, [torch.cat(t, 1).cuda() for t in (qs, ks, vs)]


def test_oneshot_forward_timeout_is_reported_and_context_survives():
    from paper_2609_36757_gb300 import fastvr as FV
    w, (q, k, v) = _noplan_case()
    cfg = FV.config_from_workload(w)
    assert FV.fastvr_get_device_status() == FV.FASTVR_OK
    ref = FV.blockcausal_attention(cfg, q, k, v)
    FV.fastvr_debug_inject_stall_noplan(1, 20_000_000)  # 20 ms per wait
    try:
        t0 = time.perf_counter()
        FV.blockcausal_attention(cfg, q, k, v)
        status = FV.fastvr_get_device_status()
        assert time.perf_counter() - t0 < 5.0
    finally:
        FV.fastvr_debug_inject_stall_noplan(0, 0)
    assert status == FV.FASTVR_ERR_TIMEOUT
    assert FV.fastvr_get_device_status() == FV.FASTVR_OK  # cleared
    out = FV.blockcausal_attention(cfg, q, k, v)
    assert FV.fastvr_get_device_status() == FV.FASTVR_OK
    assert (out == ref).all()


def test_backward_timeout_is_reported_and_context_survives():
    import torch
    from paper_2609_36757_gb300 import fastvr as FV
    w, (q, k, v) = _noplan_case()
    cfg = FV.config_from_workload(w)
    o, lse = FV.blockcausal_attention(cfg, q, k, v, want_lse=True)
    do = torch.randn_like(q.float()).to(torch.bfloat16)
    ref = FV.blockcausal_attention_bwd(cfg, q, k, v, o, do, lse)
    assert FV.fastvr_get_device_status() == FV.FASTVR_OK
    FV.fastvr_debug_inject_stall_noplan(1, 20_000_000)
    try:
        t0 = time.perf_counter()
        FV.blockcausal_attention_bwd(cfg, q, k, v, o, do, lse)
        status = FV.fastvr_get_device_status()
        assert time.perf_counter() - t0 < 5.0
    finally:
        FV.fastvr_debug_inject_stall_noplan(0, 0)
    assert status == FV.FASTVR_ERR_TIMEOUT
    got = FV.blockcausal_attention_bwd(cfg, q, k, v, o, do, lse)
    assert FV.fastvr_get_device_status() == FV.FASTVR_OK
    for a, b in zip(got, ref):
        assert torch.equal(a, b)
