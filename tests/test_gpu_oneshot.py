"""GPU parity of the one-shot (training-form) chunk-causal attention: the
whole latent sequence at once under the mask of Eq. 1 (Sec. 3.1), against
the oracle's one-shot form, and against the library's own streamed form."""
import numpy as np
import pytest
import torch

from oracle import attention as OA
from paper_2609_36757_gb300 import workloads as WL
from parity_helpers import Err, sample_rows, to64

pytestmark = pytest.mark.gpu


def _sequence(w):
    qs, ks, vs = [], [], []
    for _, q, k, v in WL.chunk_stream(w):
        qs.append(q), ks.append(k), vs.append(v)
    return torch.cat(qs, 1), torch.cat(ks, 1), torch.cat(vs, 1)


def _oneshot(w, q, k, v):
    from paper_2609_36757_gb300 import fastvr as FV
    cfg = FV.config_from_workload(w)
    o, lse = FV.blockcausal_attention(cfg, q.cuda(), k.cuda(), v.cuda(),
                                      want_lse=True)
    torch.cuda.synchronize()
    return o.cpu(), lse.cpu()


CASES = [
    # 256-row query units straddle chunk boundaries (k N = 600)
    WL.custom("N300-k2", batch=1, heads=2, head_dim=128, tokens_per_frame=300,
              frames_per_chunk=2, num_chunks=4, seed=61),
    # Eq. 1 itself: one predecessor chunk; ragged final chunk
    WL.custom("eq1-W1", batch=2, heads=2, head_dim=128, tokens_per_frame=97,
              frames_per_chunk=3, num_chunks=6, window_chunks=1,
              last_chunk_frames=2, seed=62),
    WL.custom("W0", batch=1, heads=3, head_dim=128, tokens_per_frame=150,
              frames_per_chunk=1, num_chunks=5, window_chunks=0, seed=63),
    WL.custom("d64-W2", batch=1, heads=2, head_dim=64, tokens_per_frame=130,
              frames_per_chunk=2, num_chunks=6, window_chunks=2,
              last_chunk_frames=1, seed=64),
    # token-causal (one token per frame, one frame per chunk): every key
    # tile is masked element-wise
    WL.custom("token-causal", batch=1, heads=2, head_dim=64,
              tokens_per_frame=1, frames_per_chunk=1, num_chunks=700, seed=65),
    # k N = 128: query tiles and chunks align
    WL.custom("aligned", batch=1, heads=2, head_dim=128, tokens_per_frame=64,
              frames_per_chunk=2, num_chunks=9, seed=66),
]


@pytest.mark.parametrize("w", CASES, ids=lambda w: w.name)
def test_oneshot_every_element_vs_oracle(w):
    q, k, v = _sequence(w)
    o, lse = _oneshot(w, q, k, v)
    ref_o, ref_l = OA.blockcausal_attention(
        to64(q), to64(k), to64(v), w.tokens_per_frame, w.frames_per_chunk,
        w.window_chunks, w.softmax_scale)
    err = Err()
    err.add(to64(o), ref_o, lse.numpy(), ref_l)
    err.check()


def test_oneshot_equals_streamed_on_the_gpu():
    from paper_2609_36757_gb300 import fastvr as FV
    w = WL.custom("480p-shape", batch=1, heads=12, head_dim=128,
                  tokens_per_frame=1590, frames_per_chunk=2, num_chunks=5,
                  seed=67)
    att = FV.StreamingAttention(FV.config_from_workload(w))
    outs, lses, qs, ks, vs = [], [], [], [], []
    for _, q, k, v in WL.chunk_stream(w):
        att.append(k.cuda(), v.cuda())
        o, l = att.forward(q.cuda(), want_lse=True)
        outs.append(o.cpu()), lses.append(l.cpu())
        qs.append(q), ks.append(k), vs.append(v)
    o1, l1 = _oneshot(w, torch.cat(qs, 1), torch.cat(ks, 1), torch.cat(vs, 1))
    err = Err()
    err.add(to64(o1), to64(torch.cat(outs, 1)), l1.numpy(),
            torch.cat(lses, 2).double().numpy())
    err.check()


def test_oneshot_eq1_k3_w1_1080p_frames_sampled_rows():
    w = WL.custom("eq1-1080p", batch=1, heads=4, head_dim=128,
                  tokens_per_frame=8160, frames_per_chunk=3, num_chunks=5,
                  window_chunks=1, last_chunk_frames=2, seed=68)
    q, k, v = _sequence(w)
    o, lse = _oneshot(w, q, k, v)
    L = q.shape[1]
    rows = sample_rows(L, w.tokens_per_frame, 96, 7)
    # rows on both sides of every chunk boundary
    span = w.frames_per_chunk * w.tokens_per_frame
    rows = np.unique(np.concatenate([rows] + [
        np.array([c * span - 1, c * span]) for c in range(1, w.num_chunks)]))
    ref_o, ref_l = OA.blockcausal_attention(
        to64(q), to64(k), to64(v), w.tokens_per_frame, w.frames_per_chunk,
        w.window_chunks, w.softmax_scale, rows=rows)
    err = Err()
    err.add(to64(o[:, rows]), ref_o, lse[:, :, rows].numpy(), ref_l)
    err.check()


def test_oneshot_rejects_bad_arguments():
    from paper_2609_36757_gb300 import fastvr as FV
    cfg = FV.make_config(1, 2, 96, 64, 2)
    x = torch.zeros((1, 128, 2, 96), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(FV.FastVRError) as e:
        FV.fastvr_blockcausal_attn_fwd(cfg, 2, x.data_ptr(), x.data_ptr(),
                                       x.data_ptr(), x.data_ptr(), 0, 0)
    assert e.value.status == FV.FASTVR_ERR_UNSUPPORTED
    cfg = FV.make_config(1, 2, 128, 64, 2)
    with pytest.raises(FV.FastVRError) as e:
        FV.fastvr_blockcausal_attn_fwd(cfg, 0, x.data_ptr(), x.data_ptr(),
                                       x.data_ptr(), x.data_ptr(), 0, 0)
    assert e.value.status == FV.FASTVR_ERR_INVALID_ARG
