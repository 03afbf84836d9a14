"""Pins for the CPU oracle: each check ties it to something other than itself
(hand-evaluated Eq. 1 masks, a scalar brute force, library attention in the
special cases that reduce to it, closed forms, invariants), and the planted
mistakes at the bottom show that a plausible error in the oracle fails a pin."""
import math
import os

import numpy as np
import pytest
import torch

from oracle import attention as A
from oracle import kv_cache as KC

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load_mask(name):
    rows, params = [], None
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            if params is None:
                params = dict(kv.split("=") for kv in line.split())
                continue
            rows.append([c == "1" for c in line])
    return {k: int(v) for k, v in params.items()}, np.array(rows, dtype=bool)


MASK_FILES = ["eq1_mask_T7_k3_W1.txt", "eq1_mask_T8_k2_W1.txt",
              "mask_T6_k2_unbounded.txt", "mask_T5_k1_W2.txt"]


def _rand(shape, seed, scale=1.0):
    g = np.random.default_rng(seed)
    # bf16-representable values, as the GPU path consumes
    x = torch.from_numpy(g.standard_normal(shape) * scale).to(torch.bfloat16)
    return x.double().numpy()


def _sdpa(q, k, v, scale, mask=None, causal=False):
    """torch SDPA (float64, CPU) on one head: q [L, d]."""
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x))[None, None]
    m = None if mask is None else torch.from_numpy(mask)[None, None]
    o = torch.nn.functional.scaled_dot_product_attention(
        t(q), t(k), t(v), attn_mask=m, is_causal=causal, scale=scale)
    return o[0, 0].numpy()


# ---------------------------------------------------------------- masks
@pytest.mark.parametrize("name", MASK_FILES)
def test_frame_mask_matches_hand_evaluated_eq1(name):
    p, want = _load_mask(name)
    got = A.frame_mask(p["T"], p["k"], p["W"])
    assert got.shape == want.shape
    assert (got == want).all()


@pytest.mark.parametrize("name", MASK_FILES)
def test_chunk_visible_matches_hand_evaluated_eq1(name):
    p, want = _load_mask(name)
    k = p["k"]
    got = np.array([[A.chunk_visible(i // k, j // k, p["W"])
                     for j in range(p["T"])] for i in range(p["T"])])
    assert (got == want).all()


def test_token_mask_expands_frames():
    m = A.token_mask(4, 3, 2, -1)
    assert m.shape == (12, 12)
    for i in range(12):
        for j in range(12):
            assert m[i, j] == ((j // 3) // 2 <= (i // 3) // 2)


# ---------------------------------------------------------- brute force
BRUTE_CASES = [
    # (B, H, d, N, k, chunks, last_frames, W)
    (1, 1, 4, 2, 2, 3, 0, -1),
    (1, 2, 8, 3, 1, 4, 0, -1),
    (2, 1, 4, 4, 3, 2, 1, 1),
    (1, 1, 8, 2, 2, 4, 0, 0),
    (1, 2, 4, 1, 3, 3, 2, 2),
    (1, 1, 6, 5, 1, 5, 0, 1),
]


@pytest.mark.parametrize("case", BRUTE_CASES)
def test_blockcausal_matches_bruteforce(case):
    B, H, d, N, k, chunks, last, W = case
    frames = [k] * chunks
    if last:
        frames[-1] = last
    L = sum(frames) * N
    q = _rand((B, L, H, d), 1)
    kk = _rand((B, L, H, d), 2)
    v = _rand((B, L, H, d), 3)
    scale = d ** -0.5
    o, lse = A.blockcausal_attention(q, kk, v, N, k, W, scale)
    ob, lb = A.bruteforce_attention(q, kk, v, N, k, W, scale)
    assert np.abs(o - ob).max() <= 1e-12
    assert np.abs(lse - lb).max() <= 1e-12


# ------------------------------------------- reductions to library routines
def test_single_chunk_is_full_bidirectional_attention():
    N, k, d = 16, 3, 32
    L = 2 * N  # two frames, one (partial) chunk
    q, kk, v = (_rand((1, L, 1, d), s) for s in (4, 5, 6))
    o, _ = A.blockcausal_attention(q, kk, v, N, k, -1, d ** -0.5)
    ref = _sdpa(q[0, :, 0], kk[0, :, 0], v[0, :, 0], d ** -0.5)
    assert np.abs(o[0, :, 0] - ref).max() <= 1e-12


def test_token_causal_when_one_token_one_frame_per_chunk():
    L, d = 40, 16
    q, kk, v = (_rand((1, L, 1, d), s) for s in (7, 8, 9))
    o, _ = A.blockcausal_attention(q, kk, v, 1, 1, -1, d ** -0.5)
    ref = _sdpa(q[0, :, 0], kk[0, :, 0], v[0, :, 0], d ** -0.5, causal=True)
    assert np.abs(o[0, :, 0] - ref).max() <= 1e-12


def test_frame_causal_when_chunk_is_one_frame():
    N, T, d = 5, 6, 16
    L = N * T
    q, kk, v = (_rand((1, L, 1, d), s) for s in (10, 11, 12))
    o, _ = A.blockcausal_attention(q, kk, v, N, 1, -1, d ** -0.5)
    idx = np.arange(L)
    frame_causal = (idx[None, :] // N) <= (idx[:, None] // N)
    ref = _sdpa(q[0, :, 0], kk[0, :, 0], v[0, :, 0], d ** -0.5,
                mask=frame_causal)
    assert np.abs(o[0, :, 0] - ref).max() <= 1e-12


def test_window_zero_is_independent_chunks():
    N, k, chunks, d = 4, 2, 3, 8
    L = N * k * chunks
    q, kk, v = (_rand((1, L, 1, d), s) for s in (13, 14, 15))
    o, _ = A.blockcausal_attention(q, kk, v, N, k, 0, d ** -0.5)
    span = N * k
    for c in range(chunks):
        s = slice(c * span, (c + 1) * span)
        ref = _sdpa(q[0, s, 0], kk[0, s, 0], v[0, s, 0], d ** -0.5)
        assert np.abs(o[0, s, 0] - ref).max() <= 1e-12


def test_lse_is_logsumexp_of_masked_scores():
    N, k, W, d = 3, 2, 1, 8
    L = N * 8
    q, kk = _rand((1, L, 1, d), 16), _rand((1, L, 1, d), 17)
    v = _rand((1, L, 1, d), 18)
    _, lse = A.blockcausal_attention(q, kk, v, N, k, W, 0.3)
    s = torch.from_numpy(0.3 * q[0, :, 0] @ kk[0, :, 0].T)
    mask = torch.from_numpy(A.token_mask(L // N, N, k, W))
    ref = torch.logsumexp(s.masked_fill(~mask, -math.inf), dim=1).numpy()
    assert np.abs(lse[0, 0] - ref).max() <= 1e-12


# --------------------------------------------------------------- closed forms
def test_zero_queries_average_the_visible_values():
    N, k, W, d, chunks = 3, 2, 1, 4, 4
    L = N * k * chunks
    q = np.zeros((1, L, 2, d))
    kk = _rand((1, L, 2, d), 19)
    v = _rand((1, L, 2, d), 20)
    o, lse = A.blockcausal_attention(q, kk, v, N, k, W, 0.125)
    for i in range(L):
        ci = i // (N * k)
        lo = max(0, ci - W) * N * k
        hi = (ci + 1) * N * k
        assert np.abs(o[0, i] - v[0, lo:hi].mean(axis=0)).max() <= 1e-12
        assert abs(lse[0, 0, i] - math.log(hi - lo)) <= 1e-12


def test_unit_values_give_unit_output():
    N, k, d = 4, 3, 8
    L = N * 7
    q, kk = _rand((2, L, 1, d), 21, 3.0), _rand((2, L, 1, d), 22, 3.0)
    v = np.ones((2, L, 1, d))
    o, _ = A.blockcausal_attention(q, kk, v, N, k, 2, d ** -0.5)
    assert np.abs(o - 1.0).max() <= 1e-12


def test_visible_pair_count_closed_form():
    # unbounded window, C full chunks of k*N tokens: sum_c (kN)(c+1)(kN)
    N, k, C = 3, 2, 5
    mask = A.token_mask(C * k, N, k, -1)
    closed = (k * N) ** 2 * C * (C + 1) // 2
    assert mask.sum() == closed
    assert sum(A.visible_pairs_per_chunk([k] * C, N, -1)) == closed
    # window W, ragged last chunk: count against the explicit mask
    frames = [3, 3, 3, 3, 1]
    mask = A.token_mask(sum(frames), N, 3, 1)
    assert mask.sum() == sum(A.visible_pairs_per_chunk(frames, N, 1))


def test_attention_cost_grows_linearly_with_a_window():
    # Sec. 3.1: with fixed k and W, attention cost is O(T k), not O(T^2)
    N, k, W = 2, 3, 1
    per = [sum(A.visible_pairs_per_chunk([k] * C, N, W)) for C in (10, 20, 40)]
    assert per[2] - per[1] == 2 * (per[1] - per[0])


# ------------------------------------------------------------------ invariants
def test_softmax_rows_sum_to_one():
    N, k, W, d = 4, 2, 1, 8
    L = N * 6
    q, kk = _rand((1, L, 1, d), 23, 2.0), _rand((1, L, 1, d), 24, 2.0)
    mask = A.token_mask(L // N, N, k, W)
    p = A.softmax_rows(q[0, :, 0], kk[0, :, 0], d ** -0.5, mask)
    assert np.abs(p.sum(axis=1) - 1.0).max() <= 1e-12
    assert (p[~mask] == 0).all()


@pytest.mark.parametrize("W,frames", [(-1, [2, 2, 2, 2]), (1, [3, 3, 3, 1]),
                                      (0, [2, 2, 1]), (2, [1, 1, 1, 1, 1])])
def test_streamed_equals_oneshot(W, frames):
    N, d, H, B = 3, 8, 2, 2
    k = max(frames)
    qs, ks, vs = [], [], []
    for c, f in enumerate(frames):
        qs.append(_rand((B, f * N, H, d), 100 + c))
        ks.append(_rand((B, f * N, H, d), 200 + c))
        vs.append(_rand((B, f * N, H, d), 300 + c))
    out = A.streamed_attention(qs, ks, vs, W, d ** -0.5)
    o1, l1 = A.blockcausal_attention(np.concatenate(qs, 1),
                                     np.concatenate(ks, 1),
                                     np.concatenate(vs, 1), N, k, W,
                                     d ** -0.5)
    o2 = np.concatenate([o for o, _ in out], 1)
    l2 = np.concatenate([l for _, l in out], 2)
    assert np.abs(o1 - o2).max() <= 1e-12
    assert np.abs(l1 - l2).max() <= 1e-12


def test_key_order_inside_the_visible_set_does_not_matter():
    q = _rand((1, 6, 2, 8), 25)
    kk, v = _rand((1, 20, 2, 8), 26), _rand((1, 20, 2, 8), 27)
    perm = np.random.default_rng(0).permutation(20)
    o1, l1 = A.chunk_attention(q, kk, v, 0.35)
    o2, l2 = A.chunk_attention(q, kk[:, perm], v[:, perm], 0.35)
    assert np.abs(o1 - o2).max() <= 1e-12
    assert np.abs(l1 - l2).max() <= 1e-12


def test_row_subset_equals_full():
    N, k, W, d = 3, 2, 1, 8
    L = N * 10
    q, kk, v = (_rand((1, L, 2, d), s) for s in (28, 29, 30))
    rows = [0, 5, 7, 17, L - 1]
    o, lse = A.blockcausal_attention(q, kk, v, N, k, W, 0.4)
    os_, ls = A.blockcausal_attention(q, kk, v, N, k, W, 0.4, rows=rows,
                                      row_block=2)
    # identical up to BLAS summation order
    assert np.abs(o[:, rows] - os_).max() <= 1e-14
    assert np.abs(lse[:, :, rows] - ls).max() <= 1e-14


@pytest.mark.parametrize("W", [0, 1, 4])
def test_list_cache_stays_bounded(W):
    N, k = 3, 2
    cache = A.ListKVCache(W)
    for c in range(12):
        kv = np.zeros((1, k * N, 1, 2))
        cache.append(c, kv, kv)
        assert cache.tokens() <= (W + 1) * k * N
    assert cache.tokens() == (W + 1) * k * N


# --------------------------------------------------------- KV cache oracle
def test_ring_cache_matches_elementwise_placement():
    B, H, d, N, k, W = 2, 3, 4, 2, 2, 1
    rc = KC.RingCache(B, H, d, N, k, W, 0, fill=7)
    rng = np.random.default_rng(1)
    history = []
    for c in range(5):
        f = 1 if c == 4 else k
        kb = rng.integers(0, 65536, (B, f * N, H, d), dtype=np.uint16)
        vb = rng.integers(0, 65536, (B, f * N, H, d), dtype=np.uint16)
        rc.append(kb, vb)
        history.append((kb, vb))
    S = W + 1
    for b in range(B):
        for h in range(H):
            for tok in range(S * k * N):
                slot, t = divmod(tok, k * N)
                # the newest chunk written to this slot that covers token t
                want_k = want_v = 7
                for c, (kb, vb) in enumerate(history):
                    if c % S == slot and t < kb.shape[1]:
                        want_k, want_v = kb[b, t, h], vb[b, t, h]
                assert (rc.k[b, h, tok] == want_k).all()
                assert (rc.v[b, h, tok] == want_v).all()


# ------------------------------------------------------------ planted mistakes
def _pins_pass():
    """A compact run of the pins above; False when any of them fails."""
    try:
        for case in BRUTE_CASES[:3]:
            test_blockcausal_matches_bruteforce(case)
        test_single_chunk_is_full_bidirectional_attention()
        test_token_causal_when_one_token_one_frame_per_chunk()
        test_lse_is_logsumexp_of_masked_scores()
        test_zero_queries_average_the_visible_values()
        test_streamed_equals_oneshot(1, [3, 3, 3, 1])
    except AssertionError:
        return False
    return True


def _mutant_softmax_no_scale(q, k, v, scale, mask=None):
    return _ORIG_SOFTMAX(q, k, v, 1.0, mask)


def _mutant_softmax_values_are_keys(q, k, v, scale, mask=None):
    return _ORIG_SOFTMAX(q, k, k, scale, mask)


def _mutant_softmax_lse_drops_max(q, k, v, scale, mask=None):
    o, lse = _ORIG_SOFTMAX(q, k, v, scale, mask)
    s = scale * (q @ k.T)
    if mask is not None:
        s = np.where(mask, s, -np.inf)
    return o, lse - s.max(axis=1)


def _mutant_softmax_transposed_scores(q, k, v, scale, mask=None):
    if q.shape[0] != k.shape[0]:
        return _ORIG_SOFTMAX(q, k, v, scale, mask)
    s = scale * (k @ q.T)
    if mask is not None:
        s = np.where(mask, s, -np.inf)
    m = s.max(axis=1, keepdims=True)
    p = np.exp(s - m)
    return (p @ v) / p.sum(1, keepdims=True), m[:, 0] + np.log(p.sum(1))


def _mutant_visible_window_off_by_one(qc, kc, W):
    d = qc - kc
    return d >= 0 and (W < 0 or d <= W + 1)


def _mutant_visible_future_chunk(qc, kc, W):
    d = qc - kc
    return d >= -1 and (W < 0 or d <= W)


_ORIG_SOFTMAX = A.softmax_attention


@pytest.mark.parametrize("target,mutant", [
    ("softmax_attention", _mutant_softmax_no_scale),
    ("softmax_attention", _mutant_softmax_values_are_keys),
    ("softmax_attention", _mutant_softmax_lse_drops_max),
    ("softmax_attention", _mutant_softmax_transposed_scores),
    ("chunk_visible", _mutant_visible_window_off_by_one),
    ("chunk_visible", _mutant_visible_future_chunk),
])
def test_planted_oracle_mistake_fails_a_pin(monkeypatch, target, mutant):
    assert _pins_pass()
    monkeypatch.setattr(A, target, mutant)
    assert not _pins_pass()
