"""CPU oracle for FastVR chunk-wise causal attention -- TEST INFRASTRUCTURE.

Only the tests, the smoke check and the benchmark's CPU-baseline leg may import
this module.  The product path (the C-ABI library and its Python binding) never
calls it and shares no code with it.

Everything is plain NumPy in float64 on the exact bfloat16 input values.

What it computes (Sec. 3.1, "Chunk-wise causal attention", Eq. 1).  Latent
frames are grouped into non-overlapping chunks of k frames; the visibility mask
between a query frame i and a key frame j is M_ij = 1 iff floor(i/k) - floor(j/k)
is in {0, 1}.  The paper's mask keeps the current chunk and one predecessor; the
window W generalises the upper end of that set to {0, ..., W} (W = 1 is Eq. 1,
W < 0 means every earlier chunk).  Tokens are laid out frame after frame, N per
frame, so token t belongs to frame t // N.  The mask is applied inside softmax
self-attention in every layer (Sec. 3.1): for one head,

    s_j = scale * <q_i, k_j>  for visible j,  -inf otherwise
    o_i = sum_j exp(s_j - m) v_j / sum_j exp(s_j - m),  m = max_j s_j
    lse_i = m + ln sum_j exp(s_j - m)

During training the whole sequence is processed at once under M; during
inference chunks are processed one after the other with a KV cache (Sec. 3.1,
last paragraph).  `blockcausal_attention` is the first form and
`streamed_attention` the second; they must agree.

parity pins: every function here is pinned by tests/test_oracle.py against a
brute-force scalar loop, library attention (torch SDPA in float64) in the
special cases that reduce to it, closed forms and invariants.
"""
from __future__ import annotations

import math
from typing import List, Optional, Sequence, Tuple

import numpy as np


# --------------------------------------------------------------------------
# Visibility (Eq. 1, generalised to a window of W chunks)
# --------------------------------------------------------------------------
def chunk_visible(query_chunk: int, key_chunk: int, window: int) -> bool:
    """Eq. 1 at chunk granularity: the difference of chunk indices must lie in
    {0, ..., W} (W < 0: unbounded above)."""
    delta = query_chunk - key_chunk
    if delta < 0:
        return False
    return window < 0 or delta <= window


def frame_mask(num_frames: int, k: int, window: int) -> np.ndarray:
    """The T x T temporal mask M of Eq. 1 over latent frame indices."""
    i = np.arange(num_frames)[:, None] // k
    j = np.arange(num_frames)[None, :] // k
    delta = i - j
    ok = delta >= 0
    if window >= 0:
        ok &= delta <= window
    return ok


def token_mask(num_frames: int, tokens_per_frame: int, k: int,
               window: int) -> np.ndarray:
    """Eq. 1 expanded to tokens: token t lies in frame t // N."""
    fm = frame_mask(num_frames, k, window)
    return np.repeat(np.repeat(fm, tokens_per_frame, axis=0),
                     tokens_per_frame, axis=1)


def visible_chunks(c: int, window: int) -> List[int]:
    """Chunks whose keys chunk c's queries see (Eq. 1 with window W)."""
    lo = 0 if window < 0 else max(0, c - window)
    return list(range(lo, c + 1))


# --------------------------------------------------------------------------
# Softmax attention for one head (the plain definition)
# --------------------------------------------------------------------------
def softmax_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray,
                      scale: float, mask: Optional[np.ndarray] = None
                      ) -> Tuple[np.ndarray, np.ndarray]:
    """q [Lq, d], k [Lk, d], v [Lk, dv] float64; mask [Lq, Lk] bool or None.

    Returns (o [Lq, dv], lse [Lq]) with lse the natural-log sum of exp(s)."""
    s = scale * (q @ k.T)
    if mask is not None:
        s = np.where(mask, s, -np.inf)
    m = s.max(axis=1, keepdims=True)
    p = np.exp(s - m)
    l = p.sum(axis=1, keepdims=True)
    o = (p @ v) / l
    lse = m[:, 0] + np.log(l[:, 0])
    return o, lse


def softmax_rows(q: np.ndarray, k: np.ndarray, scale: float,
                 mask: Optional[np.ndarray] = None) -> np.ndarray:
    """The attention probabilities themselves (for the row-sum invariant)."""
    s = scale * (q @ k.T)
    if mask is not None:
        s = np.where(mask, s, -np.inf)
    p = np.exp(s - s.max(axis=1, keepdims=True))
    return p / p.sum(axis=1, keepdims=True)


# --------------------------------------------------------------------------
# Training form: the whole sequence at once under the mask
# --------------------------------------------------------------------------
def blockcausal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray,
                          tokens_per_frame: int, frames_per_chunk: int,
                          window: int, scale: float,
                          rows: Optional[Sequence[int]] = None,
                          row_block: int = 512
                          ) -> Tuple[np.ndarray, np.ndarray]:
    """One-shot chunk-causal attention over a whole token sequence.

    q, k, v: [B, L, H, d] (token-major) float64, L = T * N.
    rows: optional query-token indices to compute (all when None).
    Returns O [B, len(rows), H, d] and LSE [B, H, len(rows)].

    Query rows are processed in blocks of `row_block` so that memory stays
    bounded; rows are independent, so this does not change the result.  Keys
    after the last chunk of a block are invisible to every row of the block
    (Eq. 1 forbids negative chunk differences), so the explicit mask is built
    over the key prefix that ends there.
    """
    B, L, H, d = q.shape
    N, kf = tokens_per_frame, frames_per_chunk
    if L % N:
        raise ValueError("sequence length must be a whole number of frames")
    rows = np.arange(L) if rows is None else np.asarray(rows, dtype=np.int64)
    o = np.zeros((B, len(rows), H, v.shape[-1]))
    lse = np.zeros((B, H, len(rows)))
    key_chunk = (np.arange(L) // N) // kf
    for r0 in range(0, len(rows), row_block):
        rb = rows[r0:r0 + row_block]
        qc = (rb // N) // kf
        key_end = (int(qc.max()) + 1) * kf * N
        key_end = min(key_end, L)
        delta = qc[:, None] - key_chunk[None, :key_end]
        mask = delta >= 0
        if window >= 0:
            mask &= delta <= window
        for b in range(B):
            for h in range(H):
                ob, lb = softmax_attention(q[b, rb, h], k[b, :key_end, h],
                                           v[b, :key_end, h], scale, mask)
                o[b, r0:r0 + len(rb), h] = ob
                lse[b, h, r0:r0 + len(rb)] = lb
    return o, lse


# --------------------------------------------------------------------------
# Inference form: chunk by chunk with an explicit KV cache
# --------------------------------------------------------------------------
class ListKVCache:
    """The streaming KV cache of Sec. 3.1 as a plain list of chunks.

    It keeps only the chunks a future query can still see: with window W that
    is the newest W + 1 chunks, so its size is O(k) tokens per head whatever
    the video length (Sec. 3.1)."""

    def __init__(self, window: int):
        self.window = window
        self.chunks: List[Tuple[int, np.ndarray, np.ndarray]] = []

    def append(self, c: int, k: np.ndarray, v: np.ndarray) -> None:
        self.chunks.append((c, k, v))
        if self.window >= 0:
            self.chunks = [e for e in self.chunks
                           if chunk_visible(c, e[0], self.window)]

    def tokens(self) -> int:
        return sum(e[1].shape[1] for e in self.chunks)

    def keys_values(self, c: int) -> Tuple[np.ndarray, np.ndarray]:
        vis = [e for e in self.chunks if chunk_visible(c, e[0], self.window)]
        return (np.concatenate([e[1] for e in vis], axis=1),
                np.concatenate([e[2] for e in vis], axis=1))


def chunk_attention(q_c: np.ndarray, k_vis: np.ndarray, v_vis: np.ndarray,
                    scale: float, rows: Optional[Sequence[int]] = None
                    ) -> Tuple[np.ndarray, np.ndarray]:
    """Attention of one chunk's queries to its visible keys.

    q_c [B, Lq, H, d]; k_vis, v_vis [B, Lk, H, d] (every key visible: the mask
    acts at chunk granularity and q_c is one chunk).  Returns O [B, rows, H, d]
    and LSE [B, H, rows]."""
    B, Lq, H, _ = q_c.shape
    rows = np.arange(Lq) if rows is None else np.asarray(rows, dtype=np.int64)
    o = np.zeros((B, len(rows), H, v_vis.shape[-1]))
    lse = np.zeros((B, H, len(rows)))
    for b in range(B):
        for h in range(H):
            ob, lb = softmax_attention(q_c[b, rows, h], k_vis[b, :, h],
                                       v_vis[b, :, h], scale)
            o[b, :, h] = ob
            lse[b, h] = lb
    return o, lse


def streamed_attention(q_chunks: Sequence[np.ndarray],
                       k_chunks: Sequence[np.ndarray],
                       v_chunks: Sequence[np.ndarray],
                       window: int, scale: float
                       ) -> List[Tuple[np.ndarray, np.ndarray]]:
    """Streaming inference (Sec. 3.1): for c = 0, 1, ... append chunk c's K/V
    to the cache, then attend chunk c's queries to the cached chunks it sees."""
    cache = ListKVCache(window)
    out = []
    for c, (qc, kc, vc) in enumerate(zip(q_chunks, k_chunks, v_chunks)):
        cache.append(c, kc, vc)
        kv, vv = cache.keys_values(c)
        out.append(chunk_attention(qc, kv, vv, scale))
    return out


# --------------------------------------------------------------------------
# Brute force: scalar loops, tiny inputs only
# --------------------------------------------------------------------------
def bruteforce_attention(q, k, v, tokens_per_frame: int, frames_per_chunk: int,
                         window: int, scale: float):
    """Pure-Python triple loop over (b, h, i) with math.exp; [B, L, H, d]."""
    B, L, H, d = q.shape
    dv = v.shape[-1]
    o = np.zeros((B, L, H, dv))
    lse = np.zeros((B, H, L))
    for b in range(B):
        for h in range(H):
            for i in range(L):
                ci = (i // tokens_per_frame) // frames_per_chunk
                scores = []
                for j in range(L):
                    cj = (j // tokens_per_frame) // frames_per_chunk
                    if not chunk_visible(ci, cj, window):
                        continue
                    dot = 0.0
                    for t in range(d):
                        dot += float(q[b, i, h, t]) * float(k[b, j, h, t])
                    scores.append((j, scale * dot))
                m = max(s for _, s in scores)
                total = 0.0
                acc = [0.0] * dv
                for j, s in scores:
                    w = math.exp(s - m)
                    total += w
                    for t in range(dv):
                        acc[t] += w * float(v[b, j, h, t])
                for t in range(dv):
                    o[b, i, h, t] = acc[t] / total
                lse[b, h, i] = m + math.log(total)
    return o, lse


# --------------------------------------------------------------------------
# Cost accounting (Sec. 3.1: O(Tk) attention cost, O(k) cache)
# --------------------------------------------------------------------------
def visible_pairs_per_chunk(frames: Sequence[int], tokens_per_frame: int,
                            window: int) -> List[int]:
    """Number of visible (query, key) token pairs of each chunk, counted from
    the chunk list: Lq_c * sum of the tokens of the chunks c sees."""
    out = []
    for c, f in enumerate(frames):
        lk = sum(frames[j] for j in visible_chunks(c, window))
        out.append(f * tokens_per_frame * lk * tokens_per_frame)
    return out


# --------------------------------------------------------------------------
# Backward of the one-shot form (gradients for training under the mask)
# --------------------------------------------------------------------------
def blockcausal_attention_bwd(q: np.ndarray, k: np.ndarray, v: np.ndarray,
                              do: np.ndarray, tokens_per_frame: int,
                              frames_per_chunk: int, window: int,
                              scale: float):
    """Gradients of the one-shot chunk-causal attention (training form,
    Sec. 3.1: the whole sequence under M) with respect to q, k and v, given
    the output gradient do; all [B, L, H, d] float64.

    With s_ij = scale <q_i, k_j> on visible pairs, p_ij = softmax_j(s_ij) and
    o_i = sum_j p_ij v_j, the chain rule gives
        dv_j = sum_i p_ij do_i
        dp_ij = <do_i, v_j>
        ds_ij = p_ij (dp_ij - sum_j' p_ij' dp_ij')
        dq_i = scale sum_j ds_ij k_j,   dk_j = scale sum_i ds_ij q_i.
    """
    B, L, H, d = q.shape
    mask = token_mask(L // tokens_per_frame, tokens_per_frame,
                      frames_per_chunk, window)
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    for b in range(B):
        for h in range(H):
            p = softmax_rows(q[b, :, h], k[b, :, h], scale, mask)
            dv[b, :, h] = p.T @ do[b, :, h]
            dp = do[b, :, h] @ v[b, :, h].T
            ds = p * (dp - (p * dp).sum(axis=1, keepdims=True))
            dq[b, :, h] = scale * ds @ k[b, :, h]
            dk[b, :, h] = scale * ds.T @ q[b, :, h]
    return dq, dk, dv
