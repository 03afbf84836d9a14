"""CPU oracle for the streaming KV cache -- TEST INFRASTRUCTURE.

Only the tests, the smoke check and the benchmark's CPU-baseline leg may import
this module; the product path never does.

Streaming inference keeps the keys and values of the chunks that later queries
can still see (Sec. 3.1, last paragraph: KV caching, cache size O(k)).  With a
window of W chunks that is W + 1 chunks, so the cache is a ring of S = W + 1
chunk slots; with no window it holds every chunk (S = the chunk capacity).

Layout of the library's cache (a design choice of this implementation, which
the tests check bit for bit): K and V each [B, H, S * k * N, d] bfloat16,
head-major, chunk c in slot c mod S at token offset (c mod S) * k * N, its
f_c * N tokens in order.  Tokens of a slot past f_c * N keep whatever they held.
The arrays here are uint16 bit patterns, so the comparison is exact.
"""
from __future__ import annotations

import numpy as np


def num_slots(window: int, max_chunks: int) -> int:
    return window + 1 if window >= 0 else max_chunks


class RingCache:
    def __init__(self, batch: int, heads: int, head_dim: int,
                 tokens_per_frame: int, frames_per_chunk: int, window: int,
                 max_chunks: int, fill: int = 0):
        self.slots = num_slots(window, max_chunks)
        self.slot_tokens = frames_per_chunk * tokens_per_frame
        shape = (batch, heads, self.slots * self.slot_tokens, head_dim)
        self.k = np.full(shape, fill, dtype=np.uint16)
        self.v = np.full(shape, fill, dtype=np.uint16)
        self.next_chunk = 0

    def append(self, k_bits: np.ndarray, v_bits: np.ndarray) -> None:
        """k_bits, v_bits: uint16 [B, f*N, H, d] (token-major bit patterns)."""
        slot = self.next_chunk % self.slots
        t0 = slot * self.slot_tokens
        L = k_bits.shape[1]
        self.k[:, :, t0:t0 + L, :] = np.transpose(k_bits, (0, 2, 1, 3))
        self.v[:, :, t0:t0 + L, :] = np.transpose(v_bits, (0, 2, 1, 3))
        self.next_chunk += 1
