"""Seeded synthetic token streams for chunk-wise causal attention.

This module only describes workloads and draws their inputs; it holds none of
the attention arithmetic, so both the CUDA path and the CPU oracle can be fed
from it without sharing any of the method's code.

A workload is a streaming video in latent space (Sec. 3.1, "Chunk-wise causal
attention"): T latent frames of N tokens each, grouped into chunks of k frames,
with B batch entries (videos or spatial tiles), H heads and head dim d. Chunk c
holds frames [c*k, c*k + f_c), where f_c = k except for a ragged last chunk.

Inputs per chunk are drawn, in chunk order, from one CPU generator seeded with
the workload's seed: Q_c, then K_c, then V_c, each [B, f_c*N, H, d] float32
N(0, 1).  For a "peaked" workload two more draws follow per chunk, a [B, f_c*N]
U[0.5, 2] factor for the Q rows and another for the K rows (one factor per
batch entry and token, shared by all heads), applied in float32.  The result is
rounded to bfloat16 (round to nearest even); both sides consume those bytes.
"""
from __future__ import annotations

import dataclasses
from typing import Iterator, Tuple

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    heads: int
    head_dim: int
    tokens_per_frame: int
    frames_per_chunk: int
    num_chunks: int
    window_chunks: int = -1       # -1: every earlier chunk is visible
    last_chunk_frames: int = 0    # 0: the last chunk is full (k frames)
    seed: int = 0
    peaked: bool = False

    @property
    def softmax_scale(self) -> float:
        return self.head_dim ** -0.5

    def frames_in_chunk(self, c: int) -> int:
        if c == self.num_chunks - 1 and self.last_chunk_frames:
            return self.last_chunk_frames
        return self.frames_per_chunk

    @property
    def num_frames(self) -> int:
        return sum(self.frames_in_chunk(c) for c in range(self.num_chunks))

    @property
    def num_tokens(self) -> int:
        return self.num_frames * self.tokens_per_frame

    @property
    def max_chunks(self) -> int:
        """Chunks the cache must hold: all of them when unbounded."""
        return self.num_chunks if self.window_chunks < 0 else 0

    def chunk_shape(self, c: int) -> Tuple[int, int, int, int]:
        return (self.batch, self.frames_in_chunk(c) * self.tokens_per_frame,
                self.heads, self.head_dim)


# The five synthetic stand-ins for the paper's streaming video workloads.
# Token grids follow a 16x spatial reduction of the pixel frame (no patch size
# is stated in the paper); frames are latent frames.
TINY = Workload("tiny", 1, 2, 64, 64, 2, 3, seed=0)
W480P = Workload("480p", 1, 12, 128, 30 * 53, 2, 8, seed=1)
W720P_PEAKED = Workload("720p-peaked", 1, 12, 128, 45 * 80, 2, 8, seed=2,
                        peaked=True)
W1080P = Workload("1080p", 1, 12, 128, 68 * 120, 2, 15, seed=3)
W1080P_WINDOWED = Workload("1080p-windowed", 1, 24, 128, 68 * 120, 3, 40,
                           window_chunks=4, last_chunk_frames=1, seed=4)

# The paper's own inference shape (Sec. 4.1 "Inference"): chunks of k = 3
# latent frames, each chunk sees itself and one predecessor (Eq. 1, W = 1),
# and the frame is cut into overlapping 64 x 64 latent tiles, one DiT pass per
# tile, so the tiles of a frame batch on B.  A 1080p frame (68 x 120 latent)
# with tile stride 32 gives 2 x 3 = 6 tiles; 30 latent frames as above.  The DiT patch size is not
# stated: a 2 x 2 patch gives 32 x 32 tokens per tile frame, none gives
# 64 x 64.  Heads and head dim follow a 3072-wide DiT with 24 heads of 128.
PAPER_TILES_32 = Workload("paper-tiles-32x32", 6, 24, 128, 32 * 32, 3, 10,
                          window_chunks=1, seed=5)
PAPER_TILES_64 = Workload("paper-tiles-64x64", 6, 24, 128, 64 * 64, 3, 10,
                          window_chunks=1, seed=6)

# A training clip (Sec. 4.1: 45-frame clips at 1024 x 1024): 12 latent frames
# (4x temporal, 16x spatial reduction, 2 x 2 patch -> 32 x 32 tokens), chunks
# of 3 frames, one predecessor visible (Eq. 1), processed in one shot.
TRAIN_CLIP = Workload("train-1024-clip", 1, 24, 128, 32 * 32, 3, 4,
                      window_chunks=1, seed=7)

WORKLOADS = {w.name: w for w in
             (TINY, W480P, W720P_PEAKED, W1080P, W1080P_WINDOWED,
              PAPER_TILES_32, PAPER_TILES_64, TRAIN_CLIP)}


def chunk_stream(w: Workload, device: str = "cpu"
                 ) -> Iterator[Tuple[int, torch.Tensor, torch.Tensor,
                                 torch.Tensor]]:
    """Yield (c, Q_c, K_c, V_c) as bfloat16 tensors [B, f_c*N, H, d].

    With the default CPU device these are the seeded inputs that the CUDA
    path and the oracle share.  Another device draws with the same recipe
    from that device's generator (other values: for timing only)."""
    g = torch.Generator(device=device)
    g.manual_seed(w.seed)
    for c in range(w.num_chunks):
        shape = w.chunk_shape(c)
        kw = dict(generator=g, dtype=torch.float32, device=device)
        q = torch.randn(shape, **kw)
        k = torch.randn(shape, **kw)
        v = torch.randn(shape, **kw)
        if w.peaked:
            uq = torch.rand(shape[:2], **kw)
            uk = torch.rand(shape[:2], **kw)
            q = q * (0.5 + 1.5 * uq)[:, :, None, None]
            k = k * (0.5 + 1.5 * uk)[:, :, None, None]
        yield (c, q.to(torch.bfloat16), k.to(torch.bfloat16),
               v.to(torch.bfloat16))


def custom(name: str = "custom", **kw) -> Workload:
    """A workload with explicit sizes (used for small parity cases)."""
    base = dict(batch=1, heads=1, head_dim=64, tokens_per_frame=8,
                frames_per_chunk=2, num_chunks=2)
    base.update(kw)
    return Workload(name=name, **base)
