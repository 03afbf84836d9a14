// Backward of one-shot chunk-causal attention (the training form of
// Sec. 3.1: the whole latent sequence at once under the mask of Eq. 1),
// with tcgen05 tensor cores, TMEM accumulators and TMA-staged tiles.
//
// With s_ij = scale <q_i, k_j> on visible pairs, P = softmax(S) (row i,
// recomputed from the forward's log-sum-exp), dO the output gradient and
// D_i = <dO_i, O_i>:
//     dV = P^T dO,  dP = dO V^T,  dS = P o (dP - D),
//     dQ = scale dS K,  dK = scale dS^T Q.
// Three kernels, no atomics:
//   delta_kernel  D_i = <dO_i, O_i> (fp32) into the caller's scratch, one
//                 block per 64 tokens of one (batch, head);
//   dkdv_kernel   one CTA per 128-key tile: for every query tile that sees it
//                 S^T = K Q^T and dP^T = V dO^T (SMEM x SMEM -> TMEM); P^T in
//                 bf16 over S^T (and in registers); dV += P^T dO, then the
//                 next tile's S^T, while dS^T is written over dP^T; then
//                 dK += dS^T Q (A from TMEM, B = dO or Q read as an MN-major
//                 operand) and the next tile's dP^T;
//   dq_kernel     one CTA per 128-query tile: for every visible key tile
//                 S = Q K^T and dP = dO V^T; P in registers (then the next
//                 tile's S and dP are issued, dP into the other of two
//                 buffers), dS over dP, dQ += dS K.
// Visibility is Eq. 1 with window W per (query row, key): a key of chunk c'
// is seen by queries of chunks c' .. c' + W, a query of chunk c sees keys of
// chunks c - W .. c; only tiles inside a CTA's visible range are loaded and
// columns outside each row's range are masked (only tiles that cross a chunk
// edge take the masked form of the exponential step).
// CTAs run in head-major order, so the CTAs resident at one time stream the
// tiles of one or two heads, which stay in L2 (loads carry evict_last for
// the streamed tiles, evict_first for the resident ones); each CTA writes
// its output tile through shared memory with tiled TMA stores.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <string.h>

#include <algorithm>
#include <mutex>

#include "fastvr_internal.h"
#include "sm100_ptx.cuh"

namespace fastvr {
namespace {

using namespace sm100;

constexpr int kT = 128;           // tile rows (TMEM lanes) and tile columns
constexpr int kBox = 128 * 128;   // one TMA box: 128 rows x 64 bf16 (bytes)
constexpr int kMaxStages = 3;     // deepest streamed ring
constexpr int kStages1 = 2;       // ring 1 depth (ring 0: per kernel)
constexpr int kDkdvS0 = 3;        // dK/dV ring 0 (Q)
constexpr int kDqS0 = 3;          // dQ ring 0 (K): loads one step earlier
constexpr int kThreads = 384;     // 8 compute warps, producer, MMA issuer,
                                  // relay, row-vector loader (dK/dV)
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;
constexpr int kRelayWarp = 10;
constexpr int kVecWarp = 11;
// Named (hardware) barriers of the hand-offs to the MMA warp: P stored and
// dS stored (the eight compute warps arrive, the MMA warp syncs), and one
// per stage of each streamed ring (the relay warp arrives once the stage's
// TMA loads have landed, the MMA warp syncs).  An mbarrier poll is a
// shared-memory access that waits ~200 clk behind queued SMEM x SMEM MMAs;
// a named barrier whose arrivals are in costs the MMA warp next to nothing.
constexpr int kBarP = 1;
constexpr int kBarDS = 2;
constexpr int kBarRing0 = 3;  // + stage, up to kMaxStages
constexpr int kBarRing1 = 6;  // + stage, up to kStages1
constexpr int kBarStaged = 8;  // the compute warps' output tiles are staged
constexpr int kComputeHandoff = 9 * 32;
constexpr int kRelayHandoff = 2 * 32;
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitLimitNs = 4000000000ull;

struct BwdParams {
  CUtensorMap q_map, k_map, v_map, do_map;  // {d, L, H, B} token-major
  CUtensorMap dq_map, dk_map, dv_map;       // the outputs, the same form
  const float* lse2;   // -(forward LSE in log2 units) [B*H, Lpad] (scratch)
  const float* delta;  // -D [B*H, Lpad] (scratch); padding tokens hold 0
  uint16_t* dq;        // bf16 [B, L, H, d]
  uint16_t* dk;
  uint16_t* dv;
  int32_t seq_tokens, heads, batch, chunk_tokens, window, tiles, padded;
  float scale, scale_log2;
  int* status;             // device status word (timeouts) or null
  int32_t inject_stall;    // test hook: the MMA warp waits on o_full first
  uint64_t wait_limit_ns;  // 0 = kWaitLimitNs
};

struct BwdShared {
  uint64_t fixed_full;                 // the CTA's resident operands
  // Two streamed rings with their own barriers, [ring][stage]: ring 0 holds
  // the tile read last in a step (dq: K, read by dQ; dkdv: Q and the row
  // vectors, read by dK), ring 1 the other (dq: V, last read by dP; dkdv:
  // dO, last read by dV), so a ring-1 slot is refilled as soon as its last
  // reader has run instead of waiting for the end of the step.
  uint64_t full[2][kMaxStages], empty[2][kMaxStages];
  // dp_ready[1]: the dQ kernel's second dP buffer (one barrier per buffer,
  // so a barrier never completes a second phase before its waiters saw the
  // first)
  uint64_t s_ready, dp_ready[2], o_full, drain;
  // dK/dV: the two slots of -log2 LSE and -D slices (loaded by the
  // row-vector warp, released by the compute warps after dS)
  uint64_t vec_full[2], vec_empty[2];
  uint32_t tmem_base;
  int abort;
  int* status;
  uint64_t wait_limit_ns;
};

// Shared memory of the dQ kernel: the two fixed operands, ring 0 (kS0
// stages), ring 1 (kStages1 stages), then the barriers; the dynamic base is
// rounded up to 1024 bytes (128-byte-swizzled tiles), which the size allows
// for.
template <int D, int S0>
struct BwdLayout {
  static_assert(S0 >= 2 && S0 <= kMaxStages, "ring 0 depth");
  static constexpr int kS0 = S0;
  static constexpr int kNB = D / 64;
  __host__ __device__ static constexpr int fixed(int which, int bx) {
    return (which * kNB + bx) * kBox;
  }
  __host__ __device__ static constexpr int ring(int st, int which, int bx) {
    return ((2 + (which ? kS0 + st : st)) * kNB + bx) * kBox;
  }
  static constexpr int shared_off = (2 + kS0 + kStages1) * kNB * kBox;
  static constexpr int bytes =
      shared_off + ((int)sizeof(BwdShared) + 15) / 16 * 16 + 1024 + 64;
};

// Shared memory of the dK/dV kernel: a 3 KB front region (the barriers at 0,
// the two slots of row vectors from 1024: slot sl holds 128 -log2 LSE values
// then 128 -D values), then the two fixed operands, the three-stage Q ring
// and the two-stage dO ring.  That is 227 KB exactly at d = 128, with no room
// left to round the base up: the kernel requires (and checks) that the
// dynamic shared memory starts 1024-byte aligned.
template <int D>
struct DkdvLayout {
  static constexpr int kS0 = kDkdvS0;
  static constexpr int kNB = D / 64;
  static constexpr int kFrontBytes = 3072;
  static constexpr int shared_off = 0;
  __host__ __device__ static constexpr int vec(int slot, int which) {
    return 1024 + (slot * 2 + which) * kT * (int)sizeof(float);
  }
  __host__ __device__ static constexpr int fixed(int which, int bx) {
    return kFrontBytes + (which * kNB + bx) * kBox;
  }
  __host__ __device__ static constexpr int ring(int st, int which, int bx) {
    return kFrontBytes + ((2 + (which ? kS0 + st : st)) * kNB + bx) * kBox;
  }
  static constexpr int bytes = kFrontBytes + (2 + kS0 + kStages1) * kNB * kBox;
};
static_assert(sizeof(BwdShared) <= 1024, "barriers fit the front region");
static_assert(DkdvLayout<128>::vec(1, 1) + 128 * 4 <= DkdvLayout<128>::kFrontBytes,
              "row-vector slots fit the front region");

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity,
                                         BwdShared* S) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*reinterpret_cast<volatile int*>(&S->abort)) return false;
    if (global_timer_ns() - t0 > S->wait_limit_ns) {
      *reinterpret_cast<volatile int*>(&S->abort) = 1;
      if (S->status != nullptr) atomicExch(S->status, kDevTimeout);
      return false;
    }
  }
}

// Warp-wide waits (the MMA warp and the compute warps): every lane polls and
// each decision (phase complete, abort seen, time limit passed) is a warp
// vote, so the warp never diverges and reaches the elected MMA instructions
// and the .sync.aligned TMEM loads converged.  A phase that has already
// completed costs one try_wait and one vote.
__device__ __forceinline__ bool wait_bar_warp(uint64_t* bar, uint32_t parity,
                                              BwdShared* S) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
    const bool aborted = *reinterpret_cast<volatile int*>(&S->abort) != 0;
    const bool late = global_timer_ns() - t0 > S->wait_limit_ns;
    if (__any_sync(0xffffffffu, aborted)) return false;
    if (__any_sync(0xffffffffu, late)) {
      if ((threadIdx.x & 31) == 0) {
        *reinterpret_cast<volatile int*>(&S->abort) = 1;
        if (S->status != nullptr) atomicExch(S->status, kDevTimeout);
      }
      __syncwarp();
      return false;
    }
  }
}

__device__ __forceinline__ void compute_arrive(int id) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "n"(kComputeHandoff) : "memory");
}
__device__ __forceinline__ void compute_sync(int id) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "n"(kComputeHandoff) : "memory");
}
// All eight compute warps (256 threads), and no other warp.
__device__ __forceinline__ void compute_only_sync(int id) {
  asm volatile("bar.sync %0, 256;" ::"r"(id) : "memory");
}
__device__ __forceinline__ void relay_arrive(int id) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "n"(kRelayHandoff) : "memory");
}
__device__ __forceinline__ void relay_sync(int id) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "n"(kRelayHandoff) : "memory");
}

// The relay warp observes each step's two streamed tiles (ring 0, then
// ring 1, the order in which the MMA warp needs them) and hands each stage
// over through its named barrier.  A stage's barrier cannot be arrived at
// twice before the MMA warp has synced on it: the producer refills a stage
// only after the MMAs that read it.  Named barriers have no time limit, so
// after a failed wait the relay still makes the remaining arrivals (the
// MMA warp then computes on undefined data; the failure is recorded).
template <int kS0>
__device__ void bwd_relay(BwdShared* S, int n) {
  int a0 = 0, a1 = 0;
  bool ok = true;
  for (int j = 0; ok && j < n; ++j) {
    if (!(ok = wait_bar_warp(&S->full[0][j % kS0], (j / kS0) & 1, S))) break;
    relay_arrive(kBarRing0 + j % kS0);
    ++a0;
    if (!(ok = wait_bar_warp(&S->full[1][j % kStages1], (j / kStages1) & 1, S)))
      break;
    relay_arrive(kBarRing1 + j % kStages1);
    ++a1;
  }
  for (; a0 < n; ++a0) relay_arrive(kBarRing0 + a0 % kS0);
  for (; a1 < n; ++a1) relay_arrive(kBarRing1 + a1 % kStages1);
}

__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity))
    if (global_timer_ns() - t0 > kWaitLimitNs) return;
}

// Row of the padded [B*H, Lpad] scratch vectors.
__device__ __forceinline__ int bh_row(const BwdParams& p, int b, int h) {
  return b * p.heads + h;
}

// Visible query tokens of a key in chunk c (Eq. 1 read from the key side).
__device__ __forceinline__ void key_sees(const BwdParams& p, int key, int& lo,
                                         int& hi) {
  if (key >= p.seq_tokens) {
    lo = hi = 0;
    return;
  }
  const int c = key / p.chunk_tokens;
  lo = c * p.chunk_tokens;
  hi = p.window < 0 ? p.seq_tokens
                    : min((c + p.window + 1) * p.chunk_tokens, p.seq_tokens);
}

// Visible key tokens of a query in chunk c.
__device__ __forceinline__ void query_sees(const BwdParams& p, int row, int& lo,
                                           int& hi) {
  const int c = min(row, p.seq_tokens - 1) / p.chunk_tokens;
  lo = p.window < 0 ? 0 : max(0, c - p.window) * p.chunk_tokens;
  hi = min((c + 1) * p.chunk_tokens, p.seq_tokens);
}

// Common CTA prologue: TMEM (MMA warp) and barriers (producer thread).
__device__ __forceinline__ uint32_t bwd_setup(BwdShared* S,
                                              const BwdParams& p) {
  const int warp = threadIdx.x / 32;
  if (warp == kMmaWarp) {
    tmem_alloc(&S->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (threadIdx.x == kProducerWarp * 32) {
    mbar_init(&S->fixed_full, 1);
    for (int r = 0; r < 2; ++r)
      for (int s = 0; s < kMaxStages; ++s) {
        mbar_init(&S->full[r][s], 1);
        mbar_init(&S->empty[r][s], 1);
      }
    mbar_init(&S->s_ready, 1);
    mbar_init(&S->dp_ready[0], 1);
    mbar_init(&S->dp_ready[1], 1);
    for (int sl = 0; sl < 2; ++sl) {
      mbar_init(&S->vec_full[sl], 1);
      mbar_init(&S->vec_empty[sl], 8);  // one arrival per compute warp
    }
    mbar_init(&S->o_full, 1);
    mbar_init(&S->drain, 1);
    S->abort = 0;
    S->status = p.status;
    S->wait_limit_ns = p.wait_limit_ns ? p.wait_limit_ns : kWaitLimitNs;
    fence_barrier_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  return S->tmem_base;
}

__device__ __forceinline__ void bwd_teardown(uint32_t tmem) {
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x / 32 == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Producer: two resident tiles (maps f0, f1 at token t_fixed), then two
// streamed tiles per step (maps r0, r1 at token t0 + 128 j).
template <class L>
__device__ void bwd_producer(uint8_t* smem, BwdShared* S, const CUtensorMap* f0,
                             const CUtensorMap* f1, int t_fixed,
                             const CUtensorMap* r0, const CUtensorMap* r1,
                             int t0, int n, int h, int b) {
  constexpr int kS0 = L::kS0;
  // The resident tiles are read by this CTA alone (evict first); the
  // streamed tiles of a head are read by every CTA of the head (evict last).
  const uint64_t once = l2_policy_evict_first(), keep = l2_policy_evict_last();
  mbar_arrive_expect_tx(&S->fixed_full, 2 * L::kNB * kBox);
  for (int bx = 0; bx < L::kNB; ++bx) {
    tma_load_4d_hint(f0, smem + L::fixed(0, bx), &S->fixed_full, bx * 64,
                     t_fixed, h, b, once);
    tma_load_4d_hint(f1, smem + L::fixed(1, bx), &S->fixed_full, bx * 64,
                     t_fixed, h, b, once);
  }
  // Ring 1 first: its slot frees earlier in a step (after dP or dV), so its
  // next tile loads while the step still runs; ring 0 (after dQ or dK)
  // follows.
  int issued[2] = {0, 0};
  for (int j = 0; j < n; ++j) {
    const int s1 = j % kStages1, s0 = j % kS0;
    if (!wait_bar(&S->empty[1][s1], ((j / kStages1) & 1) ^ 1, S)) break;
    mbar_arrive_expect_tx(&S->full[1][s1], L::kNB * kBox);
    for (int bx = 0; bx < L::kNB; ++bx)
      tma_load_4d_hint(r1, smem + L::ring(s1, 1, bx), &S->full[1][s1],
                       bx * 64, t0 + j * kT, h, b, keep);
    ++issued[1];
    if (!wait_bar(&S->empty[0][s0], ((j / kS0) & 1) ^ 1, S)) break;
    mbar_arrive_expect_tx(&S->full[0][s0], L::kNB * kBox);
    for (int bx = 0; bx < L::kNB; ++bx)
      tma_load_4d_hint(r0, smem + L::ring(s0, 0, bx), &S->full[0][s0],
                       bx * 64, t0 + j * kT, h, b, keep);
    ++issued[0];
  }
  drain_wait(&S->fixed_full, 0);
  for (int i = max(0, issued[1] - kStages1); i < issued[1]; ++i)
    drain_wait(&S->full[1][i % kStages1], (i / kStages1) & 1);
  for (int i = max(0, issued[0] - kS0); i < issued[0]; ++i)
    drain_wait(&S->full[0][i % kS0], (i / kS0) & 1);
}

// One warp issues every MMA (an elected lane, the warp kept converged), and
// a tcgen05.mma takes it nearly as long to issue as the tensor pipe takes to
// run it, so the issue loops carry no
// descriptor arithmetic: each tile's descriptor low word is formed once per
// call and the K steps add constant offsets (16-byte units) to it.

// D_t = A_fixed * B_ring^T over the head dim (both K-major): TMEM col c0.
template <int D, class L>
__device__ __forceinline__ void mma_nt(uint32_t sbase, uint32_t tmem, int c0,
                                       int fixed_which, int st, int ring_which) {
  constexpr uint32_t kIdesc = idesc_bf16_f32(kT, kT, 0);
  const uint32_t hi = desc_hi_sw128(1024);
  const uint32_t a_lo = desc_lo(sbase + L::fixed(fixed_which, 0), 16);
  const uint32_t b_lo = desc_lo(sbase + L::ring(st, ring_which, 0), 16);
#pragma unroll
  for (int ks = 0; ks < D / 16; ++ks) {
    const uint32_t off = (uint32_t)((ks / 4) * kBox + (ks % 4) * 32) >> 4;
    mma_ss_warp(tmem + c0, a_lo + off, b_lo + off, hi, kIdesc, ks > 0);
  }
}

// D (+)= A_tmem * B, B an MN-major [128 x d] tile at SMEM offset b_off:
// TMEM column c0.  A is 128 x 128 bf16 written by the compute warps in two
// halves of 64 K-columns, each half's 32 packed columns at the start of its
// own 64-column range: K step kk (16 columns) is at a0 + 64 (kk / 4) + 8 (kk % 4).
template <int D>
__device__ __forceinline__ void mma_tn(uint32_t sbase, uint32_t tmem, int c0,
                                       int a0, int b_off, int acc) {
  constexpr uint32_t kIdesc = idesc_bf16_f32(kT, D, 1);
  const uint32_t hi = desc_hi_sw128(1024);
  const uint32_t b_lo = desc_lo(sbase + b_off, kBox);
#pragma unroll
  for (int kk = 0; kk < kT / 16; ++kk)
    mma_ts_warp(tmem + c0, tmem + a0 + 64 * (kk / 4) + 8 * (kk % 4),
                b_lo + (uint32_t)(kk * 2048 >> 4), hi, kIdesc, (acc | kk) != 0);
}

// Stage 32 fp32 accumulator columns [c0, c0 + 32) (scaled, as bf16) of TMEM
// row r into the output tile in shared memory: [128 x 64] bf16 boxes of
// 128-byte rows, 128-byte swizzled (16-byte chunk k of row r at chunk
// k ^ (r % 8)), the form a tiled TMA store of the token-major map reads.
// Rows leave in whole tiles (TMA stores) instead of one thread's 64 bytes at
// a stride of H d elements.
__device__ __forceinline__ void stage_row32(uint32_t taddr, float mul,
                                            uint8_t* tile, int r, int c0) {
  uint32_t v[32];
  tmem_ld32(taddr, v);
  tmem_wait_ld();
  uint32_t pk[16];
#pragma unroll
  for (int i = 0; i < 16; ++i)
    pk[i] = pack_bf16(__uint_as_float(v[2 * i]) * mul,
                      __uint_as_float(v[2 * i + 1]) * mul);
  uint8_t* row = tile + (c0 / 64) * kBox + r * 128;
  const int k0 = (c0 % 64) / 8;
#pragma unroll
  for (int q = 0; q < 4; ++q)
    *reinterpret_cast<uint4*>(row + (((k0 + q) ^ (r & 7)) << 4)) =
        make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
}

// After every compute thread staged its rows: one thread stores the staged
// tiles (one per map, kNB boxes each, rows from token t0) and waits until the
// writes are performed, so that the shared memory outlives the reads and the
// grid's completion covers the writes.
template <int kNB>
__device__ __forceinline__ void store_staged(const CUtensorMap* const* maps,
                                             uint8_t* const* tiles, int nmaps,
                                             int t0, int h, int b) {
  for (int m = 0; m < nmaps; ++m)
    for (int bx = 0; bx < kNB; ++bx)
      tma_store_4d(maps[m], tiles[m] + bx * kBox, bx * 64, t0, h, b);
  bulk_commit_group();
  bulk_wait_group0();
}

__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// 2^x of both halves of a packed pair on the FMA pipe: x = n + f with n the
// nearest integer (x + 1.5 * 2^23 rounds it into the low mantissa bits) and
// f in [-0.5, 0.5]; 2^f by a degree-3 polynomial (a relative-error minimax
// fit on [-0.5, 0.5], at most 7.5e-5 relative error in fp32: far below the
// 2^-9 of the bf16 P it feeds), then n added to its exponent field.  x is
// first clamped to >= -126 so that the exponent cannot wrap (2^x there is
// below 1.2e-38, against 0 from ex2.approx.ftz).  Some of the pairs take
// this path instead of MUFU ex2: the exponential step is bounded by the
// MUFU throughput, while the FMA pipe has room.
constexpr float kExpC0 = 0.9999281168f, kExpC1 = 0.6932609677f,
                kExpC2 = 0.2426105440f, kExpC3 = 0.0551713221f;
__device__ __forceinline__ void exp2_poly(float& x0, float& x1) {
  const uint64_t x = f2(fmaxf(x0, -126.f), fmaxf(x1, -126.f));
  const uint64_t t = f2_add(x, f2(12582912.f, 12582912.f));
  const uint64_t fr = f2_fma(f2_add(t, f2(-12582912.f, -12582912.f)),
                             f2(-1.f, -1.f), x);
  uint64_t q = f2_fma(f2(kExpC3, kExpC3), fr, f2(kExpC2, kExpC2));
  q = f2_fma(q, fr, f2(kExpC1, kExpC1));
  q = f2_fma(q, fr, f2(kExpC0, kExpC0));
  float p0, p1, t0, t1;
  f2_split(q, p0, p1);
  f2_split(t, t0, t1);
  x0 = __uint_as_float(__float_as_uint(p0) + (__float_as_uint(t0) << 23));
  x1 = __uint_as_float(__float_as_uint(p1) + (__float_as_uint(t1) << 23));
}
// Groups of four columns (of eight per 32) whose exponentials take the
// polynomial path in the unmasked step: one (training clip backward +0.5 %;
// two were slower, the FMA work then outweighing the MUFU it saves).
__device__ __forceinline__ constexpr bool poly_group(int q) { return q == 7; }

// P = 2^(s c2 - lse2) for 32 columns [c0, c0 + 32) of a half row, packed to
// bf16 pairs; with kMask, columns outside [lo, hi) are masked (p = 0).  nl
// holds -lse2 for the 32 columns, in registers: the dK/dV kernel reads its
// per-column values from shared memory ahead of use, because the SMEM x SMEM
// MMAs that run meanwhile take all of the shared-memory bandwidth and each
// read waits behind them.  The mask is a template argument, and the callers
// branch on a warp vote: a mask tested at run time inside the loop costs two
// compares and a select per element on every tile (measured: twice the time
// of the unmasked form), while only tiles that cross a chunk edge need it.
template <bool kMask>
__device__ __forceinline__ void p32(const uint32_t (&s)[32],
                                    const float4 (&nl)[8], int c0, int lo,
                                    int hi, uint64_t c2x2,
                                    uint32_t (&pp)[16]) {
#pragma unroll
  for (int q = 0; q < 8; ++q) {  // four columns at a time
    const float4 a = nl[q];
    float x[4];
    f2_split(f2_fma(f2(__uint_as_float(s[4 * q]), __uint_as_float(s[4 * q + 1])),
                    c2x2, f2(a.x, a.y)), x[0], x[1]);
    f2_split(f2_fma(f2(__uint_as_float(s[4 * q + 2]), __uint_as_float(s[4 * q + 3])),
                    c2x2, f2(a.z, a.w)), x[2], x[3]);
    if (kMask) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int col = c0 + 4 * q + u;
        if (col < lo || col >= hi) x[u] = -INFINITY;
      }
    }
    if (!kMask && poly_group(q)) {
      exp2_poly(x[0], x[1]);
      exp2_poly(x[2], x[3]);
      pp[2 * q] = pack_bf16(x[0], x[1]);
      pp[2 * q + 1] = pack_bf16(x[2], x[3]);
    } else {
      pp[2 * q] = pack_bf16(ex2(x[0]), ex2(x[1]));
      pp[2 * q + 1] = pack_bf16(ex2(x[2]), ex2(x[3]));
    }
  }
}

// dS = P (dP - D) for 32 columns: P as 16 bf16 pairs, dP fp32, nd holds -D
// for the 32 columns in registers.
__device__ __forceinline__ void ds32(const uint32_t (&pb)[16],
                                     const uint32_t (&dp)[32],
                                     const float4 (&nd)[8], uint32_t (&pd)[16]) {
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const float4 g = nd[q];
    float r[4];
    f2_split(f2_mul(f2(bf16_lo(pb[2 * q]), bf16_hi(pb[2 * q])),
                    f2_add(f2(__uint_as_float(dp[4 * q]),
                              __uint_as_float(dp[4 * q + 1])), f2(g.x, g.y))),
             r[0], r[1]);
    f2_split(f2_mul(f2(bf16_lo(pb[2 * q + 1]), bf16_hi(pb[2 * q + 1])),
                    f2_add(f2(__uint_as_float(dp[4 * q + 2]),
                              __uint_as_float(dp[4 * q + 3])), f2(g.z, g.w))),
             r[2], r[3]);
    pd[2 * q] = pack_bf16(r[0], r[1]);
    pd[2 * q + 1] = pack_bf16(r[2], r[3]);
  }
}

// ------------------------------------------------------------------ dK, dV
// TMEM: [0,128) S^T then P^T (bf16, first 64 columns), [128,256) dP^T then
// dS^T, [256,256+d) dV, [384,384+d) dK.  Resident: K (fixed 0), V (fixed 1).
// Streamed: Q (ring 0), dO (ring 1).
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
dkdv_kernel(const __grid_constant__ BwdParams p) {
  using L = DkdvLayout<D>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  // The layout fills 227 KB with no slack to round the base up: a base that
  // is not 1024-byte aligned (which the 128-byte-swizzled tiles need) is
  // reported as a failed bounds check and nothing is computed.
  if ((smem_addr(smem) & 1023u) != 0) {
    if (threadIdx.x == 0 && p.status != nullptr)
      atomicExch(p.status, kDevBounds);
    return;
  }
  BwdShared* S = reinterpret_cast<BwdShared*>(smem + L::shared_off);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  // Head-major order: the CTAs resident at one time cover one or two
  // (batch, head) rows, whose Q and dO tiles then stay in L2 for all of
  // them; within a head, key tiles ascend (the longest query ranges first).
  const int bh = blockIdx.x / p.tiles;
  const int h = bh % p.heads, b = bh / p.heads;
  const int k0 = (blockIdx.x % p.tiles) * kT;  // first key
  // Queries that see any key of the tile: chunks c(k0) .. c(k_last) + W.
  const int k_last = min(k0 + kT, p.seq_tokens) - 1;
  // Query tiles start at a multiple of 128 at or below the first visible
  // query (rows before it are masked), so each tile's 128 log2-LSE and D
  // values are one aligned slice inside the padded scratch row.
  const int q0 = (k0 / p.chunk_tokens) * p.chunk_tokens / kT * kT;
  const int q1 = p.window < 0 ? p.seq_tokens
                              : min((k_last / p.chunk_tokens + p.window + 1) *
                                        p.chunk_tokens,
                                    p.seq_tokens);
  const int n = (q1 - q0 + kT - 1) / kT;
  const uint32_t tmem = bwd_setup(S, p);

  if (warp == kProducerWarp) {
    if (lane == 0)
      bwd_producer<L>(smem, S, &p.k_map, &p.v_map, k0, &p.q_map, &p.do_map,
                      q0, n, h, b);
    __syncwarp();
  } else if (warp == kRelayWarp) {
    bwd_relay<kDkdvS0>(S, n);
  } else if (warp == kVecWarp) {
    // Row vectors: step j's 128 -log2 LSE and -D values into slot j % 2,
    // once the compute warps have released the slot (after dS of step j-2).
    if (lane == 0) {
      const int64_t row = (int64_t)bh_row(p, b, h) * p.padded;
      int issued = 0;
      for (int j = 0; j < n; ++j) {
        const int sl = j & 1;
        if (!wait_bar(&S->vec_empty[sl], ((j >> 1) & 1) ^ 1, S)) break;
        mbar_arrive_expect_tx(&S->vec_full[sl], 2 * kT * sizeof(float));
        bulk_load(smem + L::vec(sl, 0), p.lse2 + row + q0 + j * kT,
                  kT * sizeof(float), &S->vec_full[sl]);
        bulk_load(smem + L::vec(sl, 1), p.delta + row + q0 + j * kT,
                  kT * sizeof(float), &S->vec_full[sl]);
        ++issued;
      }
      for (int i = max(0, issued - 2); i < issued; ++i)
        drain_wait(&S->vec_full[i & 1], (i >> 1) & 1);
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    const uint32_t sbase = smem_addr(smem);
    // The next tile's S^T is issued right after this tile's dV (it
    // overwrites P^T, which dV has read: the pipe runs in issue order and
    // the compute warps keep P^T in registers), and the next dP^T right
    // after dK (over dS^T), so the compute warps start the next tile's P
    // as soon as they finish this tile's dS.
    // Test hook: o_full receives no arrival before the end, so this wait
    // runs out and exercises the abort path.
    bool ok = (!p.inject_stall || wait_bar_warp(&S->o_full, 0, S)) &&
              wait_bar_warp(&S->fixed_full, 0, S);
    if (ok) {
      relay_sync(kBarRing0);
      tc_fence_after();
      mma_nt<D, L>(sbase, tmem, 0, 0, 0, 0);    // S^T_0 = K Q_0^T
      mma_commit_warp(&S->s_ready);
      relay_sync(kBarRing1);
      tc_fence_after();
      mma_nt<D, L>(sbase, tmem, 128, 1, 0, 1);  // dP^T_0 = V dO_0^T
      mma_commit_warp(&S->dp_ready[0]);
    }
    for (int j = 0; ok && j < n; ++j) {
      // Q (ring 0) and dO (ring 1) run at their own depths
      const int q_st = j % kDkdvS0, q_stn = (j + 1) % kDkdvS0;
      const int o_st = j % kStages1, o_stn = (j + 1) % kStages1;
      compute_sync(kBarP);
      tc_fence_after();
      mma_tn<D>(sbase, tmem, 256, 0, L::ring(o_st, 1, 0), j > 0);    // dV
      mma_commit_warp(&S->empty[1][o_st]);  // dO_j read for the last time
      if (j + 1 < n) {
        relay_sync(kBarRing0 + q_stn);
        tc_fence_after();
        mma_nt<D, L>(sbase, tmem, 0, 0, q_stn, 0);  // S^T_{j+1}
        mma_commit_warp(&S->s_ready);
      }
      compute_sync(kBarDS);
      tc_fence_after();
      mma_tn<D>(sbase, tmem, 384, 128, L::ring(q_st, 0, 0), j > 0);  // dK
      mma_commit_warp(&S->empty[0][q_st]);  // Q_j read for the last time
      if (j + 1 < n) {
        relay_sync(kBarRing1 + o_stn);
        tc_fence_after();
        mma_nt<D, L>(sbase, tmem, 128, 1, o_stn, 1);  // dP^T_{j+1}
        mma_commit_warp(&S->dp_ready[0]);
      }
    }
    if (ok) mma_commit_warp(&S->o_full);
    mma_commit_warp(&S->drain);
    if (lane == 0) drain_wait(&S->drain, 0);
    __syncwarp();
  } else {
    // Compute warps: warp w owns key rows 32 (w % 4) .. + 31 (its TMEM
    // lanes) and query columns [64 hf, 64 hf + 64) with hf = w / 4; it writes
    // its bf16 P^T and dS^T over the first 32 of its own S^T and dP^T
    // columns, so the two warps of a row never touch each other's columns.
    const int hf = warp / 4;
    const int t = (warp % 4) * 32 + lane;  // key row within the tile
    const uint32_t row_t = tmem + ((uint32_t)((warp % 4) * 32) << 16);
    const uint32_t cs = 64 * hf, cp = 128 + 64 * hf;
    int vis_lo, vis_hi;
    key_sees(p, k0 + t, vis_lo, vis_hi);
    const uint64_t c2x2 = f2(p.scale_log2, p.scale_log2);
    bool ok = true;
    int p_arr = 0, ds_arr = 0;  // hand-offs made to the MMA warp
    for (int j = 0; j < n; ++j) {
      const int i0 = q0 + j * kT + 64 * hf;  // first query of this half
      const int sl = j & 1;
      // this step's LSE and D slices (released after dS, below)
      if (!(ok = wait_bar_warp(&S->vec_full[sl], (j >> 1) & 1, S))) break;
      // -log2 LSE and -D per column
      const float* nl = reinterpret_cast<const float*>(smem + L::vec(sl, 0)) + 64 * hf;
      const float* nd = reinterpret_cast<const float*>(smem + L::vec(sl, 1)) + 64 * hf;
      // the first half's LSE values land while S^T is computed
      float4 la[8], lb[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) la[q] = reinterpret_cast<const float4*>(nl)[q];
      if (!(ok = wait_bar_warp(&S->s_ready, j & 1, S))) break;
      tc_fence_after();
      const int lo = vis_lo - i0, hi = vis_hi - i0;
      const bool need_mask = __any_sync(0xffffffffu, lo > 0 || hi < 64);
      uint32_t x0[32], x1[32], pb0[16], pb1[16], pk[16];
      // phase 1: P^T over the first half of S^T (for the dV MMA) and in
      // registers (for dS: the next tile's S^T may overwrite it in TMEM as
      // soon as dV has run)
      tmem_ld32(row_t + cs, x0);
      tmem_ld32(row_t + cs + 32, x1);
#pragma unroll
      for (int q = 0; q < 8; ++q)
        lb[q] = reinterpret_cast<const float4*>(nl + 32)[q];
      tmem_wait_ld();
      if (need_mask) {
        p32<true>(x0, la, 0, lo, hi, c2x2, pb0);
        tmem_st16(row_t + cs, pb0);
        p32<true>(x1, lb, 32, lo, hi, c2x2, pb1);
      } else {
        p32<false>(x0, la, 0, lo, hi, c2x2, pb0);
        tmem_st16(row_t + cs, pb0);
        p32<false>(x1, lb, 32, lo, hi, c2x2, pb1);
      }
      tmem_st16(row_t + cs + 16, pb1);
      tmem_wait_st();
      tc_fence_before();
      compute_arrive(kBarP);
      ++p_arr;
      // phase 2 (overlaps the dV and next S^T MMAs): dS^T over the first
      // half of dP^T; the D values are read ahead like the LSE values
#pragma unroll
      for (int q = 0; q < 8; ++q) la[q] = reinterpret_cast<const float4*>(nd)[q];
      if (!(ok = wait_bar_warp(&S->dp_ready[0], j & 1, S))) break;
      tc_fence_after();
      tmem_ld32(row_t + cp, x0);
      tmem_ld32(row_t + cp + 32, x1);
#pragma unroll
      for (int q = 0; q < 8; ++q)
        lb[q] = reinterpret_cast<const float4*>(nd + 32)[q];
      tmem_wait_ld();
      ds32(pb0, x0, la, pk);
      tmem_st16(row_t + cp, pk);
      ds32(pb1, x1, lb, pk);
      tmem_st16(row_t + cp + 16, pk);
      tmem_wait_st();
      tc_fence_before();
      compute_arrive(kBarDS);
      ++ds_arr;
      // the row-vector slot is read for the last time
      __syncwarp();
      if (lane == 0) mbar_arrive(&S->vec_empty[sl]);
    }
    // After a failed wait the remaining hand-offs are still made (with
    // undefined contents), so that the MMA warp never waits for an arrival
    // that does not come.
    for (; p_arr < n; ++p_arr) compute_arrive(kBarP);
    for (; ds_arr < n; ++ds_arr) compute_arrive(kBarDS);
    // dV and dK are staged in the first two Q stages (free once o_full has
    // completed: every MMA has read its operands) and leave as TMA stores;
    // rows past the sequence fall outside the map and are not written.
    uint8_t* const tiles[2] = {smem + L::ring(0, 0, 0), smem + L::ring(1, 0, 0)};
    if (ok && wait_bar_warp(&S->o_full, 0, S)) {
      tc_fence_after();
#pragma unroll 1
      for (int c = hf * D / 64; c < (hf + 1) * D / 64; ++c) {
        stage_row32(row_t + 256 + c * 32, 1.f, tiles[0], t, c * 32);
        stage_row32(row_t + 384 + c * 32, p.scale, tiles[1], t, c * 32);
      }
      fence_proxy_async_smem();
    }
    compute_only_sync(kBarStaged);
    if (warp == 0 && lane == 0 && ok &&
        !*reinterpret_cast<volatile int*>(&S->abort)) {
      const CUtensorMap* const maps[2] = {&p.dv_map, &p.dk_map};
      store_staged<L::kNB>(maps, tiles, 2, k0, h, b);
    }
  }
  bwd_teardown(tmem);
}

// --------------------------------------------------------------------- dQ
// TMEM: [0,128) S, [128,256) and [384,512) dP then dS (bf16, first 64
// columns) for even and odd steps, [256,256+d) dQ.  Resident: Q (fixed 0),
// dO (fixed 1).  Streamed: K (ring 0), V (ring 1).
__device__ __forceinline__ int dq_dp_col(int j) { return (j & 1) ? 384 : 128; }
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
dq_kernel(const __grid_constant__ BwdParams p) {
  using L = BwdLayout<D, kDqS0>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  BwdShared* S = reinterpret_cast<BwdShared*>(smem + L::shared_off);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  // Head-major order (the resident CTAs share their K and V tiles in L2);
  // within a head, the longest key ranges first.
  const int bh = blockIdx.x / p.tiles;
  const int h = bh % p.heads, b = bh / p.heads;
  const int q0 = (p.tiles - 1 - blockIdx.x % p.tiles) * kT;
  const int q_last = min(q0 + kT, p.seq_tokens) - 1;
  const int c_lo = q0 / p.chunk_tokens, c_hi = q_last / p.chunk_tokens;
  const int kv0 = p.window < 0 ? 0 : max(0, c_lo - p.window) * p.chunk_tokens;
  const int kv1 = min((c_hi + 1) * p.chunk_tokens, p.seq_tokens);
  const int n = (kv1 - kv0 + kT - 1) / kT;
  const uint32_t tmem = bwd_setup(S, p);

  if (warp == kProducerWarp) {
    if (lane == 0)
      bwd_producer<L>(smem, S, &p.q_map, &p.do_map, q0, &p.k_map, &p.v_map,
                      kv0, n, h, b);
    __syncwarp();
  } else if (warp == kRelayWarp) {
    bwd_relay<kDqS0>(S, n);
  } else if (warp == kVecWarp) {
    // no row-vector warp here: each compute thread reads its own row's two
    // values once
  } else if (warp == kMmaWarp) {
    const uint32_t sbase = smem_addr(smem);
    // S and dP of the next tile are issued as soon as P of this one is in
    // registers, so they overlap the dS computation; dP alternates between
    // two buffers, so it need not wait for this tile's dQ to read dS.
    // Test hook: o_full receives no arrival before the end, so this wait
    // runs out and exercises the abort path.
    bool ok = (!p.inject_stall || wait_bar_warp(&S->o_full, 0, S)) &&
              wait_bar_warp(&S->fixed_full, 0, S);
    if (ok) {
      relay_sync(kBarRing0);
      tc_fence_after();
      mma_nt<D, L>(sbase, tmem, 0, 0, 0, 0);    // S_0 = Q K_0^T
      mma_commit_warp(&S->s_ready);
      relay_sync(kBarRing1);
      tc_fence_after();
      mma_nt<D, L>(sbase, tmem, dq_dp_col(0), 1, 0, 1);  // dP_0 = dO V_0^T
      mma_commit_warp(&S->dp_ready[0]);
      mma_commit_warp(&S->empty[1][0]);  // V_0 read for the last time
    }
    for (int j = 0; ok && j < n; ++j) {
      // K (ring 0) and V (ring 1) run at their own depths
      const int k_st = j % kDqS0, k_stn = (j + 1) % kDqS0;
      const int v_stn = (j + 1) % kStages1;
      compute_sync(kBarP);
      if (j + 1 < n) {
        relay_sync(kBarRing0 + k_stn);
        tc_fence_after();
        mma_nt<D, L>(sbase, tmem, 0, 0, k_stn, 0);  // S_{j+1}
        mma_commit_warp(&S->s_ready);
        // dP_{j+1} goes to the buffer that dQ_{j-1} (issued before) read
        relay_sync(kBarRing1 + v_stn);
        tc_fence_after();
        mma_nt<D, L>(sbase, tmem, dq_dp_col(j + 1), 1, v_stn, 1);
        mma_commit_warp(&S->dp_ready[(j + 1) & 1]);
        mma_commit_warp(&S->empty[1][v_stn]);  // V_{j+1} read for the last time
      }
      compute_sync(kBarDS);
      tc_fence_after();
      mma_tn<D>(sbase, tmem, 256, dq_dp_col(j), L::ring(k_st, 0, 0), j > 0);  // dQ
      mma_commit_warp(&S->empty[0][k_st]);  // K_j read for the last time
    }
    if (ok) mma_commit_warp(&S->o_full);
    mma_commit_warp(&S->drain);
    if (lane == 0) drain_wait(&S->drain, 0);
    __syncwarp();
  } else {
    // Compute warps: warp w owns query rows 32 (w % 4) .. + 31 and key
    // columns [64 hf, 64 hf + 64), hf = w / 4; dS goes over the first 32 of
    // its own dP columns.
    const int hf = warp / 4;
    const int t = (warp % 4) * 32 + lane;
    const uint32_t row_t = tmem + ((uint32_t)((warp % 4) * 32) << 16);
    const uint32_t cs = 64 * hf;
    const int row = q0 + t;
    const bool in_range = row < p.seq_tokens;
    int vis_lo, vis_hi;
    query_sees(p, row, vis_lo, vis_hi);
    const int64_t rl = (int64_t)bh_row(p, b, h) * p.padded + row;
    const float nl_row = p.lse2[rl];  // -log2 LSE (padded rows hold 0)
    float4 nl_v[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) nl_v[q] = make_float4(nl_row, nl_row, nl_row, nl_row);
    const float nd_row = p.delta[rl];  // -D
    float4 nd_v[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) nd_v[q] = make_float4(nd_row, nd_row, nd_row, nd_row);
    const uint64_t c2x2 = f2(p.scale_log2, p.scale_log2);
    bool ok = true;
    int p_arr = 0, ds_arr = 0;  // hand-offs made to the MMA warp
    for (int j = 0; j < n; ++j) {
      const int tok0 = kv0 + j * kT + 64 * hf;
      if (!(ok = wait_bar_warp(&S->s_ready, j & 1, S))) break;
      tc_fence_after();
      const int lo = vis_lo - tok0;
      const int hi = vis_hi - tok0;
      const bool need_mask =
          __any_sync(0xffffffffu, lo > 0 || hi < 64 || !in_range);
      const int lo_m = in_range ? lo : 64, hi_m = in_range ? hi : 0;
      uint32_t x0[32], x1[32], pb0[16], pb1[16], pk[16];
      // phase 1 (overlaps the dP MMAs): P (bf16 pairs) in registers; S is
      // then free for the next tile
      tmem_ld32(row_t + cs, x0);
      tmem_ld32(row_t + cs + 32, x1);
      tmem_wait_ld();
      if (need_mask) {
        p32<true>(x0, nl_v, 0, lo_m, hi_m, c2x2, pb0);
        p32<true>(x1, nl_v, 32, lo_m, hi_m, c2x2, pb1);
      } else {
        p32<false>(x0, nl_v, 0, lo_m, hi_m, c2x2, pb0);
        p32<false>(x1, nl_v, 32, lo_m, hi_m, c2x2, pb1);
      }
      tc_fence_before();
      compute_arrive(kBarP);
      ++p_arr;
      // phase 2 (overlaps the next tile's S and dP MMAs): dS over this
      // step's dP buffer
      if (!(ok = wait_bar_warp(&S->dp_ready[j & 1], (j >> 1) & 1, S))) break;
      tc_fence_after();
      const uint32_t cp = dq_dp_col(j) + 64 * hf;
      tmem_ld32(row_t + cp, x0);
      tmem_ld32(row_t + cp + 32, x1);
      tmem_wait_ld();
      ds32(pb0, x0, nd_v, pk);
      tmem_st16(row_t + cp, pk);
      ds32(pb1, x1, nd_v, pk);
      tmem_st16(row_t + cp + 16, pk);
      tmem_wait_st();
      tc_fence_before();
      compute_arrive(kBarDS);
      ++ds_arr;
    }
    // After a failed wait the remaining hand-offs are still made (with
    // undefined contents), so that the MMA warp never waits for an arrival
    // that does not come.
    for (; p_arr < n; ++p_arr) compute_arrive(kBarP);
    for (; ds_arr < n; ++ds_arr) compute_arrive(kBarDS);
    // dQ is staged in the first K stage (free once o_full has completed)
    // and leaves as TMA stores; rows past the sequence are not written.
    uint8_t* const tiles[1] = {smem + L::ring(0, 0, 0)};
    if (ok && wait_bar_warp(&S->o_full, 0, S)) {
      tc_fence_after();
#pragma unroll 1
      for (int c = hf * D / 64; c < (hf + 1) * D / 64; ++c)
        stage_row32(row_t + 256 + c * 32, p.scale, tiles[0], t, c * 32);
      fence_proxy_async_smem();
    }
    compute_only_sync(kBarStaged);
    if (warp == 0 && lane == 0 && ok &&
        !*reinterpret_cast<volatile int*>(&S->abort)) {
      const CUtensorMap* const maps[1] = {&p.dq_map};
      store_staged<L::kNB>(maps, tiles, 1, q0, h, b);
    }
  }
  bwd_teardown(tmem);
}

// Scratch rows for the backward: -D_i = -<dO_i, O_i> over the head dim and
// minus the forward LSE in log2 units (negated so that both enter packed
// FMAs as addends), each [B*H, Lpad] with Lpad = L rounded up to 128 and
// zeros in the padding (so every 128-token slice is aligned and in bounds).
// A block takes kDeltaTokens tokens of one (batch, head): D / 8 lanes per
// token row of O and dO (one 16-byte piece each; a row is 2 D contiguous
// bytes), every load of the block issued before the first product, then the
// block writes its kDeltaTokens values of -D and -log2 LSE as one contiguous
// run each (through shared memory), and reads the forward LSE the same way.
// Tokens past the sequence (up to the padded length) get zeros.
constexpr int kDeltaTokens = 64;
constexpr int kDeltaThreads = 256;

template <int D>
__global__ void __launch_bounds__(kDeltaThreads)
delta_kernel(const uint16_t* o, const uint16_t* dO, const float* lse,
             float* lse2, float* delta, int heads, int seq, int padded) {
  constexpr int kLanesPerRow = D / 8;
  constexpr int kRowsPerPass = kDeltaThreads / kLanesPerRow;
  constexpr int kPasses = kDeltaTokens / kRowsPerPass;
  __shared__ float red[kDeltaTokens];
  const int tiles = padded / kDeltaTokens;
  const int bh = blockIdx.x / tiles;  // b * heads + h
  const int t0 = (blockIdx.x % tiles) * kDeltaTokens;
  const int b = bh / heads, h = bh % heads;
  const int sub = threadIdx.x / kLanesPerRow, piece = threadIdx.x % kLanesPerRow;
  uint4 a[kPasses], g[kPasses];
#pragma unroll
  for (int u = 0; u < kPasses; ++u) {
    const int tok = t0 + u * kRowsPerPass + sub;
    a[u] = g[u] = make_uint4(0, 0, 0, 0);
    if (tok < seq) {
      const int64_t r = ((int64_t)b * seq + tok) * heads + h;  // [B, L, H] row
      a[u] = __ldcs(reinterpret_cast<const uint4*>(o + r * D) + piece);
      g[u] = __ldcs(reinterpret_cast<const uint4*>(dO + r * D) + piece);
    }
  }
#pragma unroll
  for (int u = 0; u < kPasses; ++u) {
    const uint32_t* ap = reinterpret_cast<const uint32_t*>(&a[u]);
    const uint32_t* gp = reinterpret_cast<const uint32_t*>(&g[u]);
    float acc = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      acc = fmaf(__uint_as_float(ap[e] << 16), __uint_as_float(gp[e] << 16), acc);
      acc = fmaf(__uint_as_float(ap[e] & 0xffff0000u),
                 __uint_as_float(gp[e] & 0xffff0000u), acc);
    }
#pragma unroll
    for (int m = kLanesPerRow / 2; m > 0; m >>= 1)
      acc += __shfl_xor_sync(0xffffffffu, acc, m);
    if (piece == 0) red[u * kRowsPerPass + sub] = acc;
  }
  __syncthreads();
  if (threadIdx.x < kDeltaTokens) {
    const int tok = t0 + threadIdx.x;
    const int64_t i = (int64_t)bh * padded + tok;
    const bool in = tok < seq;
    delta[i] = in ? -red[threadIdx.x] : 0.f;
    lse2[i] = in ? -lse[(int64_t)bh * seq + tok] * 1.4426950408889634f : 0.f;
  }
}


// Token-major [B, L, H, d] bf16 tensor as a 4-D map over (d, token, head,
// batch), box 64 x 128, 128-byte swizzle; tokens past L read as zeros.
bool token_major_map(CUtensorMap* m, const void* base, int d, int L, int H,
                     int B) {
  EncodeTiledFn enc = encode_tiled_fn();
  if (enc == nullptr) return false;
  const cuuint64_t dims[4] = {(cuuint64_t)d, (cuuint64_t)L, (cuuint64_t)H,
                              (cuuint64_t)B};
  const cuuint64_t strides[3] = {(cuuint64_t)H * d * 2, (cuuint64_t)d * 2,
                                 (cuuint64_t)L * H * d * 2};
  const cuuint32_t box[4] = {64, 128, 1, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base),
             dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// One non-blocking side stream and a fork / join event pair per device,
// created on first use and kept until exit.  Calls on one device share them:
// the caller holds g_side_mutex from the fork record to the join wait, so
// host threads cannot interleave their event records, and their dQ kernels
// run one after the other on the side stream.
struct SideStream {
  cudaStream_t stream;
  cudaEvent_t fork, join;
};
constexpr int kMaxSideDevices = 64;
std::mutex g_side_mutex;
SideStream* g_side[kMaxSideDevices] = {};

// Requires g_side_mutex held.
SideStream* side_stream(int dev) {
  if (dev < 0 || dev >= kMaxSideDevices) return nullptr;
  if (g_side[dev] == nullptr) {
    SideStream* s = new SideStream();
    if (cudaStreamCreateWithFlags(&s->stream, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&s->fork, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&s->join, cudaEventDisableTiming) != cudaSuccess) {
      cudaGetLastError();
      delete s;
      return nullptr;
    }
    g_side[dev] = s;
  }
  return g_side[dev];
}

template <int D>
cudaError_t launch_bwd_d(const BwdArgs& a, cudaStream_t stream) {
  BwdParams p;
  memset(&p, 0, sizeof(p));
  const int L = a.seq_tokens;
  if (!token_major_map(&p.q_map, a.q, D, L, a.heads, a.batch) ||
      !token_major_map(&p.k_map, a.k, D, L, a.heads, a.batch) ||
      !token_major_map(&p.v_map, a.v, D, L, a.heads, a.batch) ||
      !token_major_map(&p.do_map, a.dout, D, L, a.heads, a.batch) ||
      !token_major_map(&p.dq_map, a.dq, D, L, a.heads, a.batch) ||
      !token_major_map(&p.dk_map, a.dk, D, L, a.heads, a.batch) ||
      !token_major_map(&p.dv_map, a.dv, D, L, a.heads, a.batch))
    return cudaErrorInvalidValue;
  const int padded = (L + kT - 1) / kT * kT;
  p.lse2 = a.scratch;
  p.delta = a.scratch + (size_t)a.batch * a.heads * padded;
  p.padded = padded;
  p.dq = a.dq;
  p.dk = a.dk;
  p.dv = a.dv;
  p.seq_tokens = L;
  p.heads = a.heads;
  p.batch = a.batch;
  p.chunk_tokens = a.chunk_tokens;
  p.window = a.window;
  p.tiles = (L + kT - 1) / kT;
  p.scale = a.scale;
  p.scale_log2 = a.scale * 1.4426950408889634f;
  p.status = a.status;
  p.inject_stall = a.inject_stall;
  p.wait_limit_ns = a.wait_limit_ns;

  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t blocks =
      (int64_t)a.batch * a.heads * (padded / kDeltaTokens);
  delta_kernel<D><<<(unsigned)blocks, kDeltaThreads, 0, stream>>>(
      a.out, a.dout, a.lse, a.scratch, a.scratch + (size_t)a.batch * a.heads * padded,
      a.heads, L, padded);
  const int smem = DkdvLayout<D>::bytes;
  const int smem_dq = BwdLayout<D, kDqS0>::bytes;
  static_assert(DkdvLayout<128>::bytes <= 227 * 1024 &&
                    BwdLayout<128, kDqS0>::bytes <= 227 * 1024,
                "backward shared memory");
  cudaError_t e = cudaFuncSetAttribute(
      dkdv_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(dq_kernel<D>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem_dq);
  if (e != cudaSuccess) return e;
  const int grid = p.tiles * a.heads * a.batch;
  // dK/dV and dQ are independent (both read only the inputs and the
  // scratch rows).  With few waves, dQ runs on a side stream forked after
  // delta_kernel and joined before return, so its CTAs fill the SMs that
  // dK/dV's last, partial wave leaves idle (training clip, 15 waves: +1.7 %);
  // with many waves the tail is negligible and two long-sequence kernels at
  // once contend for L2 (1080p sequence, 151 waves: -2 %), so both run in
  // order, as they also do without a side stream.
  constexpr int kMaxForkWaves = 32;
  std::lock_guard<std::mutex> lock(g_side_mutex);
  SideStream* side = grid <= kMaxForkWaves * (sms > 0 ? sms : 152)
                         ? side_stream(dev)
                         : nullptr;
  if (side != nullptr && cudaEventRecord(side->fork, stream) == cudaSuccess &&
      cudaStreamWaitEvent(side->stream, side->fork, 0) == cudaSuccess) {
    dkdv_kernel<D><<<grid, kThreads, smem, stream>>>(p);
    dq_kernel<D><<<grid, kThreads, smem_dq, side->stream>>>(p);
    e = cudaGetLastError();
    const cudaError_t j = cudaEventRecord(side->join, side->stream);
    const cudaError_t w = j == cudaSuccess
                              ? cudaStreamWaitEvent(stream, side->join, 0)
                              : j;
    return e != cudaSuccess ? e : w;
  }
  cudaGetLastError();
  dkdv_kernel<D><<<grid, kThreads, smem, stream>>>(p);
  dq_kernel<D><<<grid, kThreads, smem_dq, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_blockcausal_attn_bwd(const BwdArgs& a, cudaStream_t stream) {
  if (a.head_dim == 64) return launch_bwd_d<64>(a, stream);
  if (a.head_dim == 128) return launch_bwd_d<128>(a, stream);
  return cudaErrorInvalidValue;
}

}  // namespace fastvr
