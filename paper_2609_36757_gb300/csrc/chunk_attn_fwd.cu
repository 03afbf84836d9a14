// Chunk-causal attention forward for sm_103a (Sec. 3.1, Eq. 1): tcgen05
// tensor cores with TMEM accumulators, TMA-staged tiles, fp32 online softmax.
//
// Masking acts at chunk granularity and a call attends one chunk's queries,
// so every key of the visible segments is visible to every query: the host
// enumerates only visible cache ranges (block-causal skipping happens before
// launch, invisible chunks are never loaded) and the only in-kernel mask is
// the ragged end of a segment.
//
// One CTA owns two 128-row query tiles of one (batch, head) and streams the
// visible keys in 128-key tiles:
//   warp 8      TMA producer of the Q tiles (once) and the K ring (3 deep);
//   warp 10     TMA producer of the V ring (2 deep); all tiles are
//               128-byte swizzled boxes of 64 columns.
//   warp 11     relay: observes the TMA completions and hands each K/V ring
//               stage to the MMA warp through a named barrier.
//   warp 9      MMA issuer (the warp runs converged, an elected lane
//               issues): S = Q_t K^T into TMEM, then O_t += P_t V with P_t
//               read from TMEM; order per key tile j: QK_0(j), PV_0(j-1),
//               QK_1(j), PV_1(j-1).
//   warps 0-3   softmax of query tile 0, one thread per row (TMEM lane);
//   warps 4-7   softmax of query tile 1.
// TMEM (512 columns): S (shared by the two tiles) | P_0 | P_1 | O_0 | O_1,
// 128 + 64 + 64 + 128 + 128 columns.  S only lives until the softmax warps
// have loaded it (they release it before the row max), so the next QK^T of
// either tile can follow at once; each tile's PV runs one key tile behind,
// which gives its softmax three MMA steps to store P_t.  The MMA warp never
// polls a shared-memory barrier: every hand-off to it (S read, P_t stored,
// K/V stage landed) is a named barrier, whose arrivals are made on every
// path (also after a failed wait), since a named barrier has no time limit.
//
// Online softmax in the exp2 domain: each row keeps a reference m (a lower
// bound of its running max) and exponentiates against it; m moves, and O is
// rescaled, only when a tile's max exceeds m by more than 8 (P stays <= 256,
// finite in bf16 and fp32).  The final O / l is the same for any reference,
// so this is exact up to rounding.  Before storing P_t(j) the softmax waits
// until PV_t(j-1) has completed, so O_t is current for the rare rescale.
//
// Epilogue: a whole unit's softmax warps stage O_t / l as bf16 in the Q_t
// buffer (free once every MMA has completed) and one thread per tile writes
// it with tiled TMA stores; a split unit's key ranges write fp32 partials
// and the log2-domain LSE for the merge kernel.  The TMA loads carry L2
// policies: evict_first for the query tiles (one CTA reads them),
// evict_last for K/V (every unit of the head reads them).
//
// Every mbarrier wait is bounded: past the limit the kernel records
// FASTVR timeout in the control word, all roles stop issuing, in-flight TMA
// loads and MMAs are drained, TMEM is released and the CTA exits.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>

#include <algorithm>

#include "fastvr_internal.h"
#include "sm100_ptx.cuh"

namespace fastvr {
namespace {

using namespace sm100;

constexpr int kBM = 128;        // query rows per tile (one TMEM lane each)
constexpr int kBN = 128;        // keys per tile
constexpr int kQTiles = 2;      // query tiles per CTA
constexpr int kKStages = 3;     // depth of the K ring
constexpr int kVStages = 2;     // depth of the V ring
constexpr int kThreads = 384;   // 8 softmax warps, K and V producers, MMA,
                                // relay
constexpr int kBox = 128 * 128; // one TMA box: 128 rows x 64 bf16 (bytes)
constexpr uint32_t kTmemCols = 512;
// TMEM columns: one S tile shared by the two query tiles, P_0 and P_1 (bf16
// pairs, 64 columns each), O_0 and O_1.
constexpr uint32_t kTmemS = 0;
constexpr uint32_t kTmemP = 128;
constexpr uint32_t kTmemO = 256;
constexpr float kRescaleThreshold = 8.0f;      // log2 units
constexpr int kMinTilesPerPart = 4;             // key tiles per split part
constexpr uint64_t kDefaultWaitLimitNs = 4000000000ull;  // 4 s per wait
// Named (hardware) barriers of the softmax -> MMA hand-offs: S read (free
// for the next QK^T) and P_t stored.  The four softmax warps of a tile
// arrive, the MMA warp syncs: kHandoff threads per generation.
constexpr int kBarSFree = 1;
constexpr int kBarPFull0 = 2;  // + t
constexpr int kHandoff = 5 * 32;
// Named barriers of the relay -> MMA hand-offs, one per ring stage: K (or V)
// stage s has landed.  The relay warp arrives, the MMA warp syncs.
constexpr int kBarKFull0 = 4;  // + stage (kKStages of them)
constexpr int kBarVFull0 = 7;  // + stage (kVStages of them)
constexpr int kRelay = 2 * 32;
// Named barrier of a query tile's four softmax warps: their rows of O are
// staged for the tile's TMA store.
constexpr int kBarOStaged0 = 9;  // + t

struct TcParams {
  CUtensorMap q_map;                  // {d, Lq, H, B}
  CUtensorMap o_map;                  // the output, the same form as q_map
  CUtensorMap k_map[kMaxSegments];    // {d, segment end, H, B} of the cache
  CUtensorMap v_map[kMaxSegments];
  uint16_t* o;
  float* lse;
  Strides o_str;
  int32_t q_tokens, heads;
  int32_t seg_start[kMaxSegments];
  int32_t seg_len[kMaxSegments];
  int32_t seg_tiles0;   // tiles of segment 0
  int32_t total_tiles;
  float scale_log2;
  int* status;
  uint64_t wait_limit_ns;
  int32_t inject_stall;
  // Work split: units of two query tiles, (b, h, pair) with the pair index
  // fastest; the first units_full run whole, the rest are cut into `split`
  // key-tile ranges whose partial results go to the workspace.
  int32_t q_pairs, units_full, split;
  int32_t sms;  // SM count: CTA index / sms is a CTA's wave
  float* ws;      // partial O: [part][d][kUnitRows]
  float* ws_lse;  // partial log2-domain LSE: [part][kUnitRows]
  int32_t ws_parts;  // partial results the workspace holds
  int64_t o_elems;   // elements of o (B Lq H d), for the debug index checks
  // One-shot (training-form) launches: the whole sequence of seq_tokens
  // tokens, chunks of chunk_tokens tokens, window W (-1: unbounded).
  int32_t seq_tokens, chunk_tokens, window, batch;
};

// The work of one CTA.
struct Work {
  int q0, h, b;
  int j0, n;   // first key tile (index into the visible tiles) and count
  int nqt;     // query tiles with at least one row in the chunk (1 or 2)
  int part;    // -1: whole unit, final output; else workspace slot
  int kv0, kv1;  // one-shot: the unit's key token range [kv0, kv1)
  bool rev;    // walk the key tiles last to first
};

// Whole units in odd waves (CTA index / SM count) walk their key tiles last
// to first.  Consecutive units of a head run together, so a head whose units
// straddle two waves is streamed by the second wave right after the first:
// walking back, that wave starts on the tiles the first one loaded last,
// which are still in L2, instead of on the oldest ones.  The online softmax
// does not depend on the order (up to rounding).
__device__ __forceinline__ bool odd_wave(const TcParams& p) {
  return ((int)blockIdx.x / p.sms) & 1;
}

// One-shot launches: the query pairs are grouped from the end of the
// sequence into blocks of kOneShotBlock pairs; unit x takes block
// x / (kOneShotBlock H B) (the units with the most keys start first), then
// (b, h) and a pair within the block with the pair fastest, so that the CTAs
// of one wave stream the keys of a few heads, each shared by up to
// kOneShotBlock CTAs, rather than of every head at once.  A unit's keys are
// the union of what its rows see: chunks max(0, c_lo - W) .. c_hi of its
// first and last rows (Eq. 1 with window W).
constexpr int kOneShotBlock = 32;

__device__ __forceinline__ Work oneshot_work(const TcParams& p) {
  Work w;
  const int hb = p.heads * p.batch;
  const int blk = blockIdx.x / (kOneShotBlock * hb);
  const int x = blockIdx.x % (kOneShotBlock * hb);
  const int in_blk = min(kOneShotBlock, p.q_pairs - blk * kOneShotBlock);
  const int bh = x / in_blk;
  const int pair = p.q_pairs - 1 - blk * kOneShotBlock - x % in_blk;
  w.h = bh % p.heads;
  w.b = bh / p.heads;
  w.q0 = pair * kQTiles * kBM;
  w.nqt = (p.q_tokens - w.q0 > kBM) ? 2 : 1;
  const int c_lo = w.q0 / p.chunk_tokens;
  const int c_hi = min(w.q0 + kQTiles * kBM, p.q_tokens) - 1;
  const int chunk_hi = c_hi / p.chunk_tokens;
  w.kv0 = p.window < 0 ? 0 : max(0, c_lo - p.window) * p.chunk_tokens;
  w.kv1 = min((chunk_hi + 1) * p.chunk_tokens, p.seq_tokens);
  w.j0 = 0;
  w.n = (w.kv1 - w.kv0 + kBN - 1) / kBN;
  w.part = -1;
  w.rev = odd_wave(p);
  return w;
}

template <bool kOneShot>
__device__ __forceinline__ Work cta_work(const TcParams& p) {
  if (kOneShot) return oneshot_work(p);
  Work w;
  w.kv0 = w.kv1 = 0;
  int unit, part = -1, nparts = 1, idx = 0;
  if ((int)blockIdx.x < p.units_full) {
    unit = blockIdx.x;
  } else {
    const int k = blockIdx.x - p.units_full;
    unit = p.units_full + k / p.split;
    idx = k % p.split;
    part = k;
    nparts = p.split;
  }
  const int pair = unit % p.q_pairs;
  w.h = (unit / p.q_pairs) % p.heads;
  w.b = unit / (p.q_pairs * p.heads);
  w.q0 = pair * kQTiles * kBM;
  w.nqt = (p.q_tokens - w.q0 > kBM) ? 2 : 1;
  w.j0 = (int)((int64_t)idx * p.total_tiles / nparts);
  w.n = (int)((int64_t)(idx + 1) * p.total_tiles / nparts) - w.j0;
  w.part = part;
  w.rev = part < 0 && odd_wave(p);
  return w;
}

struct Shared {
  uint64_t q_full;
  uint64_t k_full[kKStages], k_empty[kKStages];
  uint64_t v_full[kVStages], v_empty[kVStages];
  uint64_t s_full[kQTiles], p_free[kQTiles];
  uint64_t o_full, drain;
  uint32_t tmem_base;
  int abort;
  uint64_t wait_limit_ns;
};

template <int D>
struct Layout {
  static constexpr int kNB = D / 64;  // boxes per tile
  __host__ __device__ static constexpr int q(int t, int bx) { return (t * kNB + bx) * kBox; }
  __host__ __device__ static constexpr int k(int s, int bx) {
    return ((kQTiles + s) * kNB + bx) * kBox;
  }
  __host__ __device__ static constexpr int v(int s, int bx) {
    return ((kQTiles + kKStages + s) * kNB + bx) * kBox;
  }
  static constexpr int shared_off = (kQTiles + kKStages + kVStages) * kNB * kBox;
  static constexpr int bytes = shared_off + 1024 /*Shared*/ + 1024 /*align*/;
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Bounded wait.  Returns false when this wait timed out or another role
// already aborted; the first timeout records the error.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity,
                                      Shared* S, int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*reinterpret_cast<volatile int*>(&S->abort)) return false;
    if (global_timer_ns() - t0 > S->wait_limit_ns) {
      *reinterpret_cast<volatile int*>(&S->abort) = 1;
      if (status != nullptr) atomicExch(status, kDevTimeout);
      return false;
    }
  }
}

// Bounded wait that ignores the abort flag (draining in-flight work).
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity,
                                           const Shared* S) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > S->wait_limit_ns) return;
  }
}

// One-shot: key tile j of the unit range [kv0, kv1) (map 0).
__device__ __forceinline__ void oneshot_tile(int kv0, int kv1, int j,
                                             int& seg, int& tok0, int& valid) {
  seg = 0;
  tok0 = kv0 + j * kBN;
  valid = min(kBN, kv1 - tok0);
}

__device__ __forceinline__ void tile_coord(const TcParams& p, int j, int& seg,
                                           int& tok0, int& valid) {
  seg = j < p.seg_tiles0 ? 0 : 1;
  const int jj = seg ? j - p.seg_tiles0 : j;
  tok0 = p.seg_start[seg] + jj * kBN;
  valid = min(kBN, p.seg_len[seg] - jj * kBN);
}

// TMA producers, one thread each: the K producer also loads the query tiles.
// K and V advance independently, so a slow V slot never holds back the next
// K tile (QK^T of tile j+1 is issued before PV of tile j completes).
template <int D, bool kIsK, bool kOneShot>
__device__ void producer(const TcParams& p, uint8_t* smem, Shared* S,
                         const Work& w) {
  const int h = w.h, b = w.b;
  using L = Layout<D>;
  constexpr int kStages = kIsK ? kKStages : kVStages;
  uint64_t* full = kIsK ? S->k_full : S->v_full;
  uint64_t* empty = kIsK ? S->k_empty : S->v_empty;
  // The query tiles are read by this CTA alone (evict first); the K and V
  // tiles of a head are read by every unit of the head (evict last).
  const uint64_t keep = l2_policy_evict_last();
  if (kIsK) {
    tma_prefetch_desc(&p.q_map);
    const uint64_t once = l2_policy_evict_first();
    mbar_arrive_expect_tx(&S->q_full, w.nqt * L::kNB * kBox);
    for (int t = 0; t < w.nqt; ++t)
      for (int bx = 0; bx < L::kNB; ++bx)
        tma_load_4d_hint(&p.q_map, smem + L::q(t, bx), &S->q_full, bx * 64,
                         w.q0 + t * kBM, h, b, once);
  }
  for (int s = 0; s < kMaxSegments; ++s)
    tma_prefetch_desc(kIsK ? &p.k_map[s] : &p.v_map[s]);
  int issued = 0;
  for (int j = 0; j < w.n; ++j) {
    const int st = j % kStages;
    const uint32_t ph = (j / kStages) & 1;
    int seg, tok0, valid;
    const int jt = w.rev ? w.n - 1 - j : j;
    if (kOneShot)
      oneshot_tile(w.kv0, w.kv1, jt, seg, tok0, valid);
    else
      tile_coord(p, w.j0 + jt, seg, tok0, valid);
    if (!wait_bar(&empty[st], ph ^ 1, S, p.status)) break;
    mbar_arrive_expect_tx(&full[st], L::kNB * kBox);
    for (int bx = 0; bx < L::kNB; ++bx)
      tma_load_4d_hint(kIsK ? &p.k_map[seg] : &p.v_map[seg],
                       smem + (kIsK ? L::k(st, bx) : L::v(st, bx)), &full[st],
                       bx * 64, tok0, h, b, keep);
    ++issued;
  }
  // Every issued load has landed before the CTA may exit (a no-op wait in
  // normal operation: consumers already waited for them).
  if (kIsK) drain_wait(&S->q_full, 0, S);
  for (int i = max(0, issued - kStages); i < issued; ++i)
    drain_wait(&full[i % kStages], (i / kStages) & 1, S);
}

// The issuing warp's waits: every lane polls and each decision (phase
// complete, abort seen, time limit passed) is a warp vote, so the warp
// never diverges and reaches the elected MMA instructions converged.  A
// phase that has already completed costs one try_wait and one vote.
__device__ __forceinline__ bool wait_bar_warp(uint64_t* bar, uint32_t parity,
                                              Shared* S, int* status) {
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
        if (status != nullptr) atomicExch(status, kDevTimeout);
      }
      __syncwarp();
      return false;
    }
  }
}

// Hand-offs from the softmax warps to the MMA warp go through named
// barriers, which live in hardware rather than in shared memory: an mbarrier
// poll is a shared-memory access, and while SMEM x SMEM MMAs are queued every
// such access waits behind their operand reads (~200 clk), which the issuer
// cannot afford several times per key tile.  A named barrier has no time
// limit, so the softmax warps make exactly the arrivals the MMA warp will
// wait for on every path, also after a failed wait (see softmax_role).
__device__ __forceinline__ void named_arrive(int id) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "n"(kHandoff) : "memory");
}
__device__ __forceinline__ void named_sync(int id) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "n"(kHandoff) : "memory");
}
__device__ __forceinline__ void relay_arrive(int id) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "n"(kRelay) : "memory");
}
// The four softmax warps of one query tile (128 threads), and no other warp.
__device__ __forceinline__ void tile_sync(int id) {
  asm volatile("bar.sync %0, 128;" ::"r"(id) : "memory");
}
__device__ __forceinline__ void relay_sync(int id) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "n"(kRelay) : "memory");
}

// The relay warp observes the TMA completions in the order the MMA warp
// needs them (K(j), then V(j - 1)) and hands each over through the named
// barrier of its ring stage, so the MMA warp itself never polls a
// shared-memory barrier.  A stage's barrier cannot be arrived at twice
// before the MMA warp has synced on it: the producer refills the stage only
// after the MMAs that read it.  After a failed wait the remaining arrivals
// are still made (the MMA warp then computes on undefined data, and the
// failure is recorded), so the MMA warp never waits for one that does not
// come.
__device__ void relay_role(const TcParams& p, Shared* S, int n) {
  int k_arr = 0, v_arr = 0;
  bool ok = true;
  for (int j = 0; ok && j <= n; ++j) {
    if (j < n) {
      if (!(ok = wait_bar_warp(&S->k_full[j % kKStages], (j / kKStages) & 1,
                               S, p.status)))
        break;
      relay_arrive(kBarKFull0 + j % kKStages);
      ++k_arr;
    }
    const int jp = j - 1;
    if (jp >= 0) {
      if (!(ok = wait_bar_warp(&S->v_full[jp % kVStages],
                               (jp / kVStages) & 1, S, p.status)))
        break;
      relay_arrive(kBarVFull0 + jp % kVStages);
      ++v_arr;
    }
  }
  for (; k_arr < n; ++k_arr) relay_arrive(kBarKFull0 + k_arr % kKStages);
  for (; v_arr < n; ++v_arr) relay_arrive(kBarVFull0 + v_arr % kVStages);
}

template <int D>
__device__ void mma_issuer(const TcParams& p, uint8_t* smem, Shared* S,
                           uint32_t tmem, const Work& w) {
  using L = Layout<D>;
  constexpr uint32_t kIdescQK = idesc_bf16_f32(kBM, kBN, 0);
  constexpr uint32_t kIdescPV = idesc_bf16_f32(kBM, D, 1);
  const uint32_t sbase = smem_addr(smem);
  const int n = w.n;
  const bool two = w.nqt == 2;

  // One warp issues every MMA (an elected lane, the warp kept converged) and
  // a tcgen05.mma takes it ~54 clk to issue against 64 clk of tensor work
  // (M128 N128 K16), so the issue loop carries no descriptor arithmetic: the
  // descriptor words are formed once here and each MMA only adds a constant
  // offset (16-byte units) to the low word.
  const uint32_t hi = desc_hi_sw128(1024);
  const uint32_t q_lo = desc_lo(sbase + L::q(0, 0), 16);
  const uint32_t k_lo = desc_lo(sbase + L::k(0, 0), 16);
  const uint32_t v_lo = desc_lo(sbase + L::v(0, 0), kBox);
  constexpr uint32_t kStage16 = (uint32_t)(L::kNB * kBox) >> 4;
  // S = Q_t K^T into the shared S columns: both operands K-major, 128-byte
  // swizzle; a K step of 16 elements is 32 bytes inside a 64-column box.
  auto qk = [&](int t, int st) {
    const uint32_t a0 = q_lo + (uint32_t)(L::q(t, 0) >> 4);
    const uint32_t b0 = k_lo + (uint32_t)st * kStage16;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
      const uint32_t off = (uint32_t)((ks / 4) * kBox + (ks % 4) * 32) >> 4;
      mma_ss_warp(tmem + kTmemS, a0 + off, b0 + off, hi, kIdescQK, ks > 0);
    }
  };
  // O_t += P_t V: P_t from its TMEM columns (8 per 16 keys), V MN-major (d
  // contiguous): 16 keys are two 8-row groups (2048 bytes), the two 64-column
  // halves of d are one box apart.
  auto pv = [&](int t, int st, int acc) {
    const uint32_t b0 = v_lo + (uint32_t)st * kStage16;
#pragma unroll
    for (int kk = 0; kk < kBN / 16; ++kk)
      mma_ts_warp(tmem + kTmemO + t * 128, tmem + kTmemP + t * 64 + kk * 8,
                  b0 + (uint32_t)(kk * 2048 >> 4), hi, kIdescPV,
                  (acc | kk) != 0);
  };
  // The k-th QK^T (of either tile) may overwrite S once the softmax warps
  // have read the previous one into registers (generation k - 1 of the S
  // barrier).
  int s_uses = 0;
  auto take_s = [&]() {
    if (s_uses > 0) named_sync(kBarSFree);
    ++s_uses;
    tc_fence_after();
  };

  // Test hook: o_full receives no arrival before the end of the stream, so
  // this wait runs out and exercises the abort path.
  bool ok = !p.inject_stall || wait_bar_warp(&S->o_full, 0, S, p.status);
  ok = ok && wait_bar_warp(&S->q_full, 0, S, p.status);
  // Issue order per key tile j: QK_0(j), PV_0(j-1), QK_1(j), PV_1(j-1).  A
  // tile's PV runs one key tile behind its QK^T, so the softmax of S_t(j)
  // has the MMAs of three other steps (about 2000 clk) to produce P_t(j)
  // before the pipe needs it, while S, which only has to survive until the
  // softmax has loaded it, alternates between the tiles.
  for (int j = 0; ok && j <= n; ++j) {
    const bool has_qk = j < n;
    const int st = j % kKStages;
    const int jp = j - 1;  // the key tile whose PV runs now
    const int vs = jp % kVStages;
    if (has_qk) {
      relay_sync(kBarKFull0 + st);
      take_s();
      qk(0, st);
      mma_commit_warp(&S->s_full[0]);
      if (!two) mma_commit_warp(&S->k_empty[st]);
    }
    if (jp >= 0) {
      relay_sync(kBarVFull0 + vs);
      named_sync(kBarPFull0);
      tc_fence_after();
      pv(0, vs, jp > 0);
      mma_commit_warp(&S->p_free[0]);
      if (!two) mma_commit_warp(&S->v_empty[vs]);
    }
    if (two) {
      if (has_qk) {
        take_s();
        qk(1, st);
        mma_commit_warp(&S->s_full[1]);
        mma_commit_warp(&S->k_empty[st]);
      }
      if (jp >= 0) {
        named_sync(kBarPFull0 + 1);
        tc_fence_after();
        pv(1, vs, jp > 0);
        mma_commit_warp(&S->p_free[1]);
        mma_commit_warp(&S->v_empty[vs]);
      }
    }
  }
  if (ok) mma_commit_warp(&S->o_full);
  mma_commit_warp(&S->drain);
  if ((threadIdx.x & 31) == 0) drain_wait(&S->drain, 0, S);
  __syncwarp();
}

__device__ __forceinline__ uint64_t f2_pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// P = 2^(s * scale_log2 - m) for the 32 columns of s[c] (a packed FFMA per
// pair, one MUFU ex2 per element), packed as 16 bf16 pairs; the row sums go
// to four independent packed accumulators.
__device__ __forceinline__ void exp_pack32(const uint32_t (&sc)[32],
                                           uint64_t sl2x2, uint64_t neg2,
                                           uint32_t (&pk)[16],
                                           uint64_t (&acc)[4]) {
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const uint64_t x2 = f2_fma(f2_pack(__uint_as_float(sc[2 * i]),
                                       __uint_as_float(sc[2 * i + 1])),
                               sl2x2, neg2);
    float x0, x1;
    f2_unpack(x2, x0, x1);
    const float p0 = ex2(x0), p1 = ex2(x1);
    acc[i & 3] = f2_add(acc[i & 3], f2_pack(p0, p1));
    pk[i] = pack_bf16(p0, p1);
  }
}

__device__ __forceinline__ float acc_total(const uint64_t (&acc)[4]) {
  float a0, a1, b0, b1, c0, c1, d0, d1;
  f2_unpack(acc[0], a0, a1);
  f2_unpack(acc[1], b0, b1);
  f2_unpack(acc[2], c0, c1);
  f2_unpack(acc[3], d0, d1);
  return ((a0 + a1) + (b0 + b1)) + ((c0 + c1) + (d0 + d1));
}

// Mask columns >= valid of s[c] (the ragged end of a segment) and fold the
// row max of s[c] into four independent accumulators.
__device__ __forceinline__ void mask_max32(uint32_t (&sc)[32], int c, int valid,
                                           float (&mx)[4]) {
  if (valid < (c + 1) * 32) {
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (c * 32 + i >= valid) sc[i] = 0xff800000u;  // -inf
  }
#pragma unroll
  for (int i = 0; i < 16; ++i)
    mx[i & 3] = max3(mx[i & 3], __uint_as_float(sc[2 * i]),
                     __uint_as_float(sc[2 * i + 1]));
}

// One-shot: mask the columns of s[c] outside this row's visible range
// [lo, hi) (relative to the tile) and fold the row max as mask_max32 does.
__device__ __forceinline__ void mask_range_max32(uint32_t (&sc)[32], int c,
                                                 int lo, int hi,
                                                 float (&mx)[4]) {
  if (lo > c * 32 || hi < (c + 1) * 32) {
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (c * 32 + i < lo || c * 32 + i >= hi) sc[i] = 0xff800000u;  // -inf
  }
#pragma unroll
  for (int i = 0; i < 16; ++i)
    mx[i & 3] = max3(mx[i & 3], __uint_as_float(sc[2 * i]),
                     __uint_as_float(sc[2 * i + 1]));
}

// Streaming: j0, n index the launch's visible tiles.  One-shot: the tiles of
// [kv0, kv1); a row of chunk c sees keys of chunks max(0, c - W) .. c, so a
// row can be fully masked in a tile (its reference then stays at -inf).
// Per key tile: read S (shared by both query tiles) into registers and
// release it at once, exponentiate, wait until the previous PV of this tile
// has consumed P_t (and brought O_t up to date), rescale O_t if the
// reference moved, then store P_t.
template <int D, bool kOneShot>
__device__ void softmax_role(const TcParams& p, Shared* S, uint32_t tmem,
                             int t, int nqt, int wq, int lane, int j0, int n,
                             int kv0, int kv1, int q0, bool rev) {
  const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
  const uint32_t tS = tmem + kTmemS + lane_off;
  const uint32_t tP = tmem + kTmemP + t * 64 + lane_off;
  const uint32_t tO = tmem + kTmemO + t * 128 + lane_off;
  const float sl2 = p.scale_log2;
  const uint64_t sl2x2 = f2_pack(sl2, sl2);
  float m_ref = -INFINITY;  // exp2-domain reference (scaled scores)
  float l = 0.f;
  bool ok = true;
  // Arrivals the MMA warp waits for: one per S this tile reads, except the
  // very last S of the unit (no QK^T follows it), and one per P_t.
  const int s_expected = (t == nqt - 1) ? n - 1 : n;
  int s_arrived = 0, p_arrived = 0;
  int vis_lo = 0, vis_hi = 0;  // one-shot: this row's visible key tokens
  if (kOneShot) {
    const int row = min(q0 + t * kBM + wq * 32 + lane, p.q_tokens - 1);
    const int c = row / p.chunk_tokens;
    vis_lo = p.window < 0 ? 0 : max(0, c - p.window) * p.chunk_tokens;
    vis_hi = min((c + 1) * p.chunk_tokens, p.seq_tokens);
  }
  for (int j = 0; j < n; ++j) {
    int seg, tok0, valid;
    const int jt = rev ? n - 1 - j : j;  // the producers' order
    if (kOneShot)
      oneshot_tile(kv0, kv1, jt, seg, tok0, valid);
    else
      tile_coord(p, j0 + jt, seg, tok0, valid);
    if (!(ok = wait_bar(&S->s_full[t], j & 1, S, p.status))) break;
    tc_fence_after();
    uint32_t s[4][32];
#pragma unroll
    for (int c = 0; c < 4; ++c) tmem_ld32(tS + 32 * c, s[c]);
    tmem_wait_ld();
    // S is in registers: the next QK^T (of either tile) may overwrite it.
    tc_fence_before();
    if (s_arrived < s_expected) {
      named_arrive(kBarSFree);
      ++s_arrived;
    }
    float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
    if (kOneShot) {
      const int lo = vis_lo - tok0;
      const int hi = min(vis_hi - tok0, valid);
#pragma unroll
      for (int c = 0; c < 4; ++c) mask_range_max32(s[c], c, lo, hi, mx);
    } else {
#pragma unroll
      for (int c = 0; c < 4; ++c) mask_max32(s[c], c, valid, mx);
    }
    const float mrow = fmaxf(max3(mx[0], mx[1], mx[2]), mx[3]) * sl2;
    // The reference moves only when a row max passes it by more than the
    // threshold (decided per warp: TMEM accesses are warp-wide).
    const bool rescale =
        __any_sync(0xffffffffu, mrow > m_ref + kRescaleThreshold);
    float alpha = 1.f;
    if (rescale) {
      const float m_new = fmaxf(m_ref, mrow);
      alpha = ex2(m_ref - m_new);
      if (kOneShot && m_new == -INFINITY) alpha = 1.f;  // still nothing seen
      l *= alpha;
      m_ref = m_new;
    }
    // A row that has seen no visible key yet exponentiates -inf against 0.
    const float neg = (kOneShot && m_ref == -INFINITY) ? 0.f : -m_ref;
    const uint64_t neg2 = f2_pack(neg, neg);
    uint64_t acc[4] = {0, 0, 0, 0};
    uint32_t pk[2][16];
#pragma unroll
    for (int c = 0; c < 2; ++c) exp_pack32(s[c], sl2x2, neg2, pk[c], acc);
    // P_t(j - 1) has been consumed and O_t holds PV_t(0 .. j-1) (PV_t(j-1)
    // was issued right after this S, so this normally does not wait).
    if (j > 0 && !(ok = wait_bar(&S->p_free[t], (j - 1) & 1, S, p.status)))
      break;
    tc_fence_after();
    if (rescale && j > 0) {
      // Scale O_t in place before PV_t(j) accumulates against the new
      // reference.
#pragma unroll 1
      for (int c = 0; c < D / 8; ++c) {
        uint32_t r[8];
        tmem_ld8(tO + c * 8, r);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 8; ++i)
          r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
        tmem_st8(tO + c * 8, r);
      }
    }
    tmem_st16(tP, pk[0]);
    tmem_st16(tP + 16, pk[1]);
#pragma unroll
    for (int c = 2; c < 4; ++c) {
      exp_pack32(s[c], sl2x2, neg2, pk[c - 2], acc);
      tmem_st16(tP + 16 * c, pk[c - 2]);
    }
    l += acc_total(acc);
    tmem_wait_st();
    tc_fence_before();
    named_arrive(kBarPFull0 + t);
    ++p_arrived;
  }
  // After a failed wait the remaining hand-offs are still made (their
  // contents are undefined, and so is the output), so that the MMA warp
  // never waits for an arrival that does not come.
  while (s_arrived < s_expected) {
    named_arrive(kBarSFree);
    ++s_arrived;
  }
  while (p_arrived < n) {
    named_arrive(kBarPFull0 + t);
    ++p_arrived;
  }
  const bool have = ok && wait_bar(&S->o_full, 0, S, p.status);
  const Work w = cta_work<kOneShot>(p);
  const int r_unit = t * kBM + wq * 32 + lane;  // row within the unit
  const int row = w.q0 + r_unit;
  const float inv_l = 1.f / l;
  if (w.part >= 0) {
    // Partial result of a key range: O / l in fp32 (transposed, so a warp's
    // stores are contiguous) and the log2-domain log-sum-exp.
    if (!have) return;
    tc_fence_after();
    float* ws_o = p.ws + (size_t)w.part * D * kUnitRows;
    float* ws_l = p.ws_lse + (size_t)w.part * kUnitRows;
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      uint32_t r[32];
      tmem_ld32(tO + c * 32, r);
      tmem_wait_ld();
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int64_t x = (int64_t)w.part * D * kUnitRows +
                          (int64_t)(c * 32 + i) * kUnitRows + r_unit;
        if (in_bounds(x, (int64_t)p.ws_parts * D * kUnitRows, p.status))
          ws_o[(c * 32 + i) * kUnitRows + r_unit] = __uint_as_float(r[i]) * inv_l;
      }
    }
    if (in_bounds((int64_t)w.part * kUnitRows + r_unit,
                  (int64_t)p.ws_parts * kUnitRows, p.status))
      ws_l[r_unit] = m_ref + __log2f(l);
    return;
  }
  // Whole unit: the tile's rows of O / l, as bf16, are staged in its Q tile
  // (free: every MMA has completed) as 128-byte-swizzled [128 x 64] boxes,
  // and leave as TMA tile stores (rows past the chunk fall outside the map
  // and are not written), instead of each thread writing 16-byte pieces of
  // its row at a stride of H d elements.  Every thread of the tile reaches
  // the barrier, also after a failed wait.
  uint8_t* tile = reinterpret_cast<uint8_t*>(S) - Layout<D>::shared_off +
                  Layout<D>::q(t, 0);
  const int rt = wq * 32 + lane;  // row within the tile
  if (have) {
    tc_fence_after();
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      uint32_t r[32];
      tmem_ld32(tO + c * 32, r);
      tmem_wait_ld();
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 16; ++i)
        pk[i] = pack_bf16(__uint_as_float(r[2 * i]) * inv_l,
                          __uint_as_float(r[2 * i + 1]) * inv_l);
      uint8_t* line = tile + (c / 2) * kBox + rt * 128;
#pragma unroll
      for (int q = 0; q < 4; ++q)
        *reinterpret_cast<uint4*>(line + ((((c % 2) * 4 + q) ^ (rt & 7)) << 4)) =
            make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
    }
    fence_proxy_async_smem();
  }
  tile_sync(kBarOStaged0 + t);
  if (wq == 0 && lane == 0 && have &&
      !*reinterpret_cast<volatile int*>(&S->abort)) {
    for (int bx = 0; bx < Layout<D>::kNB; ++bx)
      tma_store_4d(&p.o_map, tile + bx * kBox, bx * 64, w.q0 + t * kBM, w.h,
                   w.b);
    bulk_commit_group();
    bulk_wait_group0();
  }
  const int64_t lse_i = ((int64_t)w.b * p.heads + w.h) * p.q_tokens + row;
  if (have && p.lse != nullptr && row < p.q_tokens &&
      in_bounds(lse_i, (int64_t)p.batch * p.heads * p.q_tokens, p.status))
    p.lse[lse_i] = (m_ref + __log2f(l)) * 0.6931471805599453f;
}

// Merge the partial results of the split units: weights 2^(lse_i - m),
// O = sum_i w_i O_i / sum_i w_i, LSE = m + log2(sum_i w_i) (natural log out).
// A CTA merges a block of 32 query rows x 32 columns of one unit: thread
// (r, g) accumulates columns [4 g, 4 g + 4) of the block for row r, so a
// warp reads 32 consecutive rows of one column of a part (coalesced).  The
// parts are walked once, kPartUnroll at a time with all their loads issued
// together, the reference max moving with each group (what was accumulated
// is rescaled by 2^(m_old - m_new)): the merge reads tens of MB that are
// mostly still in L2, and it is the latency of those reads, not their
// volume, that sets its time.  The bf16 rows are written contiguously
// through shared memory.
constexpr int kMergeRows = 32;
constexpr int kMergeCols = 32;
constexpr int kMergeThreads = kMergeRows * kMergeCols / 4;  // 256
constexpr int kPartUnroll = 16;

template <int D>
__global__ void __launch_bounds__(kMergeThreads)
combine_kernel(const __grid_constant__ TcParams p) {
  constexpr int kCols = 4;  // columns per thread
  __shared__ __align__(16) uint16_t tile[kMergeRows][kMergeCols + 8];
  pdl_trigger();
  pdl_wait();  // the partial results of the attention kernel are complete
  const int ut = blockIdx.x;
  const int r = threadIdx.x % kMergeRows;
  const int g = threadIdx.x / kMergeRows;
  const int r_unit = blockIdx.y * kMergeRows + r;
  const int col0 = blockIdx.z * kMergeCols + g * kCols;
  const int unit = p.units_full + ut;
  const int pair = unit % p.q_pairs;
  const int h = (unit / p.q_pairs) % p.heads;
  const int b = unit / (p.q_pairs * p.heads);
  const int row0 = pair * kQTiles * kBM + blockIdx.y * kMergeRows;
  if (row0 >= p.q_tokens) return;  // the whole block is past the chunk end
  const int k0 = ut * p.split;
  // every part this block reads lies in the workspace
  if (!in_bounds(k0 + p.split - 1, p.ws_parts, p.status)) return;
  const float* lse = p.ws_lse + (size_t)k0 * kUnitRows + r_unit;
  float m = -INFINITY;  // reference: the max of the parts seen so far
  float acc[kCols];
#pragma unroll
  for (int x = 0; x < kCols; ++x) acc[x] = 0.f;
  float wsum = 0.f;
  const float* src0 = p.ws + ((size_t)k0 * D + col0) * kUnitRows + r_unit;
  for (int i0 = 0; i0 < p.split; i0 += kPartUnroll) {
    float w8[kPartUnroll], v[kPartUnroll][kCols];
#pragma unroll
    for (int u = 0; u < kPartUnroll; ++u) {
      const bool have = i0 + u < p.split;
      w8[u] = have ? lse[(size_t)(i0 + u) * kUnitRows] : -INFINITY;
      const float* src = src0 + (size_t)(i0 + u) * D * kUnitRows;
#pragma unroll
      for (int x = 0; x < kCols; ++x)
        v[u][x] = have ? src[(size_t)x * kUnitRows] : 0.f;
    }
    float mg = m;
#pragma unroll
    for (int u = 0; u < kPartUnroll; ++u) mg = fmaxf(mg, w8[u]);
    if (mg == -INFINITY) continue;  // nothing finite yet
    // 0 on the first finite group (nothing accumulated), else <= 1
    const float sc = m == -INFINITY ? 0.f : ex2(m - mg);
    wsum *= sc;
#pragma unroll
    for (int x = 0; x < kCols; ++x) acc[x] *= sc;
    m = mg;
#pragma unroll
    for (int u = 0; u < kPartUnroll; ++u) {
      const float wi = ex2(w8[u] - m);  // 0 for the missing parts
      wsum += wi;
#pragma unroll
      for (int x = 0; x < kCols; ++x) acc[x] = fmaf(wi, v[u][x], acc[x]);
    }
  }
  const float inv = 1.f / wsum;
#pragma unroll
  for (int x = 0; x < kCols; x += 2)
    *reinterpret_cast<uint32_t*>(&tile[r][g * kCols + x]) =
        pack_bf16(acc[x] * inv, acc[x + 1] * inv);
  const int64_t lse_i = ((int64_t)b * p.heads + h) * p.q_tokens + row0 + r;
  if (blockIdx.z == 0 && g == 0 && p.lse != nullptr && row0 + r < p.q_tokens &&
      in_bounds(lse_i, (int64_t)p.batch * p.heads * p.q_tokens, p.status))
    p.lse[lse_i] = (m + __log2f(wsum)) * 0.6931471805599453f;
  __syncthreads();
  // Each row of the block is 32 bf16 = 4 16-byte pieces; one piece per
  // thread of the first 128.
  if (threadIdx.x < kMergeRows * kMergeCols / 8) {
    const int rr = threadIdx.x / (kMergeCols / 8);
    const int piece = threadIdx.x % (kMergeCols / 8);
    const int row = row0 + rr;
    const int64_t x = (int64_t)b * p.o_str.batch + (int64_t)row * p.o_str.token +
                      (int64_t)h * p.o_str.head + blockIdx.z * kMergeCols +
                      piece * 8;
    if (row < p.q_tokens && in_bounds(x, p.o_elems - 7, p.status))
      *reinterpret_cast<uint4*>(p.o + x) =
          *reinterpret_cast<const uint4*>(&tile[rr][piece * 8]);
  }
}

template <int D, bool kOneShot>
__global__ void __launch_bounds__(kThreads, 1)
chunk_attn_tc_kernel(const __grid_constant__ TcParams p) {
  using L = Layout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Shared* S = reinterpret_cast<Shared*>(smem + L::shared_off);
  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  const Work w = cta_work<kOneShot>(p);

  if (warp == 9) {
    tmem_alloc(&S->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (threadIdx.x == 256) {
    mbar_init(&S->q_full, 1);
    for (int s = 0; s < kKStages; ++s) {
      mbar_init(&S->k_full[s], 1);
      mbar_init(&S->k_empty[s], 1);
    }
    for (int s = 0; s < kVStages; ++s) {
      mbar_init(&S->v_full[s], 1);
      mbar_init(&S->v_empty[s], 1);
    }
    for (int t = 0; t < kQTiles; ++t) {
      mbar_init(&S->s_full[t], 1);
      mbar_init(&S->p_free[t], 1);
    }
    mbar_init(&S->o_full, 1);
    mbar_init(&S->drain, 1);
    S->abort = 0;
    S->wait_limit_ns = p.wait_limit_ns ? p.wait_limit_ns : kDefaultWaitLimitNs;
    fence_barrier_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = S->tmem_base;
  // Set-up above touched no global memory; Q, K, V and the outputs may
  // belong to the previous kernel on the stream until it has completed.
  pdl_trigger();
  pdl_wait();

  if (warp == 8) {
    if (lane == 0) producer<D, true, kOneShot>(p, smem, S, w);
    __syncwarp();
  } else if (warp == 10) {
    if (lane == 0) producer<D, false, kOneShot>(p, smem, S, w);
    __syncwarp();
  } else if (warp == 9) {
    mma_issuer<D>(p, smem, S, tmem, w);
  } else if (warp == 11) {
    relay_role(p, S, w.n);
  } else {
    // A query tile that lies past the end of the chunk has no work.
    if (warp / 4 < w.nqt)
      softmax_role<D, kOneShot>(p, S, tmem, warp / 4, w.nqt, warp % 4, lane,
                                w.j0, w.n, w.kv0, w.kv1, w.q0, w.rev);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ host

// 4-D bf16 map over (x = d, token, head, batch) with a box of 64 x 128
// (one 128-byte swizzled row per token); element strides in bytes.
int sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

// Units of two query tiles: whole waves of units run whole, and the units of
// a last partial wave are cut along the keys so that every SM has work (at
// least kMinTilesPerPart key tiles per part, at most max_parts parts).
void split_units(int units, int tiles, int sms, int max_parts, int* units_full,
                 int* split) {
  const int rem = units % sms;
  int s = 1;
  if (rem > 0) {
    s = std::min(sms / rem, tiles / kMinTilesPerPart);
    s = std::min(s, std::min(kMaxParts, max_parts) / rem);
  }
  if (s >= 2) {
    *units_full = units - rem;
    *split = s;
  } else {
    *units_full = units;
    *split = 1;
  }
}

int total_tiles(const AttnParams& a) {
  int tiles = 0;
  for (int s = 0; s < a.num_segments; ++s) tiles += (a.seg_len[s] + kBN - 1) / kBN;
  return tiles;
}

bool make_map(CUtensorMap* m, const void* base, int d, int64_t tokens,
              int heads, int batch, int64_t token_stride_b,
              int64_t head_stride_b, int64_t batch_stride_b) {
  EncodeTiledFn enc = encode_tiled_fn();
  if (enc == nullptr) return false;
  const cuuint64_t dims[4] = {(cuuint64_t)d, (cuuint64_t)tokens,
                              (cuuint64_t)heads, (cuuint64_t)batch};
  const cuuint64_t strides[3] = {(cuuint64_t)token_stride_b,
                                 (cuuint64_t)head_stride_b,
                                 (cuuint64_t)batch_stride_b};
  const cuuint32_t box[4] = {64, 128, 1, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base),
             dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D>
cudaError_t launch_d(const AttnParams& a, cudaStream_t stream, int* launches) {
  TcParams p;
  memset(&p, 0, sizeof(p));
  const int64_t es = 2;  // bytes per bf16
  if (!make_map(&p.q_map, a.q, D, a.q_tokens, a.heads, a.batch,
                a.q_str.token * es, a.q_str.head * es, a.q_str.batch * es) ||
      !make_map(&p.o_map, a.o, D, a.q_tokens, a.heads, a.batch,
                a.q_str.token * es, a.q_str.head * es, a.q_str.batch * es))
    return cudaErrorInvalidValue;
  int tiles = 0;
  for (int s = 0; s < kMaxSegments; ++s) {
    const int src = s < a.num_segments ? s : 0;
    // The map ends where the segment ends: keys past it read as zeros.
    const int64_t end = a.seg_start[src] + a.seg_len[src];
    if (!make_map(&p.k_map[s], a.k, D, end, a.heads, a.batch,
                  a.kv_str.token * es, a.kv_str.head * es, a.kv_str.batch * es) ||
        !make_map(&p.v_map[s], a.v, D, end, a.heads, a.batch,
                  a.kv_str.token * es, a.kv_str.head * es, a.kv_str.batch * es))
      return cudaErrorInvalidValue;
    p.seg_start[s] = (int32_t)a.seg_start[src];
    p.seg_len[s] = s < a.num_segments ? a.seg_len[s] : 0;
    const int t = (p.seg_len[s] + kBN - 1) / kBN;
    if (s == 0) p.seg_tiles0 = t;
    tiles += t;
  }
  p.total_tiles = tiles;
  p.o = a.o;
  p.lse = a.lse;
  p.o_str = a.q_str;
  p.o_elems = a.q_str.batch * a.batch;
  p.q_tokens = a.q_tokens;
  p.heads = a.heads;
  p.batch = a.batch;
  p.ws_parts = a.workspace_parts;
  p.scale_log2 = a.scale_log2;
  p.status = a.status;
  p.wait_limit_ns = a.wait_limit_ns;
  p.inject_stall = a.inject_stall;
  p.ws = a.workspace;

  p.q_pairs = (a.q_tokens + kQTiles * kBM - 1) / (kQTiles * kBM);
  const int units = p.q_pairs * a.heads * a.batch;
  p.sms = sm_count();
  split_units(units, tiles, p.sms, a.workspace_parts, &p.units_full,
              &p.split);
  p.ws_lse = p.ws + (size_t)a.workspace_parts * D * kUnitRows;
  const int grid = p.units_full + (units - p.units_full) * p.split;
  const int smem = Layout<D>::bytes;
  cudaError_t e = cudaFuncSetAttribute(
      chunk_attn_tc_kernel<D, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
      smem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(chunk_attn_tc_kernel<D, false>, dim3(grid), dim3(kThreads),
                 smem, stream, p);
  if (e != cudaSuccess) return e;
  *launches = 1;
  if (p.split > 1) {
    e = launch_pdl(combine_kernel<D>,
                   dim3(units - p.units_full, kUnitRows / kMergeRows,
                        D / kMergeCols),
                   dim3(kMergeThreads), 0, stream, p);
    if (e != cudaSuccess) return e;
    *launches = 2;
  }
  return cudaSuccess;
}

// One unit per pair of query tiles, no key splitting: the units differ in
// length (later chunks see more keys) and run longest first.
template <int D>
cudaError_t launch_oneshot_d(const OneShotParams& a, cudaStream_t stream) {
  TcParams p;
  memset(&p, 0, sizeof(p));
  const int64_t es = 2;
  const int64_t tok = (int64_t)a.heads * D, bat = (int64_t)a.seq_tokens * tok;
  if (!make_map(&p.q_map, a.q, D, a.seq_tokens, a.heads, a.batch, tok * es,
                D * es, bat * es) ||
      !make_map(&p.k_map[0], a.k, D, a.seq_tokens, a.heads, a.batch, tok * es,
                D * es, bat * es) ||
      !make_map(&p.v_map[0], a.v, D, a.seq_tokens, a.heads, a.batch, tok * es,
                D * es, bat * es) ||
      !make_map(&p.o_map, a.o, D, a.seq_tokens, a.heads, a.batch, tok * es,
                D * es, bat * es))
    return cudaErrorInvalidValue;
  p.k_map[1] = p.k_map[0];
  p.v_map[1] = p.v_map[0];
  p.o = a.o;
  p.lse = a.lse;
  p.o_str.token = tok;
  p.o_str.head = D;
  p.o_str.batch = bat;
  p.o_elems = bat * a.batch;
  p.q_tokens = a.seq_tokens;
  p.heads = a.heads;
  p.batch = a.batch;
  p.scale_log2 = a.scale_log2;
  p.status = a.status;
  p.inject_stall = a.inject_stall;
  p.wait_limit_ns = a.wait_limit_ns;
  p.seq_tokens = a.seq_tokens;
  p.chunk_tokens = a.chunk_tokens;
  p.window = a.window;
  p.q_pairs = (a.seq_tokens + kQTiles * kBM - 1) / (kQTiles * kBM);
  p.split = 1;
  p.sms = sm_count();
  const int grid = p.q_pairs * a.heads * a.batch;
  p.units_full = grid;
  const int smem = Layout<D>::bytes;
  cudaError_t e = cudaFuncSetAttribute(
      chunk_attn_tc_kernel<D, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
      smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(chunk_attn_tc_kernel<D, true>, dim3(grid), dim3(kThreads),
                    smem, stream, p);
}

}  // namespace

cudaError_t launch_blockcausal_attn(const OneShotParams& p, cudaStream_t stream) {
  if (p.head_dim == 64) return launch_oneshot_d<64>(p, stream);
  if (p.head_dim == 128) return launch_oneshot_d<128>(p, stream);
  return cudaErrorInvalidValue;
}

int chunk_attn_parts(const AttnParams& a) {
  const int pairs = (a.q_tokens + kQTiles * kBM - 1) / (kQTiles * kBM);
  const int units = pairs * a.heads * a.batch;
  int full = 0, split = 1;
  split_units(units, total_tiles(a), sm_count(), kMaxParts, &full, &split);
  return split > 1 ? (units - full) * split : 0;
}

cudaError_t launch_chunk_attn(const AttnParams& p, cudaStream_t stream,
                              int* launches) {
  *launches = 0;
  if (p.head_dim == 64) return launch_d<64>(p, stream, launches);
  if (p.head_dim == 128) return launch_d<128>(p, stream, launches);
  return cudaErrorInvalidValue;
}

// Resolved once; C++ initialises the function-local static exactly once even
// when several host threads make their first call at the same time.
EncodeTiledFn encode_tiled_fn() {
  static const EncodeTiledFn fn = []() -> EncodeTiledFn {
    cudaDriverEntryPointQueryResult q;
    void* ptr = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<EncodeTiledFn>(ptr);
    cudaGetLastError();
    return nullptr;
  }();
  return fn;
}

}  // namespace fastvr
