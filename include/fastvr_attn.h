/*
 * fastvr_attn.h -- C ABI of the GB300 (sm_103a) chunk-wise causal attention
 * library for streaming video diffusion transformers.
 *
 * The operation (FastVR, Sec. 3.1 "Chunk-wise causal attention", Eq. 1):
 * latent frames are grouped into non-overlapping chunks of k frames; a query
 * of frame i sees a key of frame j iff floor(i/k) - floor(j/k) lies in
 * {0, ..., W}.  Eq. 1 itself is W = 1; window_chunks = -1 widens the set to
 * every earlier chunk.  Inference processes the chunks one after the other
 * and keeps the keys and values of the chunks that later queries still see in
 * a KV cache (Sec. 3.1, last paragraph), so a chunk's cost is bounded by its
 * visible window and the cache holds O(k) tokens for a bounded window.
 *
 * Per chunk c, in stream order:
 *   fastvr_kv_append(plan, K_c, V_c, f_c, stream);        // K/V into the cache
 *   fastvr_chunk_attn_fwd(plan, Q_c, O_c, lse_c, stream);  // Q_c over its window
 *
 * Conventions shared by every entry point:
 *  - The caller owns all device memory (cache, q, k, v, out, lse).  The plan
 *    owns host state only and binds the cache pointer given at plan time.
 *  - Tensors are bfloat16, contiguous, 16-byte aligned.  Per-chunk tensors are
 *    token-major [B, f*N, H, d] (the layout a fused QKV projection emits);
 *    out has the same layout; lse is float32 [B, H, f*N] (natural log).
 *  - Device pointers are CUDA device addresses on the current device; the
 *    stream argument is a cudaStream_t (NULL = legacy default stream).  Work
 *    is enqueued on that stream; nothing is synchronised by the library except
 *    in fastvr_get_status.
 *  - Errors are returned as status codes; nothing throws or aborts across the
 *    ABI.  A call that returns an error enqueues no work and leaves the plan's
 *    counters unchanged.  Device-side failures (a bounded wait that gave up;
 *    in the debug library also a failed index check)
 *    are recorded in the cache's control word and reported by
 *    fastvr_get_status.
 *  - There is no CPU fallback: on a device that is not sm_103 the first
 *    device call returns FASTVR_ERR_UNSUPPORTED.
 *  - A plan is not thread-safe; use one plan per stream of chunks.
 */
#ifndef FASTVR_ATTN_H_
#define FASTVR_ATTN_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define FASTVR_API __attribute__((visibility("default")))
#else
#define FASTVR_API
#endif

struct CUstream_st; /* cudaStream_t is struct CUstream_st* */

typedef enum {
  FASTVR_OK = 0,
  FASTVR_ERR_INVALID_ARG = 1,  /* null/misaligned pointer, bad shape, frames<1 */
  FASTVR_ERR_UNSUPPORTED = 2,  /* head_dim not 64/128, device not sm_103      */
  FASTVR_ERR_CAPACITY = 3,     /* frames > k, more chunks than max_chunks,
                                  cache buffer too small                      */
  FASTVR_ERR_SEQUENCE = 4,     /* fwd before any append; append after a
                                  ragged (final) chunk                        */
  FASTVR_ERR_CUDA = 5,         /* a CUDA runtime/driver call failed           */
  FASTVR_ERR_TIMEOUT = 6,      /* a bounded device-side wait gave up          */
  FASTVR_ERR_BOUNDS = 7        /* a device-side index or layout check failed
                                  and the access was skipped (index checks:
                                  debug library only)                        */
} fastvr_status_t;

typedef struct {
  int32_t batch;             /* B: videos or spatial tiles                    */
  int32_t heads;             /* H                                             */
  int32_t head_dim;          /* d: 64 or 128                                  */
  int32_t tokens_per_frame;  /* N: tokens of one latent frame                 */
  int32_t frames_per_chunk;  /* k: latent frames per chunk (Eq. 1)            */
  int32_t window_chunks;     /* W: earlier chunks a chunk sees; Eq. 1 is 1;
                                -1 = every earlier chunk                      */
  int32_t max_chunks;        /* capacity in chunks when window_chunks == -1;
                                ignored otherwise                             */
  float softmax_scale;       /* 0 => 1/sqrt(head_dim)                         */
} fastvr_attn_config_t;

typedef struct fastvr_plan_s* fastvr_plan_t;

/* Bytes of device memory the caller must provide for the KV cache of cfg.
 * The cache is the one of streaming inference (Sec. 3.1, last paragraph):
 * it keeps the keys and values of the chunks that later queries still see
 * under Eq. 1 with window W, so it holds O(k) tokens per head for a bounded
 * window.  Layout:
 * K and V, each [B, H, S*k*N, d] bfloat16 with S = window_chunks + 1 slots
 * (bounded window) or max_chunks slots (unbounded), then the attention
 * kernel's split-KV workspace (256 x 256 x (d + 1) floats), then a 256-byte
 * control block.  Host only; no device work.
 * Errors: INVALID_ARG (null, non-positive sizes), UNSUPPORTED (head_dim). */
FASTVR_API fastvr_status_t fastvr_kv_cache_bytes(const fastvr_attn_config_t* cfg,
                                      size_t* bytes);

/* Validate cfg and bind a caller-owned cache buffer of `bytes` bytes (device
 * memory, 256-byte aligned, at least fastvr_kv_cache_bytes).  The plan holds
 * the streaming state of Sec. 3.1 (last paragraph): the chunk counter c and
 * the ring of cache slots, from which each chunk's visible set under Eq. 1
 * (chunks max(0, c-W) .. c) is resolved on the host.  The cache
 * contents need no initialisation.  Host only: device set-up (TMA
 * descriptors, device check, clearing the control block) happens on the
 * first device call.  *out receives a new plan, released by
 * fastvr_plan_destroy.
 * Errors: INVALID_ARG, UNSUPPORTED, CAPACITY (buffer too small). */
FASTVR_API fastvr_status_t fastvr_attn_plan(const fastvr_attn_config_t* cfg,
                                 void* kv_cache, size_t bytes,
                                 fastvr_plan_t* out);

/* KV caching for streaming inference (Sec. 3.1): copy the next chunk's keys
 * and values, k_new and v_new bfloat16 [B, frames*N, H, d] token-major, into
 * cache slot (c mod S) at token offset (c mod S)*k*N of the head-major cache,
 * where c is the plan's chunk counter, then advance the counter.  The copy is
 * bit-exact.  frames is 1..k; frames < k marks the final (ragged) chunk of the
 * stream, after which appends fail until fastvr_plan_reset.
 * Errors: INVALID_ARG, CAPACITY (frames > k; unbounded window and c ==
 * max_chunks), SEQUENCE (after a ragged chunk), UNSUPPORTED, CUDA. */
FASTVR_API fastvr_status_t fastvr_kv_append(fastvr_plan_t plan, const void* k_new,
                                 const void* v_new, int32_t frames,
                                 struct CUstream_st* stream);

/* Chunk-causal attention of the most recently appended chunk c (Eq. 1 with
 * window W): q bfloat16 [B, f_c*N, H, d] token-major attends to the cached
 * keys/values of chunks max(0, c-W) .. c (all of 0..c when unbounded), with
 * softmax scale cfg.softmax_scale, accumulating in float32.  out receives
 * bfloat16 [B, f_c*N, H, d]; lse (nullable) receives float32 [B, H, f_c*N],
 * the natural-log sum of exp(scaled scores).  Only visible cache slots are
 * read.  Does not advance the chunk counter (may be repeated).
 * Errors: INVALID_ARG, SEQUENCE (no chunk appended yet), UNSUPPORTED, CUDA. */
FASTVR_API fastvr_status_t fastvr_chunk_attn_fwd(fastvr_plan_t plan, const void* q,
                                      void* out, float* lse,
                                      struct CUstream_st* stream);

/* Start a new video: chunk counter back to 0; the cache contents are ignored
 * from then on.  Host only. */
FASTVR_API fastvr_status_t fastvr_plan_reset(fastvr_plan_t plan);

/* Synchronise the device, then report (and clear) any device-side failure
 * recorded in the cache's control block: FASTVR_ERR_TIMEOUT when a bounded
 * wait inside a kernel gave up, FASTVR_ERR_CUDA when a CUDA error is pending,
 * FASTVR_OK otherwise. */
FASTVR_API fastvr_status_t fastvr_get_status(fastvr_plan_t plan);

/* Streaming state for checkpoint/resume: the number of chunks appended and
 * the frame count of the newest chunk.  Together with the cache bytes it is
 * the whole state of a stream.  Host only. */
FASTVR_API fastvr_status_t fastvr_plan_get_state(fastvr_plan_t plan, int64_t* chunks,
                                      int32_t* last_frames);
FASTVR_API fastvr_status_t fastvr_plan_set_state(fastvr_plan_t plan, int64_t chunks,
                                      int32_t last_frames);

/* The visible key set of the most recently appended chunk as at most two
 * contiguous token ranges of one head's cache [start, start+len) (the ring
 * wraps), and their total Lk.  This is the set fastvr_chunk_attn_fwd reads.
 * seg_start and seg_len must hold 2 entries.  Host only.
 * Errors: INVALID_ARG, SEQUENCE (no chunk appended). */
FASTVR_API fastvr_status_t fastvr_plan_visible(fastvr_plan_t plan, int32_t* num_segments,
                                    int64_t* seg_start, int64_t* seg_len,
                                    int64_t* visible_tokens);

/* One-shot chunk-causal attention over a whole sequence: the training form
 * of Sec. 3.1, where the entire latent sequence is processed in parallel
 * under the mask M of Eq. 1 (window cfg.window_chunks, -1 = every earlier
 * chunk).  q, k, v: bfloat16 [B, L, H, d] token-major with L = num_frames *
 * N; out bfloat16 [B, L, H, d]; lse nullable, float32 [B, H, L].  Frame f
 * belongs to chunk f / k; a ragged final chunk is simply shorter.  Each
 * block of 256 query rows reads only the keys its rows can see (invisible
 * chunks are never loaded); rows that straddle a chunk boundary are masked
 * element-wise.  No plan, no cache and no scratch memory are involved; a
 * bounded-wait timeout leaves out undefined and is reported by
 * fastvr_get_device_status.  The result
 * equals the streamed form (fastvr_kv_append + fastvr_chunk_attn_fwd, chunk
 * by chunk) up to rounding.
 * Errors: INVALID_ARG, UNSUPPORTED (head_dim, device not sm_103), CUDA. */
FASTVR_API fastvr_status_t fastvr_blockcausal_attn_fwd(
    const fastvr_attn_config_t* cfg, int32_t num_frames, const void* q,
    const void* k, const void* v, void* out, float* lse,
    struct CUstream_st* stream);

/* Scratch bytes fastvr_blockcausal_attn_bwd needs for cfg and num_frames:
 * 2 * B * H * round_up(L, 128) floats (per-row log-sum-exp and D).  Host only.
 * Errors: INVALID_ARG, UNSUPPORTED. */
FASTVR_API fastvr_status_t fastvr_blockcausal_bwd_scratch_bytes(
    const fastvr_attn_config_t* cfg, int32_t num_frames, size_t* bytes);

/* Gradients of the one-shot chunk-causal attention (the training form of
 * Sec. 3.1; the paper trains the DiT under the mask M of Eq. 1).  Inputs:
 * q, k, v, out (the forward output) and dout (its gradient), bfloat16
 * [B, L, H, d] token-major; lse, float32 [B, H, L], the forward's
 * log-sum-exp (fastvr_blockcausal_attn_fwd).  Outputs dq, dk, dv bfloat16
 * [B, L, H, d].  scratch: caller-owned device memory of at least
 * fastvr_blockcausal_bwd_scratch_bytes bytes, overwritten.  Computes
 * D = rowsum(dout * out), then dk/dv (one CTA per 128 keys, over the query
 * tiles that see them) and dq (one CTA per 128 queries); P is recomputed
 * from lse, P and dS enter the tensor cores in bfloat16, accumulation is
 * fp32.  All pointers 16-byte aligned.  A bounded-wait timeout leaves the
 * outputs undefined and is reported by fastvr_get_device_status
 * (FASTVR_ERR_TIMEOUT); so is a dynamic shared-memory base that is not
 * 1024-byte aligned, which the dK/dV kernel's 227 KB layout requires and
 * checks (FASTVR_ERR_BOUNDS, nothing computed).
 * Errors: INVALID_ARG, UNSUPPORTED, CAPACITY (scratch too small), CUDA. */
FASTVR_API fastvr_status_t fastvr_blockcausal_attn_bwd(
    const fastvr_attn_config_t* cfg, int32_t num_frames, const void* q,
    const void* k, const void* v, const void* out, const void* dout,
    const float* lse, void* dq, void* dk, void* dv, float* scratch,
    size_t scratch_bytes, struct CUstream_st* stream);

/* FastVR's one-step restoration update (Eq. `eq:one_step`, used at
 * inference and in Stage II training): z_hat = z_lq - sigma * v, with v the
 * DiT's predicted velocity at t = tau and sigma = sigma_tau (an input: the
 * shifted schedule's constants are not given in the paper).  Elementwise
 * over n elements in any layout (the same for all three buffers); z_lq and
 * z_hat are bfloat16 (dtype 0) or float32 (dtype 1), v is bfloat16.
 * Computed as one fp32 FMA per element and rounded once (round to nearest
 * even) to the output type.  z_hat may be z_lq (in place).  Pointers must be
 * 16-byte aligned device addresses.
 * Errors: INVALID_ARG, UNSUPPORTED (device not sm_103), CUDA. */
FASTVR_API fastvr_status_t fastvr_one_step_update(const void* z_lq,
                                                  const void* v, void* z_hat,
                                                  int64_t n, float sigma,
                                                  int32_t dtype,
                                                  struct CUstream_st* stream);

/* Chunk-causal attention that allocates nothing (no counterpart in the
 * paper; an interface for callers that cannot allocate device memory).
 * Callers such as serving runtimes that own all device memory through their
 * own pool, or real-time pipelines that forbid cudaMalloc/cudaFree after
 * start-up because those calls can synchronise the device, keep K and V in
 * their own buffers and cannot give the library the workspace region of
 * fastvr_kv_cache_bytes.  This entry point needs neither a plan nor that
 * region: its scratch (the partial results of query units whose key range
 * is split across SMs, and a status word) is a fixed 24 MiB array in device
 * memory, part of the library image, which every GPU that loads the library
 * holds until the process exits.
 *   q        bf16 [B, q_frames*N, H, d] token-major (cfg: B, H, d, N, scale;
 *            frames_per_chunk, window_chunks and max_chunks are not used)
 *   k_cache, v_cache  bf16 [B, H, cache_tokens, d] head-major (any buffers
 *            of the caller, e.g. a plan's cache regions)
 *   num_segments (1..2), seg_start, seg_len: the visible key ranges of one
 *            head's cache, as fastvr_plan_visible reports them
 *   out      bf16 [B, q_frames*N, H, d]; lse nullable, float32 [B, H, Lq]
 * The result equals fastvr_chunk_attn_fwd's for the same inputs (same
 * kernels, same work split).  The first call on each device resolves the
 * array's device address (a symbol lookup, no allocation): make that first
 * call before any stream capture.  Every call on a device shares the array
 * and it keeps the last call's contents (nothing in it needs clearing:
 * every partial result is written before it is read), so calls that overlap
 * on the GPU (other streams, other threads) race: serialise them.  A bounded-wait timeout leaves out undefined and is
 * recorded in the per-device status word that fastvr_get_device_status
 * reports.  No cudaMalloc, cudaFree or allocating library routine is
 * called.  Limits: q_frames * N and every seg_start + seg_len at most
 * 2^30 - 1 (the kernels index tokens in 32 bits); softmax_scale finite.
 * Errors: INVALID_ARG (null or misaligned pointers, bad sizes or ranges),
 * UNSUPPORTED (head_dim, device not sm_103), CAPACITY (the call's split
 * needs more partial results than the array holds: 190 at d = 128, 378 at
 * d = 64), CUDA. */
FASTVR_API fastvr_status_t fastvr_chunk_attn_fwd_static(
    const fastvr_attn_config_t* cfg, const void* q, int32_t q_frames,
    const void* k_cache, const void* v_cache, int64_t cache_tokens,
    int32_t num_segments, const int64_t* seg_start, const int64_t* seg_len,
    void* out, float* lse, struct CUstream_st* stream);

/* Number of kernel launches this plan has enqueued since it was created
 * (an append is one launch; an attention call is one, or two when the key
 * range of some query units is split across SMs and merged).  Host only. */
FASTVR_API fastvr_status_t fastvr_plan_launch_count(fastvr_plan_t plan,
                                                    int64_t* launches);

/* Failure-detection hook (tests).  stall != 0 makes the next attention
 * launches of this plan wait, in the MMA-issuing warp, on a barrier that
 * nothing arrives on; the kernel's bounded wait runs out after
 * wait_limit_ns, every role stops, in-flight copies and MMAs are drained,
 * tensor memory is released and FASTVR_ERR_TIMEOUT is recorded for
 * fastvr_get_status.  The output of such a launch is undefined.  No GPU
 * fault or hang results.  wait_limit_ns = 0 keeps the default limit
 * (4 s per wait); stall = 0 with wait_limit_ns = 0 restores normal
 * operation.  Host only.  Errors: INVALID_ARG. */
FASTVR_API fastvr_status_t fastvr_debug_inject_stall(fastvr_plan_t plan,
                                                     int32_t stall,
                                                     uint64_t wait_limit_ns);

/* Device-side failures of the calls without a plan (the one-shot forward
 * fastvr_blockcausal_attn_fwd, the backward fastvr_blockcausal_attn_bwd and
 * the allocation-free fastvr_chunk_attn_fwd_static):
 * a bounded wait that gave up — or, in the debug library, a failed index
 * check — is recorded in a status word of the current device, shared by all
 * such calls on it.  This call waits for the device to finish (it
 * synchronises), returns FASTVR_ERR_TIMEOUT or FASTVR_ERR_BOUNDS for a
 * recorded failure and clears the word, FASTVR_OK otherwise.  The outputs
 * of a call that failed this way are undefined.  Errors: CUDA. */
FASTVR_API fastvr_status_t fastvr_get_device_status(void);

/* Failure-detection hook (tests) for the calls without a plan, process-wide:
 * stall != 0 makes every following one-shot forward and backward launch
 * wait, in its MMA-issuing warp, on a barrier that nothing arrives on; the
 * bounded wait runs out after wait_limit_ns (0 = the 4 s default), every
 * role stops, in-flight copies and MMAs are drained, tensor memory is
 * released and FASTVR_ERR_TIMEOUT is recorded for fastvr_get_device_status.
 * No GPU fault or hang results.  stall = 0 restores normal operation.
 * Host only; always FASTVR_OK. */
FASTVR_API fastvr_status_t fastvr_debug_inject_stall_noplan(
    int32_t stall, uint64_t wait_limit_ns);

/* Index-check hook (tests of the debug library).  The debug library,
 * libfastvr_attn_debug.so (built with FASTVR_BOUNDS_CHECK), checks every
 * computed global-memory index of the append and attention kernels before
 * the access; a failed check skips the access and records
 * FASTVR_ERR_BOUNDS for fastvr_get_status.  This call makes the next
 * fastvr_kv_append of the plan write its chunk `tokens` cache tokens past
 * the start of its slot (0 <= tokens <= k * N), a deliberately wrong
 * destination for those checks to catch: every write they let through
 * stays inside the plan's cache buffer.  The cache contents are undefined
 * afterwards (reset the plan).  Host only.  Errors: INVALID_ARG (tokens out
 * of range), UNSUPPORTED (the release library, which has no checks). */
FASTVR_API fastvr_status_t fastvr_debug_shift_next_append(fastvr_plan_t plan,
                                                          int64_t tokens);

/* Release a plan (host memory only; the cache stays the caller's). */
FASTVR_API void fastvr_plan_destroy(fastvr_plan_t plan);

/* A static, human-readable name for a status code. */
FASTVR_API const char* fastvr_status_string(fastvr_status_t status);

#ifdef __cplusplus
}
#endif

#endif /* FASTVR_ATTN_H_ */
