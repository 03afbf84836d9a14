// Internal interfaces between the host library (fastvr_host.cpp) and the
// CUDA kernels.  Not part of the public ABI.
#pragma once

#include <cuda.h>  // CUtensorMap types (the driver itself is reached
                   // through the runtime's entry-point query)
#include <cuda_runtime.h>
#include <stdint.h>

namespace fastvr {

// At most two contiguous token ranges of one head's cache make up the keys a
// chunk sees: the visible chunk slots are consecutive modulo the ring size
// and only the newest chunk can be partly filled (Eq. 1 at chunk granularity,
// Sec. 3.1 KV caching).
constexpr int kMaxSegments = 2;

// Split-KV workspace of the attention kernel: at most kMaxParts partial
// results of 256 query rows, each d fp32 outputs plus one log-sum-exp.
constexpr int kMaxParts = 256;
constexpr int kUnitRows = 256;
inline size_t workspace_bytes(int head_dim) {
  return (size_t)kMaxParts * kUnitRows * (head_dim + 1) * sizeof(float);
}

// cuTensorMapEncodeTiled, looked up through the CUDA runtime's driver entry
// point (the library links the runtime statically and not libcuda); null
// when the driver does not provide it.
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType,
                                  cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled_fn();

// Error codes a kernel writes into the cache's control block.
constexpr int kDevOk = 0;
constexpr int kDevTimeout = 1;
constexpr int kDevBounds = 2;  // an index check (debug builds) or a layout
                               // check failed

#ifdef __CUDACC__
// Debug builds (-DFASTVR_BOUNDS_CHECK, libfastvr_attn_debug.so) check every
// computed global-memory index of the streaming path before the access: an
// index outside [0, n) records kDevBounds in the status word (the first
// error wins) and the access is skipped.  Release builds compile the check
// away.  compute-sanitizer is not available, and a trap or failed assert
// would take the GPU down with it.
#ifdef FASTVR_BOUNDS_CHECK
__device__ __forceinline__ bool in_bounds(int64_t i, int64_t n, int* status) {
  if (i >= 0 && i < n) return true;
  if (status != nullptr) atomicCAS(status, kDevOk, kDevBounds);
  return false;
}
#else
__device__ __forceinline__ bool in_bounds(int64_t, int64_t, int*) {
  return true;
}
#endif
#endif

#ifdef __CUDACC__
// Programmatic dependent launch.  The streaming kernels (append, attention,
// split merge) and the one-step update are launched with programmatic stream
// serialization, so a kernel may become resident and do its set-up (barrier
// and TMEM initialisation) while the previous kernel on the stream drains.
// Each of them executes pdl_wait() before its first global-memory access
// that a preceding kernel may produce or still read (the wait returns once
// that kernel has completed and its writes are visible), and pdl_trigger()
// early, so that the next kernel's launch can begin.
__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block,
                              size_t smem, cudaStream_t stream,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}
#endif

// Strided view of a bfloat16 [B, L, H, d] token-major tensor or of a head-major
// cache [B, H, L, d]: element (b, t, h, x) lives at
// base + b*batch + t*token + h*head + x (strides in elements).
struct Strides {
  int64_t batch, token, head;
};

struct AppendParams {
  const uint16_t* k_new;  // [B, L, H, d] token-major
  const uint16_t* v_new;
  uint16_t* k_cache;      // [B, H, cache_tokens, d] head-major
  uint16_t* v_cache;
  int32_t batch, tokens, heads, head_dim;
  int64_t cache_tokens;   // tokens per head in the cache (S * k * N)
  int64_t token_offset;   // first cache token of the destination slot
  int* status;            // control block word (bounds checks), or null
};

struct AttnParams {
  const uint16_t* q;      // bfloat16 [B, Lq, H, d] token-major
  uint16_t* o;            // bfloat16 [B, Lq, H, d] token-major
  float* lse;             // float32 [B, H, Lq] or null
  const uint16_t* k;      // keys: head-major cache view
  const uint16_t* v;      // values: same layout as k
  Strides q_str;          // strides of q and o
  Strides kv_str;         // strides of k and v
  int32_t batch, heads, head_dim, q_tokens;
  int64_t kv_tokens;      // tokens per head addressable through k/v
  int32_t num_segments;
  int64_t seg_start[kMaxSegments];
  int32_t seg_len[kMaxSegments];
  float scale_log2;       // softmax_scale * log2(e)
  int* status;            // control word (device)
  float* workspace;       // split-KV scratch (device): workspace_parts
                          // partial results of kUnitRows x (d + 1) floats
  int32_t workspace_parts;
  uint64_t wait_limit_ns; // bound of every in-kernel wait (0 = default)
  int32_t inject_stall;   // test hook: stall the MMA issuer until timeout
};

cudaError_t launch_kv_append(const AppendParams& p, cudaStream_t stream);
// The one-step update z_hat = z - sigma * v over n elements; z and out are
// bf16 (dtype 0) or float32 (dtype 1), v is bf16.
cudaError_t launch_one_step(const void* z, const void* v, void* out, int64_t n,
                            float sigma, int dtype, cudaStream_t stream);

// One-shot (training-form) attention over a whole token-major sequence.
struct OneShotParams {
  const uint16_t* q;      // bfloat16 [B, L, H, d] token-major
  const uint16_t* k;
  const uint16_t* v;
  uint16_t* o;            // bfloat16 [B, L, H, d]
  float* lse;             // float32 [B, H, L] or null
  int32_t batch, heads, head_dim;
  int32_t seq_tokens;     // L = frames * tokens per frame
  int32_t chunk_tokens;   // k * N
  int32_t window;         // W, -1 = unbounded
  float scale_log2;
  int* status;            // device status word or null (not reported)
  int32_t inject_stall;   // failure-detection test hook
  uint64_t wait_limit_ns; // 0 = kernel default
};
cudaError_t launch_blockcausal_attn(const OneShotParams& p, cudaStream_t stream);

// Backward of the one-shot attention.
struct BwdArgs {
  const uint16_t *q, *k, *v, *out, *dout;  // bf16 [B, L, H, d] token-major
  const float* lse;                        // forward LSE [B, H, L]
  uint16_t *dq, *dk, *dv;                  // bf16 [B, L, H, d]
  float* scratch;  // 2 * B * H * round_up(L, 128) floats
  int32_t batch, heads, head_dim, seq_tokens, chunk_tokens, window;
  float scale;
  int* status;             // device status word or null (not reported)
  int32_t inject_stall;    // failure-detection test hook
  uint64_t wait_limit_ns;  // 0 = kernel default
};
cudaError_t launch_blockcausal_attn_bwd(const BwdArgs& a, cudaStream_t stream);

// The status word of the current device for the calls without a plan (the
// one-shot forward and the backward), or null if it cannot be looked up.
int* device_status_word();

// Workspace parts (partial results) a launch of p uses on the current device
// (0 when no unit is split), with at most kMaxParts parts.
int chunk_attn_parts(const AttnParams& p);
// Enqueues the attention kernel (and the merge kernel when the key range of
// some units is split); *launches receives the number of kernels enqueued.
cudaError_t launch_chunk_attn(const AttnParams& p, cudaStream_t stream,
                              int* launches);

}  // namespace fastvr
