// KV-cache append for streaming chunk-causal attention (Sec. 3.1: during
// inference chunks are restored one after the other with KV caching).
//
// Moves one chunk's keys and values from the token-major layout a QKV
// projection emits, [B, L, H, d], into the head-major ring-buffer cache
// [B, H, S*k*N, d] at the chunk's slot.  The copy is bit-exact and purely
// bandwidth-bound: every byte is read once and written once with 16-byte
// vector accesses.  Consecutive threads read consecutive 16-byte pieces of the
// source, and the d/8 pieces of one (token, head) row land contiguously in the
// cache, so both sides are fully coalesced at 32-byte sector granularity.
#include "fastvr_internal.h"

namespace fastvr {
namespace {

__global__ void __launch_bounds__(256)
kv_append_kernel(AppendParams p) {
  const int vec_per_row = p.head_dim / 8;  // 16-byte vectors per (t, h) row
  const int64_t per_tensor =
      (int64_t)p.batch * p.tokens * p.heads * vec_per_row;
  const int64_t total = 2 * per_tensor;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += stride) {
    const bool is_v = i >= per_tensor;
    const int64_t j = is_v ? i - per_tensor : i;
    const int vec = (int)(j % vec_per_row);
    int64_t r = j / vec_per_row;
    const int h = (int)(r % p.heads);
    r /= p.heads;
    const int64_t t = r % p.tokens;
    const int64_t b = r / p.tokens;
    const uint4* src = reinterpret_cast<const uint4*>(is_v ? p.v_new : p.k_new);
    uint4* dst = reinterpret_cast<uint4*>(is_v ? p.v_cache : p.k_cache);
    const int64_t d_idx =
        ((b * p.heads + h) * p.cache_tokens + p.token_offset + t) * vec_per_row +
        vec;
    dst[d_idx] = __ldg(src + j);
  }
}

}  // namespace

cudaError_t launch_kv_append(const AppendParams& p, cudaStream_t stream) {
  const int64_t total =
      2LL * p.batch * p.tokens * p.heads * (p.head_dim / 8);
  if (total == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms <= 0) sms = 152;
  // Enough resident threads to cover HBM latency: 8 CTAs of 256 per SM,
  // never more CTAs than work.
  int64_t blocks = (int64_t)sms * 8;
  const int64_t need = (total + 255) / 256;
  if (blocks > need) blocks = need;
  kv_append_kernel<<<(unsigned)blocks, 256, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace fastvr
