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
// Each thread keeps eight loads in flight before it stores (enough bytes in
// flight to cover HBM latency with a few CTAs per SM); the source is read
// with an evict-first hint since it is not read again.
#include "fastvr_internal.h"

namespace fastvr {
namespace {

constexpr int kUnroll = 8;

template <int VPR>  // 16-byte vectors per (token, head) row: d / 8
__device__ __forceinline__ int64_t cache_index(const AppendParams& p,
                                               uint32_t j) {
  const uint32_t vec = j % VPR;
  const uint32_t r = j / VPR;  // (b, t, h) row, h fastest
  const uint32_t h = r % (uint32_t)p.heads;
  const uint32_t bt = r / (uint32_t)p.heads;
  const uint32_t t = bt % (uint32_t)p.tokens;
  const uint32_t b = bt / (uint32_t)p.tokens;
#ifdef FASTVR_BOUNDS_CHECK
  // a destination token past this head's cache is out of bounds even when
  // the flat index still lands inside the buffer
  if (p.token_offset + t >= p.cache_tokens) return -1;
#endif
  return (((int64_t)b * p.heads + h) * p.cache_tokens + p.token_offset + t) *
             VPR + vec;
}

// blockIdx.y selects K (0) or V (1).
template <int VPR>
__global__ void __launch_bounds__(256) kv_append_kernel(AppendParams p) {
  pdl_trigger();
  pdl_wait();  // the chunk's K/V and the slot's previous readers are done
  const uint4* src =
      reinterpret_cast<const uint4*>(blockIdx.y ? p.v_new : p.k_new);
  uint4* dst = reinterpret_cast<uint4*>(blockIdx.y ? p.v_cache : p.k_cache);
  const uint32_t n = (uint32_t)p.batch * p.tokens * p.heads * VPR;
  const int64_t cache_vecs = (int64_t)p.batch * p.heads * p.cache_tokens * VPR;
  const uint32_t stride = gridDim.x * blockDim.x;
  // Every pass issues all of its (predicated) loads before the first store,
  // also the last, partial one: a small chunk gives each thread only a few
  // vectors, and one load at a time would leave it latency-bound.  Indices
  // stay below n + kUnroll * stride, which the launch keeps within 32 bits.
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += kUnroll * stride) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (i + u * stride < n) v[u] = __ldcs(src + i + u * stride);
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      if (i + u * stride >= n) break;
      const int64_t c = cache_index<VPR>(p, i + u * stride);
      if (in_bounds(c, cache_vecs, p.status)) dst[c] = v[u];
    }
  }
}

}  // namespace

cudaError_t launch_kv_append(const AppendParams& p, cudaStream_t stream) {
  const int vpr = p.head_dim / 8;
  const int64_t n = (int64_t)p.batch * p.tokens * p.heads * vpr;
  if (n == 0) return cudaSuccess;
  if (n > 0x7fffffffLL) return cudaErrorInvalidValue;  // 32-bit indexing
  // (n < 2^31 and kUnroll * stride < 2^31: i + u * stride never wraps)
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms <= 0) sms = 152;
  // Four CTAs of 256 threads per SM and tensor, never more than the work.
  int64_t blocks = (int64_t)sms * 4;
  const int64_t need = (n + 255) / 256;
  if (blocks > need) blocks = need;
  const dim3 grid((unsigned)blocks, 2);
  if (vpr == 16)
    return launch_pdl(kv_append_kernel<16>, grid, dim3(256), 0, stream, p);
  if (vpr == 8)
    return launch_pdl(kv_append_kernel<8>, grid, dim3(256), 0, stream, p);
  return cudaErrorInvalidValue;
}

}  // namespace fastvr
