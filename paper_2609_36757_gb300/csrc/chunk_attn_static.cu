// Chunk-causal attention with no memory allocation anywhere: the variant of
// fastvr_chunk_attn_fwd for callers that cannot allocate device memory.
//
// Who needs it: runtimes that own every byte of device memory through their
// own pool and hand a library only the tensors of the call (a DiT serving
// engine with a preallocated KV cache, an inference-server backend), and
// real-time video pipelines that forbid cudaMalloc/cudaFree after start-up
// because those calls can synchronise the device and stall the stream.
// Such a caller keeps K and V in its own buffers and cannot provide the
// workspace region that the plan's cache buffer carries.
//
// The split-KV scratch (partial results of the units that are cut along the
// keys) lives instead in one file-scope device array of a fixed size, which
// every GPU that loads this library holds until exit.  The kernels are the
// ones fastvr_chunk_attn_fwd launches, with the same work split, so the
// outputs are the same.  A bounded wait that gives up is recorded in the
// per-device status word of the calls without a plan (also a file-scope
// device variable), which fastvr_get_device_status reads and clears.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <mutex>

#include "../../include/fastvr_attn.h"
#include "fastvr_internal.h"

namespace {

// 24 MiB: room for 190 partial results at d = 128 (378 at d = 64); a GB300
// launch uses at most one per SM (152).
constexpr size_t kScratchBytes = size_t(24) << 20;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
unsigned char* g_scratch_addr[kMaxDevices] = {};

// Device address of g_scratch on device `dev` (which must be current),
// looked up once per device: in host code the symbol is only a stand-in,
// never a device address.
unsigned char* scratch_on_current_device(int dev) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (g_scratch_addr[dev] == nullptr) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_scratch) != cudaSuccess || ptr == nullptr) {
      cudaGetLastError();
      return nullptr;
    }
    g_scratch_addr[dev] = static_cast<unsigned char*>(ptr);
  }
  return g_scratch_addr[dev];
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// The status word of the calls without a plan, one per device.
static __device__ int g_device_status;
int* g_status_addr[kMaxDevices] = {};

}  // namespace

int* fastvr::device_status_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_mutex);
  if (g_status_addr[dev] == nullptr) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_device_status) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    g_status_addr[dev] = static_cast<int*>(ptr);
  }
  return g_status_addr[dev];
}

extern "C" fastvr_status_t fastvr_chunk_attn_fwd_static(
    const fastvr_attn_config_t* cfg, const void* q, int32_t q_frames,
    const void* k_cache, const void* v_cache, int64_t cache_tokens,
    int32_t num_segments, const int64_t* seg_start, const int64_t* seg_len,
    void* out, float* lse, struct CUstream_st* stream) {
  if (cfg == nullptr || q == nullptr || k_cache == nullptr ||
      v_cache == nullptr || out == nullptr || seg_start == nullptr ||
      seg_len == nullptr || q_frames < 1 || cache_tokens < 1 ||
      num_segments < 1 || num_segments > fastvr::kMaxSegments ||
      cfg->batch < 1 || cfg->heads < 1 || cfg->tokens_per_frame < 1 ||
      !(cfg->softmax_scale >= 0.f) || !isfinite(cfg->softmax_scale) ||
      !aligned16(q) || !aligned16(out) ||
      !aligned16(k_cache) || !aligned16(v_cache) || (((uintptr_t)lse) & 3u))
    return FASTVR_ERR_INVALID_ARG;
  if (cfg->head_dim != 64 && cfg->head_dim != 128) return FASTVR_ERR_UNSUPPORTED;
  // The kernels index query rows and key tokens in 32-bit arithmetic (a key
  // coordinate is a segment start plus a tile offset), so the query length
  // and the end of every segment must stay within INT32_MAX / 2.
  const int64_t q_tokens = (int64_t)q_frames * cfg->tokens_per_frame;
  if (q_tokens > INT32_MAX / 2) return FASTVR_ERR_INVALID_ARG;
  for (int s = 0; s < num_segments; ++s)
    if (seg_start[s] < 0 || seg_len[s] < 1 || seg_len[s] > INT32_MAX / 2 ||
        seg_start[s] > INT32_MAX / 2 ||
        seg_start[s] + seg_len[s] > INT32_MAX / 2 ||
        seg_start[s] + seg_len[s] > cache_tokens)
      return FASTVR_ERR_INVALID_ARG;

  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) !=
          cudaSuccess)
    return FASTVR_ERR_CUDA;
  if (major != 10 || minor != 3) return FASTVR_ERR_UNSUPPORTED;
  unsigned char* scratch = scratch_on_current_device(dev);
  if (scratch == nullptr) return FASTVR_ERR_CUDA;

  const int d = cfg->head_dim;
  fastvr::AttnParams a;
  memset(&a, 0, sizeof(a));
  a.q = static_cast<const uint16_t*>(q);
  a.o = static_cast<uint16_t*>(out);
  a.lse = lse;
  a.k = static_cast<const uint16_t*>(k_cache);
  a.v = static_cast<const uint16_t*>(v_cache);
  a.batch = cfg->batch;
  a.heads = cfg->heads;
  a.head_dim = d;
  a.q_tokens = (int32_t)q_tokens;
  a.q_str.head = d;
  a.q_str.token = (int64_t)cfg->heads * d;
  a.q_str.batch = (int64_t)a.q_tokens * cfg->heads * d;
  a.kv_str.token = d;
  a.kv_str.head = cache_tokens * d;
  a.kv_str.batch = (int64_t)cfg->heads * cache_tokens * d;
  a.kv_tokens = cache_tokens;
  a.num_segments = num_segments;
  for (int s = 0; s < num_segments; ++s) {
    a.seg_start[s] = seg_start[s];
    a.seg_len[s] = (int32_t)seg_len[s];
  }
  const float scale =
      cfg->softmax_scale == 0.f ? 1.f / sqrtf((float)d) : cfg->softmax_scale;
  a.scale_log2 = scale * 1.4426950408889634f;

  // The array holds partial results only.  A call whose split needs more of
  // them than fit is refused rather than run with a different split.  The
  // array keeps the last call's contents, which needs no clearing: every
  // partial result is written before it is read.
  const size_t part_bytes = (size_t)fastvr::kUnitRows * (d + 1) * sizeof(float);
  const int capacity = (int)(kScratchBytes / part_bytes);
  if (fastvr::chunk_attn_parts(a) > capacity) return FASTVR_ERR_CAPACITY;
  a.workspace = reinterpret_cast<float*>(scratch);
  a.workspace_parts = capacity;
  // Timeouts go to the sticky per-device word (zero at load, cleared when
  // fastvr_get_device_status reads it).
  a.status = fastvr::device_status_word();
  if (a.status == nullptr) return FASTVR_ERR_CUDA;
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int launched = 0;
  if (fastvr::launch_chunk_attn(a, st, &launched) != cudaSuccess)
    return FASTVR_ERR_CUDA;
  return FASTVR_OK;
}
