// Host side of the chunk-causal attention library: the C ABI declared in
// include/fastvr_attn.h.  Plans, ring-slot bookkeeping and the visibility
// computation are plain host code; the device work is in kv_append.cu and
// chunk_attn_fwd.cu.
//
// Visibility (Sec. 3.1, Eq. 1, window W): chunk c's queries see the keys of
// chunks max(0, c - W) .. c, or 0 .. c when unbounded.  Chunk c' lives in
// cache slot c' mod S (S = W + 1 for a bounded window, else the chunk
// capacity), so the visible chunks occupy consecutive slots modulo S and, in
// slot order, form at most two contiguous token ranges of a head's cache: only
// the newest chunk may be partly filled (a ragged final chunk), and the ring
// wrap can split the set once.  Attention does not depend on the order of
// the keys, so slot order is as good as chunk order.
#include <cuda_runtime.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <new>
#include <vector>

#include "../../include/fastvr_attn.h"
#include "fastvr_internal.h"

namespace {

constexpr size_t kControlBytes = 256;

struct Segment {
  int64_t start, len;
};

}  // namespace

struct fastvr_plan_s {
  fastvr_attn_config_t cfg;
  int64_t slots;         // S
  int64_t slot_tokens;   // k * N
  int64_t cache_tokens;  // S * k * N per head
  size_t kv_bytes;       // bytes of the K region (= the V region)
  char* base;            // caller's cache buffer
  int64_t chunks;        // chunks appended since the last reset
  int32_t last_frames;   // frames of the newest chunk
  bool device_ready;
  int device;
  int64_t launches;        // kernels enqueued since creation
  int32_t inject_stall;    // failure-detection test hook
  uint64_t wait_limit_ns;  // 0 = kernel default
  int64_t append_shift;    // debug builds: next append's destination shift
};

namespace {

// Failure-detection hook for the calls without a plan (process-wide).
std::atomic<int32_t> g_noplan_stall{0};
std::atomic<uint64_t> g_noplan_wait_ns{0};

bool valid_config(const fastvr_attn_config_t* c) {
  return c != nullptr && c->batch > 0 && c->heads > 0 && c->head_dim > 0 &&
         c->tokens_per_frame > 0 && c->frames_per_chunk > 0 &&
         c->window_chunks >= -1 && !(c->softmax_scale < 0.f) &&
         isfinite(c->softmax_scale) &&
         (c->window_chunks >= 0 || c->max_chunks > 0);
}

bool supported_dim(int d) { return d == 64 || d == 128; }

int64_t num_slots(const fastvr_attn_config_t& c) {
  return c.window_chunks >= 0 ? (int64_t)c.window_chunks + 1 : c.max_chunks;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// Visible segments of the newest chunk, in slot order, merged when adjacent.
std::vector<Segment> visible_segments(const fastvr_plan_s& p) {
  std::vector<Segment> segs;
  const int64_t c = p.chunks - 1;
  const int32_t W = p.cfg.window_chunks;
  const int64_t lo = W < 0 ? 0 : std::max<int64_t>(0, c - W);
  std::vector<Segment> parts;
  for (int64_t cc = lo; cc <= c; ++cc) {
    const int64_t slot = cc % p.slots;
    const int64_t frames = cc == c ? p.last_frames : p.cfg.frames_per_chunk;
    parts.push_back({slot * p.slot_tokens, frames * p.cfg.tokens_per_frame});
  }
  std::sort(parts.begin(), parts.end(),
            [](const Segment& a, const Segment& b) { return a.start < b.start; });
  for (const Segment& s : parts) {
    if (!segs.empty() && segs.back().start + segs.back().len == s.start)
      segs.back().len += s.len;
    else
      segs.push_back(s);
  }
  return segs;
}

float* workspace(const fastvr_plan_s* p) {
  return reinterpret_cast<float*>(p->base + 2 * p->kv_bytes);
}

int* control_word(const fastvr_plan_s* p) {
  return reinterpret_cast<int*>(p->base + 2 * p->kv_bytes +
                                fastvr::workspace_bytes(p->cfg.head_dim));
}

fastvr_status_t ensure_device(fastvr_plan_s* p) {
  if (p->device_ready) return FASTVR_OK;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return FASTVR_ERR_CUDA;
  int major = 0, minor = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) !=
          cudaSuccess)
    return FASTVR_ERR_CUDA;
  if (major != 10 || minor != 3) return FASTVR_ERR_UNSUPPORTED;
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, p->base) != cudaSuccess ||
      attr.type != cudaMemoryTypeDevice || attr.device != dev) {
    cudaGetLastError();
    return FASTVR_ERR_INVALID_ARG;
  }
  // Clear the control block once; kernels only ever set it.
  if (cudaMemset(control_word(p), 0, kControlBytes) != cudaSuccess)
    return FASTVR_ERR_CUDA;
  p->device = dev;
  p->device_ready = true;
  return FASTVR_OK;
}

}  // namespace

extern "C" {

const char* fastvr_status_string(fastvr_status_t s) {
  switch (s) {
    case FASTVR_OK: return "FASTVR_OK";
    case FASTVR_ERR_INVALID_ARG: return "FASTVR_ERR_INVALID_ARG";
    case FASTVR_ERR_UNSUPPORTED: return "FASTVR_ERR_UNSUPPORTED";
    case FASTVR_ERR_CAPACITY: return "FASTVR_ERR_CAPACITY";
    case FASTVR_ERR_SEQUENCE: return "FASTVR_ERR_SEQUENCE";
    case FASTVR_ERR_CUDA: return "FASTVR_ERR_CUDA";
    case FASTVR_ERR_TIMEOUT: return "FASTVR_ERR_TIMEOUT";
    case FASTVR_ERR_BOUNDS: return "FASTVR_ERR_BOUNDS";
  }
  return "FASTVR_ERR_UNKNOWN";
}

fastvr_status_t fastvr_kv_cache_bytes(const fastvr_attn_config_t* cfg,
                                      size_t* bytes) {
  if (!valid_config(cfg) || bytes == nullptr) return FASTVR_ERR_INVALID_ARG;
  if (!supported_dim(cfg->head_dim)) return FASTVR_ERR_UNSUPPORTED;
  const int64_t tokens =
      num_slots(*cfg) * cfg->frames_per_chunk * (int64_t)cfg->tokens_per_frame;
  const int64_t per = (int64_t)cfg->batch * cfg->heads * tokens * cfg->head_dim * 2;
  // K and V regions, each a multiple of 256 bytes (d*2 >= 128 and tokens of
  // a slot are whole rows, so per is a multiple of 128; round up anyway).
  const int64_t region = (per + 255) / 256 * 256;
  *bytes = (size_t)(2 * region) + fastvr::workspace_bytes(cfg->head_dim) +
           kControlBytes;
  return FASTVR_OK;
}

fastvr_status_t fastvr_attn_plan(const fastvr_attn_config_t* cfg,
                                 void* kv_cache, size_t bytes,
                                 fastvr_plan_t* out) {
  if (out == nullptr) return FASTVR_ERR_INVALID_ARG;
  *out = nullptr;
  if (!valid_config(cfg) || kv_cache == nullptr ||
      ((uintptr_t)kv_cache & 255u) != 0)
    return FASTVR_ERR_INVALID_ARG;
  if (!supported_dim(cfg->head_dim)) return FASTVR_ERR_UNSUPPORTED;
  size_t need = 0;
  fastvr_status_t st = fastvr_kv_cache_bytes(cfg, &need);
  if (st != FASTVR_OK) return st;
  if (bytes < need) return FASTVR_ERR_CAPACITY;
  fastvr_plan_s* p = new (std::nothrow) fastvr_plan_s();
  if (p == nullptr) return FASTVR_ERR_INVALID_ARG;
  p->cfg = *cfg;
  if (p->cfg.softmax_scale == 0.f)
    p->cfg.softmax_scale = 1.f / sqrtf((float)cfg->head_dim);
  if (p->cfg.window_chunks >= 0) p->cfg.max_chunks = 0;
  p->slots = num_slots(*cfg);
  p->slot_tokens = (int64_t)cfg->frames_per_chunk * cfg->tokens_per_frame;
  p->cache_tokens = p->slots * p->slot_tokens;
  p->kv_bytes =
      (need - kControlBytes - fastvr::workspace_bytes(cfg->head_dim)) / 2;
  p->base = static_cast<char*>(kv_cache);
  p->chunks = 0;
  p->last_frames = 0;
  p->device_ready = false;
  p->device = -1;
  p->launches = 0;
  p->inject_stall = 0;
  p->wait_limit_ns = 0;
  *out = p;
  return FASTVR_OK;
}

fastvr_status_t fastvr_kv_append(fastvr_plan_t p, const void* k_new,
                                 const void* v_new, int32_t frames,
                                 struct CUstream_st* stream) {
  if (p == nullptr || k_new == nullptr || v_new == nullptr || frames < 1 ||
      !aligned16(k_new) || !aligned16(v_new))
    return FASTVR_ERR_INVALID_ARG;
  if (frames > p->cfg.frames_per_chunk) return FASTVR_ERR_CAPACITY;
  if (p->chunks > 0 && p->last_frames < p->cfg.frames_per_chunk)
    return FASTVR_ERR_SEQUENCE;  // the stream already ended with a ragged chunk
  if (p->cfg.window_chunks < 0 && p->chunks >= p->cfg.max_chunks)
    return FASTVR_ERR_CAPACITY;
  fastvr_status_t st = ensure_device(p);
  if (st != FASTVR_OK) return st;

  fastvr::AppendParams a;
  a.k_new = static_cast<const uint16_t*>(k_new);
  a.v_new = static_cast<const uint16_t*>(v_new);
  a.k_cache = reinterpret_cast<uint16_t*>(p->base);
  a.v_cache = reinterpret_cast<uint16_t*>(p->base + p->kv_bytes);
  a.batch = p->cfg.batch;
  a.tokens = frames * p->cfg.tokens_per_frame;
  a.heads = p->cfg.heads;
  a.head_dim = p->cfg.head_dim;
  a.cache_tokens = p->cache_tokens;
  a.token_offset = (p->chunks % p->slots) * p->slot_tokens + p->append_shift;
  a.status = control_word(p);
  p->append_shift = 0;
  if (fastvr::launch_kv_append(a, reinterpret_cast<cudaStream_t>(stream)) !=
      cudaSuccess)
    return FASTVR_ERR_CUDA;
  p->launches += 1;
  p->chunks += 1;
  p->last_frames = frames;
  return FASTVR_OK;
}

fastvr_status_t fastvr_chunk_attn_fwd(fastvr_plan_t p, const void* q, void* out,
                                      float* lse, struct CUstream_st* stream) {
  if (p == nullptr || q == nullptr || out == nullptr || !aligned16(q) ||
      !aligned16(out) || (((uintptr_t)lse) & 3u) != 0)
    return FASTVR_ERR_INVALID_ARG;
  if (p->chunks == 0) return FASTVR_ERR_SEQUENCE;
  fastvr_status_t st = ensure_device(p);
  if (st != FASTVR_OK) return st;

  const std::vector<Segment> segs = visible_segments(*p);
  if ((int)segs.size() > fastvr::kMaxSegments) return FASTVR_ERR_INVALID_ARG;
  const fastvr_attn_config_t& c = p->cfg;
  fastvr::AttnParams a;
  memset(&a, 0, sizeof(a));
  a.q = static_cast<const uint16_t*>(q);
  a.o = static_cast<uint16_t*>(out);
  a.lse = lse;
  a.k = reinterpret_cast<const uint16_t*>(p->base);
  a.v = reinterpret_cast<const uint16_t*>(p->base + p->kv_bytes);
  a.batch = c.batch;
  a.heads = c.heads;
  a.head_dim = c.head_dim;
  a.q_tokens = p->last_frames * c.tokens_per_frame;
  a.q_str.head = c.head_dim;
  a.q_str.token = (int64_t)c.heads * c.head_dim;
  a.q_str.batch = (int64_t)a.q_tokens * c.heads * c.head_dim;
  a.kv_str.token = c.head_dim;
  a.kv_str.head = p->cache_tokens * c.head_dim;
  a.kv_str.batch = (int64_t)c.heads * p->cache_tokens * c.head_dim;
  a.kv_tokens = p->cache_tokens;
  a.num_segments = (int32_t)segs.size();
  for (size_t i = 0; i < segs.size(); ++i) {
    a.seg_start[i] = segs[i].start;
    a.seg_len[i] = (int32_t)segs[i].len;
  }
  a.scale_log2 = c.softmax_scale * 1.4426950408889634f;
  a.status = control_word(p);
  a.workspace = workspace(p);
  a.workspace_parts = fastvr::kMaxParts;
  a.wait_limit_ns = p->wait_limit_ns;
  a.inject_stall = p->inject_stall;
  int launched = 0;
  const cudaError_t e = fastvr::launch_chunk_attn(
      a, reinterpret_cast<cudaStream_t>(stream), &launched);
  p->launches += launched;
  if (e != cudaSuccess) return FASTVR_ERR_CUDA;
  return FASTVR_OK;
}

fastvr_status_t fastvr_plan_reset(fastvr_plan_t p) {
  if (p == nullptr) return FASTVR_ERR_INVALID_ARG;
  p->chunks = 0;
  p->last_frames = 0;
  return FASTVR_OK;
}

fastvr_status_t fastvr_get_status(fastvr_plan_t p) {
  if (p == nullptr) return FASTVR_ERR_INVALID_ARG;
  if (!p->device_ready) return FASTVR_OK;
  if (cudaDeviceSynchronize() != cudaSuccess) return FASTVR_ERR_CUDA;
  int word = 0;
  if (cudaMemcpy(&word, control_word(p), sizeof(int), cudaMemcpyDeviceToHost) !=
      cudaSuccess)
    return FASTVR_ERR_CUDA;
  if (word != fastvr::kDevOk) {
    const int zero = 0;
    cudaMemcpy(control_word(p), &zero, sizeof(int), cudaMemcpyHostToDevice);
    return word == fastvr::kDevBounds ? FASTVR_ERR_BOUNDS : FASTVR_ERR_TIMEOUT;
  }
  return FASTVR_OK;
}

fastvr_status_t fastvr_plan_get_state(fastvr_plan_t p, int64_t* chunks,
                                      int32_t* last_frames) {
  if (p == nullptr || chunks == nullptr || last_frames == nullptr)
    return FASTVR_ERR_INVALID_ARG;
  *chunks = p->chunks;
  *last_frames = p->last_frames;
  return FASTVR_OK;
}

fastvr_status_t fastvr_plan_set_state(fastvr_plan_t p, int64_t chunks,
                                      int32_t last_frames) {
  if (p == nullptr || chunks < 0) return FASTVR_ERR_INVALID_ARG;
  if (chunks == 0 ? last_frames != 0
                  : (last_frames < 1 || last_frames > p->cfg.frames_per_chunk))
    return FASTVR_ERR_INVALID_ARG;
  if (p->cfg.window_chunks < 0 && chunks > p->cfg.max_chunks)
    return FASTVR_ERR_CAPACITY;
  p->chunks = chunks;
  p->last_frames = last_frames;
  return FASTVR_OK;
}

fastvr_status_t fastvr_plan_visible(fastvr_plan_t p, int32_t* num_segments,
                                    int64_t* seg_start, int64_t* seg_len,
                                    int64_t* visible_tokens) {
  if (p == nullptr || num_segments == nullptr || seg_start == nullptr ||
      seg_len == nullptr || visible_tokens == nullptr)
    return FASTVR_ERR_INVALID_ARG;
  if (p->chunks == 0) return FASTVR_ERR_SEQUENCE;
  const std::vector<Segment> segs = visible_segments(*p);
  if ((int)segs.size() > fastvr::kMaxSegments) return FASTVR_ERR_INVALID_ARG;
  int64_t total = 0;
  for (size_t i = 0; i < segs.size(); ++i) {
    seg_start[i] = segs[i].start;
    seg_len[i] = segs[i].len;
    total += segs[i].len;
  }
  *num_segments = (int32_t)segs.size();
  *visible_tokens = total;
  return FASTVR_OK;
}

fastvr_status_t fastvr_blockcausal_attn_fwd(const fastvr_attn_config_t* cfg,
                                            int32_t num_frames, const void* q,
                                            const void* k, const void* v,
                                            void* out, float* lse,
                                            struct CUstream_st* stream) {
  if (cfg == nullptr || cfg->batch < 1 || cfg->heads < 1 ||
      cfg->tokens_per_frame < 1 || cfg->frames_per_chunk < 1 ||
      cfg->window_chunks < -1 || !(cfg->softmax_scale >= 0.f) ||
      !isfinite(cfg->softmax_scale) || num_frames < 1 || q == nullptr ||
      k == nullptr || v == nullptr || out == nullptr || !aligned16(q) ||
      !aligned16(k) || !aligned16(v) || !aligned16(out) ||
      (((uintptr_t)lse) & 3u) != 0)
    return FASTVR_ERR_INVALID_ARG;
  if (!supported_dim(cfg->head_dim)) return FASTVR_ERR_UNSUPPORTED;
  const int64_t L = (int64_t)num_frames * cfg->tokens_per_frame;
  const int64_t chunk = (int64_t)cfg->frames_per_chunk * cfg->tokens_per_frame;
  if (L > INT32_MAX / 2 || chunk > INT32_MAX / 2) return FASTVR_ERR_INVALID_ARG;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) !=
          cudaSuccess)
    return FASTVR_ERR_CUDA;
  if (major != 10 || minor != 3) return FASTVR_ERR_UNSUPPORTED;
  fastvr::OneShotParams a;
  memset(&a, 0, sizeof(a));
  a.q = static_cast<const uint16_t*>(q);
  a.k = static_cast<const uint16_t*>(k);
  a.v = static_cast<const uint16_t*>(v);
  a.o = static_cast<uint16_t*>(out);
  a.lse = lse;
  a.batch = cfg->batch;
  a.heads = cfg->heads;
  a.head_dim = cfg->head_dim;
  a.seq_tokens = (int32_t)L;
  a.chunk_tokens = (int32_t)chunk;
  a.window = cfg->window_chunks;
  const float scale = cfg->softmax_scale == 0.f
                          ? 1.f / sqrtf((float)cfg->head_dim)
                          : cfg->softmax_scale;
  a.scale_log2 = scale * 1.4426950408889634f;
  a.status = fastvr::device_status_word();
  a.inject_stall = g_noplan_stall.load();
  a.wait_limit_ns = g_noplan_wait_ns.load();
  if (fastvr::launch_blockcausal_attn(a, reinterpret_cast<cudaStream_t>(stream)) !=
      cudaSuccess)
    return FASTVR_ERR_CUDA;
  return FASTVR_OK;
}

namespace {
// Validation shared by the one-shot backward entry points.
fastvr_status_t check_oneshot_cfg(const fastvr_attn_config_t* cfg,
                                  int32_t num_frames) {
  if (cfg == nullptr || cfg->batch < 1 || cfg->heads < 1 ||
      cfg->tokens_per_frame < 1 || cfg->frames_per_chunk < 1 ||
      cfg->window_chunks < -1 || !(cfg->softmax_scale >= 0.f) ||
      !isfinite(cfg->softmax_scale) || num_frames < 1)
    return FASTVR_ERR_INVALID_ARG;
  if (!supported_dim(cfg->head_dim)) return FASTVR_ERR_UNSUPPORTED;
  const int64_t L = (int64_t)num_frames * cfg->tokens_per_frame;
  if (L > INT32_MAX / 2 ||
      (int64_t)cfg->frames_per_chunk * cfg->tokens_per_frame > INT32_MAX / 2)
    return FASTVR_ERR_INVALID_ARG;
  return FASTVR_OK;
}
}  // namespace

fastvr_status_t fastvr_blockcausal_bwd_scratch_bytes(
    const fastvr_attn_config_t* cfg, int32_t num_frames, size_t* bytes) {
  fastvr_status_t st = check_oneshot_cfg(cfg, num_frames);
  if (st != FASTVR_OK) return st;
  if (bytes == nullptr) return FASTVR_ERR_INVALID_ARG;
  const int64_t L = (int64_t)num_frames * cfg->tokens_per_frame;
  const int64_t padded = (L + 127) / 128 * 128;
  *bytes = (size_t)(2 * (int64_t)cfg->batch * cfg->heads * padded * 4);
  return FASTVR_OK;
}

fastvr_status_t fastvr_blockcausal_attn_bwd(
    const fastvr_attn_config_t* cfg, int32_t num_frames, const void* q,
    const void* k, const void* v, const void* out, const void* dout,
    const float* lse, void* dq, void* dk, void* dv, float* scratch,
    size_t scratch_bytes, struct CUstream_st* stream) {
  fastvr_status_t st = check_oneshot_cfg(cfg, num_frames);
  if (st != FASTVR_OK) return st;
  const void* ptrs[] = {q, k, v, out, dout, lse, dq, dk, dv, scratch};
  for (const void* ptr : ptrs)
    if (ptr == nullptr || !aligned16(ptr)) return FASTVR_ERR_INVALID_ARG;
  size_t need = 0;
  fastvr_blockcausal_bwd_scratch_bytes(cfg, num_frames, &need);
  if (scratch_bytes < need) return FASTVR_ERR_CAPACITY;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) !=
          cudaSuccess)
    return FASTVR_ERR_CUDA;
  if (major != 10 || minor != 3) return FASTVR_ERR_UNSUPPORTED;
  fastvr::BwdArgs a;
  memset(&a, 0, sizeof(a));
  a.q = static_cast<const uint16_t*>(q);
  a.k = static_cast<const uint16_t*>(k);
  a.v = static_cast<const uint16_t*>(v);
  a.out = static_cast<const uint16_t*>(out);
  a.dout = static_cast<const uint16_t*>(dout);
  a.lse = lse;
  a.dq = static_cast<uint16_t*>(dq);
  a.dk = static_cast<uint16_t*>(dk);
  a.dv = static_cast<uint16_t*>(dv);
  a.scratch = scratch;
  a.batch = cfg->batch;
  a.heads = cfg->heads;
  a.head_dim = cfg->head_dim;
  a.seq_tokens = num_frames * cfg->tokens_per_frame;
  a.chunk_tokens = cfg->frames_per_chunk * cfg->tokens_per_frame;
  a.window = cfg->window_chunks;
  a.scale = cfg->softmax_scale == 0.f ? 1.f / sqrtf((float)cfg->head_dim)
                                      : cfg->softmax_scale;
  a.status = fastvr::device_status_word();
  a.inject_stall = g_noplan_stall.load();
  a.wait_limit_ns = g_noplan_wait_ns.load();
  if (fastvr::launch_blockcausal_attn_bwd(
          a, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return FASTVR_ERR_CUDA;
  return FASTVR_OK;
}

fastvr_status_t fastvr_one_step_update(const void* z_lq, const void* v,
                                       void* z_hat, int64_t n, float sigma,
                                       int32_t dtype,
                                       struct CUstream_st* stream) {
  if (z_lq == nullptr || v == nullptr || z_hat == nullptr || n < 0 ||
      !isfinite(sigma) || (dtype != 0 && dtype != 1) || !aligned16(z_lq) ||
      !aligned16(v) || !aligned16(z_hat))
    return FASTVR_ERR_INVALID_ARG;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) !=
          cudaSuccess)
    return FASTVR_ERR_CUDA;
  if (major != 10 || minor != 3) return FASTVR_ERR_UNSUPPORTED;
  if (fastvr::launch_one_step(z_lq, v, z_hat, n, sigma, dtype,
                              reinterpret_cast<cudaStream_t>(stream)) !=
      cudaSuccess)
    return FASTVR_ERR_CUDA;
  return FASTVR_OK;
}

fastvr_status_t fastvr_plan_launch_count(fastvr_plan_t p, int64_t* launches) {
  if (p == nullptr || launches == nullptr) return FASTVR_ERR_INVALID_ARG;
  *launches = p->launches;
  return FASTVR_OK;
}

fastvr_status_t fastvr_debug_inject_stall(fastvr_plan_t p, int32_t stall,
                                          uint64_t wait_limit_ns) {
  if (p == nullptr) return FASTVR_ERR_INVALID_ARG;
  p->inject_stall = stall != 0;
  p->wait_limit_ns = wait_limit_ns;
  return FASTVR_OK;
}

fastvr_status_t fastvr_debug_shift_next_append(fastvr_plan_t p,
                                              int64_t tokens) {
  if (p == nullptr || tokens < 0 || tokens > p->slot_tokens)
    return FASTVR_ERR_INVALID_ARG;
#ifdef FASTVR_BOUNDS_CHECK
  p->append_shift = tokens;
  return FASTVR_OK;
#else
  return FASTVR_ERR_UNSUPPORTED;
#endif
}

fastvr_status_t fastvr_get_device_status(void) {
  int* word = fastvr::device_status_word();
  if (word == nullptr) return FASTVR_ERR_CUDA;
  if (cudaDeviceSynchronize() != cudaSuccess) return FASTVR_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, word, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return FASTVR_ERR_CUDA;
  if (v == fastvr::kDevOk) return FASTVR_OK;
  const int zero = 0;
  cudaMemcpy(word, &zero, sizeof(int), cudaMemcpyHostToDevice);
  return v == fastvr::kDevBounds ? FASTVR_ERR_BOUNDS : FASTVR_ERR_TIMEOUT;
}

fastvr_status_t fastvr_debug_inject_stall_noplan(int32_t stall,
                                                 uint64_t wait_limit_ns) {
  g_noplan_stall.store(stall != 0);
  g_noplan_wait_ns.store(wait_limit_ns);
  return FASTVR_OK;
}

void fastvr_plan_destroy(fastvr_plan_t p) { delete p; }

}  // extern "C"
