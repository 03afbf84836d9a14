// Chunk-causal attention forward (Sec. 3.1, Eq. 1), first GPU kernel.
//
// One CTA computes 128 query rows of one (batch, head) against the visible
// key segments of the cache, with an online softmax in float32 (exp2 domain)
// and bf16 tensor-core MMAs (m16n8k16) accumulating in float32.  Masking
// happens at chunk granularity, so every key inside a visible segment is
// visible to every query of the chunk; the only in-kernel mask is the ragged
// end of a segment, whose tail columns are set to -inf.
#include <cuda_bf16.h>

#include "fastvr_internal.h"

namespace fastvr {
namespace {

constexpr int kBlockM = 128;  // query rows per CTA (16 per warp)
constexpr int kBlockN = 64;   // keys per tile
constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src,
                                           bool valid) {
  const int n = valid ? 16 : 0;  // zero-fill when the row is out of range
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst),
               "l"(src), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;\n" ::);
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0,
                                        uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0,
                                          uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile(
      "ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
      : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
      : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float* c, const uint32_t* a,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Locate tile `it` of the flattened visible segment list.
__device__ __forceinline__ void tile_at(const AttnParams& p, int it,
                                        int64_t& tok0, int& valid) {
  for (int s = 0; s < p.num_segments; ++s) {
    const int tiles = (p.seg_len[s] + kBlockN - 1) / kBlockN;
    if (it < tiles) {
      tok0 = p.seg_start[s] + (int64_t)it * kBlockN;
      valid = min(kBlockN, p.seg_len[s] - it * kBlockN);
      return;
    }
    it -= tiles;
  }
  tok0 = 0;
  valid = 0;
}

template <int D>
__global__ void __launch_bounds__(kThreads)
chunk_attn_mma_kernel(const AttnParams p) {
  constexpr int kStride = D + 8;  // padded smem row (elements): no conflicts
  constexpr int kChunks = D / 8;  // 16-byte pieces per row
  extern __shared__ __align__(16) uint16_t smem[];
  uint16_t* sQ = smem;                          // [kBlockM][kStride]
  uint16_t* sK = sQ + kBlockM * kStride;        // [2][kBlockN][kStride]
  uint16_t* sV = sK + 2 * kBlockN * kStride;    // [2][kBlockN][kStride]

  const int tid = threadIdx.x, warp = tid / 32, lane = tid % 32;
  const int q0 = blockIdx.x * kBlockM;
  const int h = blockIdx.y, b = blockIdx.z;

  const uint16_t* qbase = p.q + b * p.q_str.batch + h * p.q_str.head;
  const uint16_t* kbase = p.k + b * p.kv_str.batch + h * p.kv_str.head;
  const uint16_t* vbase = p.v + b * p.kv_str.batch + h * p.kv_str.head;

  int num_tiles = 0;
  for (int s = 0; s < p.num_segments; ++s)
    num_tiles += (p.seg_len[s] + kBlockN - 1) / kBlockN;

  // Q tile (zero rows past the end of the chunk).
  for (int i = tid; i < kBlockM * kChunks; i += kThreads) {
    const int r = i / kChunks, c = i % kChunks;
    const bool ok = q0 + r < p.q_tokens;
    const uint16_t* src = qbase + (int64_t)(ok ? q0 + r : 0) * p.q_str.token + c * 8;
    cp_async16(smem_u32(sQ + r * kStride + c * 8), src, ok);
  }
  cp_async_commit();

  auto load_kv = [&](int it, int stage) {
    int64_t tok0;
    int valid;
    tile_at(p, it, tok0, valid);
    uint16_t* dk = sK + stage * kBlockN * kStride;
    uint16_t* dv = sV + stage * kBlockN * kStride;
    for (int i = tid; i < kBlockN * kChunks; i += kThreads) {
      const int r = i / kChunks, c = i % kChunks;
      const int64_t t = tok0 + r;
      const bool ok = r < valid && t < p.kv_tokens;
      const int64_t off = (ok ? t : 0) * p.kv_str.token + c * 8;
      cp_async16(smem_u32(dk + r * kStride + c * 8), kbase + off, ok);
      cp_async16(smem_u32(dv + r * kStride + c * 8), vbase + off, ok);
    }
  };

  if (num_tiles > 0) load_kv(0, 0);
  cp_async_commit();

  // Q fragments stay in registers for the whole key stream.
  cp_async_wait<1>();
  __syncthreads();
  uint32_t qf[D / 16][4];
  {
    const int row = warp * 16 + (lane % 16);
    const int col = (lane / 16) * 8;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks)
      ldsm_x4(smem_u32(sQ + row * kStride + ks * 16 + col), qf[ks][0],
              qf[ks][1], qf[ks][2], qf[ks][3]);
  }

  float o_acc[D / 8][4];
#pragma unroll
  for (int j = 0; j < D / 8; ++j)
    o_acc[j][0] = o_acc[j][1] = o_acc[j][2] = o_acc[j][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY};  // exp2-domain running max
  float l_run[2] = {0.f, 0.f};              // per-thread partial sums

  const int g = lane / 4, t4 = lane % 4;
  for (int it = 0; it < num_tiles; ++it) {
    if (it + 1 < num_tiles) load_kv(it + 1, (it + 1) & 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();

    int64_t tok0;
    int valid;
    tile_at(p, it, tok0, valid);
    const uint16_t* k_s = sK + (it & 1) * kBlockN * kStride;
    const uint16_t* v_s = sV + (it & 1) * kBlockN * kStride;

    // S = Q K^T for this warp's 16 rows x 64 keys.
    float s[kBlockN / 8][4];
#pragma unroll
    for (int n = 0; n < kBlockN / 8; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
#pragma unroll
      for (int n2 = 0; n2 < kBlockN / 16; ++n2) {
        const int mi = lane / 8, rr = lane % 8;
        const int row = n2 * 16 + (mi / 2) * 8 + rr;
        const int col = ks * 16 + (mi % 2) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(k_s + row * kStride + col), b0, b1, b2, b3);
        mma_bf16(s[2 * n2], qf[ks], b0, b1);
        mma_bf16(s[2 * n2 + 1], qf[ks], b2, b3);
      }
    }

    // Online softmax over the tile (rows g and g + 8 of this warp).
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int n = 0; n < kBlockN / 8; ++n) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int col = n * 8 + 2 * t4 + (e & 1);
        float x = s[n][e] * p.scale_log2;
        if (col >= valid) x = -INFINITY;
        s[n][e] = x;
        mx[e >> 1] = fmaxf(mx[e >> 1], x);
      }
    }
    float alpha[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
      const float m_new = fmaxf(m_run[r], mx[r]);
      alpha[r] = ex2(m_run[r] - m_new);
      m_run[r] = m_new;
      l_run[r] *= alpha[r];
    }
#pragma unroll
    for (int n = 0; n < kBlockN / 8; ++n) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float pe = ex2(s[n][e] - m_run[e >> 1]);
        s[n][e] = pe;
        l_run[e >> 1] += pe;
      }
    }
#pragma unroll
    for (int j = 0; j < D / 8; ++j) {
      o_acc[j][0] *= alpha[0];
      o_acc[j][1] *= alpha[0];
      o_acc[j][2] *= alpha[1];
      o_acc[j][3] *= alpha[1];
    }

    // O += P V.
#pragma unroll
    for (int kk = 0; kk < kBlockN / 16; ++kk) {
      uint32_t a[4];
      a[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      a[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      a[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      a[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int n2 = 0; n2 < D / 16; ++n2) {
        const int mi = lane / 8, rr = lane % 8;
        const int row = kk * 16 + (mi % 2) * 8 + rr;
        const int col = n2 * 16 + (mi / 2) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(v_s + row * kStride + col), b0, b1, b2, b3);
        mma_bf16(o_acc[2 * n2], a, b0, b1);
        mma_bf16(o_acc[2 * n2 + 1], a, b2, b3);
      }
    }
    __syncthreads();  // stage (it & 1) is refilled by the next iteration
  }

  // Epilogue: normalise, stage through shared memory, store coalesced.
  float inv_l[2];
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 1);
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 2);
    inv_l[r] = 1.f / l_run[r];
  }
  const int r0 = warp * 16 + g;
#pragma unroll
  for (int j = 0; j < D / 8; ++j) {
    const int col = j * 8 + 2 * t4;
    *reinterpret_cast<uint32_t*>(sQ + r0 * kStride + col) =
        pack_bf16(o_acc[j][0] * inv_l[0], o_acc[j][1] * inv_l[0]);
    *reinterpret_cast<uint32_t*>(sQ + (r0 + 8) * kStride + col) =
        pack_bf16(o_acc[j][2] * inv_l[1], o_acc[j][3] * inv_l[1]);
  }
  if (p.lse != nullptr && t4 == 0) {
    float* lse = p.lse + ((int64_t)b * p.heads + h) * p.q_tokens;
    const float ln2 = 0.6931471805599453f;
    if (q0 + r0 < p.q_tokens) lse[q0 + r0] = (m_run[0] + __log2f(l_run[0])) * ln2;
    if (q0 + r0 + 8 < p.q_tokens)
      lse[q0 + r0 + 8] = (m_run[1] + __log2f(l_run[1])) * ln2;
  }
  __syncthreads();
  uint16_t* obase = p.o + b * p.q_str.batch + h * p.q_str.head;
  for (int i = tid; i < kBlockM * kChunks; i += kThreads) {
    const int r = i / kChunks, c = i % kChunks;
    if (q0 + r < p.q_tokens)
      *reinterpret_cast<uint4*>(obase + (int64_t)(q0 + r) * p.q_str.token + c * 8) =
          *reinterpret_cast<const uint4*>(sQ + r * kStride + c * 8);
  }
}

template <int D>
cudaError_t launch_d(const AttnParams& p, cudaStream_t stream) {
  constexpr int kStride = D + 8;
  const size_t smem = (size_t)(kBlockM + 4 * kBlockN) * kStride * sizeof(uint16_t);
  cudaError_t e = cudaFuncSetAttribute(chunk_attn_mma_kernel<D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((p.q_tokens + kBlockM - 1) / kBlockM, p.heads, p.batch);
  chunk_attn_mma_kernel<D><<<grid, kThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_chunk_attn(const AttnParams& p, cudaStream_t stream) {
  if (p.head_dim == 64) return launch_d<64>(p, stream);
  if (p.head_dim == 128) return launch_d<128>(p, stream);
  return cudaErrorInvalidValue;
}

}  // namespace fastvr
