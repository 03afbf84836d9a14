// FastVR's one-step restoration update (Eq. `eq:one_step`): after the DiT
// predicts the velocity v from the low-quality latent z_LQ at t = tau, the
// restored latent is z_hat = z_LQ - sigma_tau * v.  Elementwise and purely
// bandwidth-bound: 16-byte loads of v (8 bf16) and of the matching z_LQ
// elements, one fp32 FMA per element, a single rounding to the output type.
#include <cuda_bf16.h>

#include "fastvr_internal.h"

namespace fastvr {
namespace {

template <typename T>
struct Vec8;  // 8 elements of T
template <>
struct Vec8<__nv_bfloat16> {
  uint4 u;
  __device__ float get(int i) const {
    const __nv_bfloat16* e = reinterpret_cast<const __nv_bfloat16*>(&u);
    return __bfloat162float(e[i]);
  }
  __device__ void set(int i, float x) {
    reinterpret_cast<__nv_bfloat16*>(&u)[i] = __float2bfloat16_rn(x);
  }
};
template <>
struct Vec8<float> {
  float4 a, b;
  __device__ float get(int i) const {
    return i < 4 ? (&a.x)[i] : (&b.x)[i - 4];
  }
  __device__ void set(int i, float x) { (i < 4 ? (&a.x)[i] : (&b.x)[i - 4]) = x; }
};

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ void from_f(float& d, float x) { d = x; }
__device__ __forceinline__ void from_f(__nv_bfloat16& d, float x) {
  d = __float2bfloat16_rn(x);
}

// z and out may be the same buffer (in-place update): every element is read
// and then written by the same thread.  Each thread keeps kUnroll groups of
// loads in flight before it computes and stores, so that a few CTAs per SM
// cover the HBM latency.
constexpr int kUnroll = 4;

template <typename T>
__device__ __forceinline__ void update8(const Vec8<T>& zv,
                                        const Vec8<__nv_bfloat16>& vv,
                                        float neg_sigma, Vec8<T>* dst) {
  Vec8<T> o;
#pragma unroll
  for (int e = 0; e < 8; ++e) o.set(e, fmaf(neg_sigma, vv.get(e), zv.get(e)));
  *dst = o;
}

template <typename T>
__global__ void __launch_bounds__(256)
one_step_kernel(const T* z, const __nv_bfloat16* __restrict__ v, T* out,
                int64_t n, float neg_sigma) {
  pdl_trigger();
  pdl_wait();  // z and v may come from the previous kernel on the stream
  const int64_t n8 = n / 8;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const Vec8<T>* z8 = reinterpret_cast<const Vec8<T>*>(z);
  const uint4* v8 = reinterpret_cast<const uint4*>(v);
  Vec8<T>* o8 = reinterpret_cast<Vec8<T>*>(out);
  int64_t i = tid;
  for (; i + (kUnroll - 1) * stride < n8; i += kUnroll * stride) {
    Vec8<T> zv[kUnroll];
    Vec8<__nv_bfloat16> vv[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      zv[u] = z8[i + u * stride];
      vv[u].u = __ldcs(v8 + i + u * stride);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      update8(zv[u], vv[u], neg_sigma, o8 + i + u * stride);
  }
  for (; i < n8; i += stride) {
    Vec8<__nv_bfloat16> vv;
    vv.u = __ldcs(v8 + i);
    update8(z8[i], vv, neg_sigma, o8 + i);
  }
  for (int64_t i = n8 * 8 + tid; i < n; i += stride)  // fewer than 8 left
    from_f(out[i], fmaf(neg_sigma, __bfloat162float(v[i]), to_f(z[i])));
}

}  // namespace

cudaError_t launch_one_step(const void* z, const void* v, void* out, int64_t n,
                            float sigma, int dtype, cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms <= 0) sms = 152;
  int64_t blocks = (int64_t)sms * 8;
  const int64_t need = (n / 8 + 255) / 256 + 1;
  if (blocks > need) blocks = need;
  const float neg_sigma = -sigma;
  if (dtype == 0)
    return launch_pdl(one_step_kernel<__nv_bfloat16>, dim3((unsigned)blocks),
                      dim3(256), 0, stream,
                      static_cast<const __nv_bfloat16*>(z),
                      static_cast<const __nv_bfloat16*>(v),
                      static_cast<__nv_bfloat16*>(out), n, neg_sigma);
  return launch_pdl(one_step_kernel<float>, dim3((unsigned)blocks), dim3(256),
                    0, stream, static_cast<const float*>(z),
                    static_cast<const __nv_bfloat16*>(v),
                    static_cast<float*>(out), n, neg_sigma);
}

}  // namespace fastvr
