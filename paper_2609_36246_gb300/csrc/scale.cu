// scale.cu -- y = x * (*scale) elementwise on bf16 or fp32 buffers, the scale
// read on the device.  Not a step of the paper's method: it lets a caller
// that learns the loss gradient only after olive_token_loss_fwd_bwd (autograd)
// apply it to the gradients that call produced for a unit loss gradient.
// 16-byte vectors in a grid-stride loop (HBM-bound: 2 n elt bytes moved).
#include "internal.h"

#include <cuda_bf16.h>

namespace olive {
namespace {

__global__ void scale_bf16_kernel(const uint4* __restrict__ x, uint4* __restrict__ y, size_t n8,
                                  const __nv_bfloat16* __restrict__ xt, __nv_bfloat16* yt,
                                  size_t tail, const float* __restrict__ scale) {
  const float s = *scale;
  const size_t stride = static_cast<size_t>(gridDim.x) * blockDim.x;
  for (size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n8; i += stride) {
    uint4 v = x[i];
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&v);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = __bfloat1622float2(h[q]);
      h[q] = __floats2bfloat162_rn(f.x * s, f.y * s);
    }
    y[i] = v;
  }
  if (blockIdx.x == 0 && threadIdx.x < tail)
    yt[threadIdx.x] = __float2bfloat16_rn(__bfloat162float(xt[threadIdx.x]) * s);
}

__global__ void scale_f32_kernel(const float4* __restrict__ x, float4* __restrict__ y, size_t n4,
                                 const float* __restrict__ xt, float* yt, size_t tail,
                                 const float* __restrict__ scale) {
  const float s = *scale;
  const size_t stride = static_cast<size_t>(gridDim.x) * blockDim.x;
  for (size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const float4 v = x[i];
    y[i] = make_float4(v.x * s, v.y * s, v.z * s, v.w * s);
  }
  if (blockIdx.x == 0 && threadIdx.x < tail) yt[threadIdx.x] = xt[threadIdx.x] * s;
}

}  // namespace

olive_status launch_scale(const Ctx& c, const void* x, void* y, size_t n, int dtype,
                          const float* scale) {
  const int threads = 256;
  const int blocks = c.num_sms * 8;
  if (dtype == OLIVE_DTYPE_BF16) {
    const size_t n8 = n / 8;
    scale_bf16_kernel<<<blocks, threads, 0, c.stream>>>(
        static_cast<const uint4*>(x), static_cast<uint4*>(y), n8,
        static_cast<const __nv_bfloat16*>(x) + 8 * n8, static_cast<__nv_bfloat16*>(y) + 8 * n8,
        n - 8 * n8, scale);
  } else {
    const size_t n4 = n / 4;
    scale_f32_kernel<<<blocks, threads, 0, c.stream>>>(
        static_cast<const float4*>(x), static_cast<float4*>(y), n4,
        static_cast<const float*>(x) + 4 * n4, static_cast<float*>(y) + 4 * n4, n - 4 * n4, scale);
  }
  return cudaGetLastError() == cudaSuccess ? OLIVE_OK : OLIVE_ERR_CUDA;
}

}  // namespace olive
