// Memory-bound passes that unfused schedules run after a GEMM, plus the L2
// flush used between timed runs. Every pass moves 16-byte vectors (8 bf16 or
// 4 fp32) per thread with a grid-stride loop sized to the SM count.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "rc_internal.h"

namespace {

__device__ __forceinline__ float silu_f(float x) { return x / (1.f + __expf(-x)); }

union V8 {
  uint4 u;
  __nv_bfloat16 h[8];
};

int grid_for(int64_t work, const LaunchCtx& c, int threads = 256) {
  int64_t g = (work + threads - 1) / threads;
  const int64_t cap = (int64_t)c.num_sms * 8;
  if (g > cap) g = cap;
  return (int)(g < 1 ? 1 : g);
}

// h[m, n] = silu(gu[m, n]) * gu[m, I + n]; I % 8 == 0.
__global__ void swiglu_pass_kernel(const __nv_bfloat16* __restrict__ gu, int64_t M, int64_t I,
                                   __nv_bfloat16* __restrict__ h) {
  const int64_t per_row = I / 8;
  const int64_t total = M * per_row;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < total;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t m = v / per_row, c = (v % per_row) * 8;
    V8 g, u, o;
    g.u = *reinterpret_cast<const uint4*>(gu + m * 2 * I + c);
    u.u = *reinterpret_cast<const uint4*>(gu + m * 2 * I + I + c);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float gf = __bfloat162float(g.h[i]);
      o.h[i] = __float2bfloat16_rn(silu_f(gf) * __bfloat162float(u.h[i]));
    }
    *reinterpret_cast<uint4*>(h + m * I + c) = o.u;
  }
}

// out[r, c] = act(y[r, c] + bias[c]); C % 8 == 0.
__global__ void bias_silu_pass_kernel(const __nv_bfloat16* __restrict__ y, const __nv_bfloat16* __restrict__ bias,
                                      int64_t rows, int64_t C, int silu, __nv_bfloat16* __restrict__ out) {
  const int64_t per_row = C / 8;
  const int64_t total = rows * per_row;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < total;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t c = (v % per_row) * 8;
    V8 a, o;
    a.u = *reinterpret_cast<const uint4*>(y + v * 8);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float f = __bfloat162float(a.h[i]) + (bias ? __bfloat162float(bias[c + i]) : 0.f);
      o.h[i] = __float2bfloat16_rn(silu ? silu_f(f) : f);
    }
    *reinterpret_cast<uint4*>(out + v * 8) = o.u;
  }
}

// out[m, n] = bf16(sum_z part[z, m, n]); N % 4 == 0.
__global__ void splitk_reduce_kernel(const float* __restrict__ part, int splits, int64_t MN,
                                     __nv_bfloat16* __restrict__ out) {
  const int64_t total = MN / 4;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < total;
       v += (int64_t)gridDim.x * blockDim.x) {
    float4 s = reinterpret_cast<const float4*>(part)[v];
    for (int z = 1; z < splits; ++z) {
      const float4 p = reinterpret_cast<const float4*>(part + (int64_t)z * MN)[v];
      s.x += p.x;
      s.y += p.y;
      s.z += p.z;
      s.w += p.w;
    }
    __nv_bfloat162 lo = __floats2bfloat162_rn(s.x, s.y), hi = __floats2bfloat162_rn(s.z, s.w);
    uint2 pk;
    pk.x = *reinterpret_cast<uint32_t*>(&lo);
    pk.y = *reinterpret_cast<uint32_t*>(&hi);
    reinterpret_cast<uint2*>(out)[v] = pk;
  }
}

// xp[n][p + pad][q + pad][c] = x[n][p][q][c], zero border of width `pad`.
__global__ void pad_nhwc_kernel(const uint4* __restrict__ x, int64_t N, int64_t H, int64_t W, int64_t C16,
                                int64_t pad, uint4* __restrict__ xp) {
  const int64_t Hp = H + 2 * pad, Wp = W + 2 * pad;
  const int64_t total = N * Hp * Wp * C16;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < total; v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t c = v % C16;
    const int64_t pix = v / C16;
    const int64_t q = pix % Wp, p = (pix / Wp) % Hp, n = pix / (Wp * Hp);
    const int64_t ih = p - pad, iw = q - pad;
    xp[v] = (ih >= 0 && ih < H && iw >= 0 && iw < W) ? x[((n * H + ih) * W + iw) * C16 + c] : make_uint4(0, 0, 0, 0);
  }
}

__global__ void f32_to_bf16_kernel(const float* __restrict__ in, int64_t n4, __nv_bfloat16* __restrict__ out) {
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < n4; v += (int64_t)gridDim.x * blockDim.x) {
    const float4 s = reinterpret_cast<const float4*>(in)[v];
    __nv_bfloat162 lo = __floats2bfloat162_rn(s.x, s.y), hi = __floats2bfloat162_rn(s.z, s.w);
    uint2 pk;
    pk.x = *reinterpret_cast<uint32_t*>(&lo);
    pk.y = *reinterpret_cast<uint32_t*>(&hi);
    reinterpret_cast<uint2*>(out)[v] = pk;
  }
}

__global__ void l2_flush_kernel(uint4* buf, int64_t n16) {
  const uint4 v = make_uint4(threadIdx.x, blockIdx.x, 0x5a5a5a5a, 0);
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n16; i += (int64_t)gridDim.x * blockDim.x)
    buf[i] = v;
}

rc_status launched(const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "%s launch: %s", what, cudaGetErrorString(e));
  return RC_OK;
}

}  // namespace

rc_status rc_launch_swiglu_pass(const void* gu, int64_t M, int64_t I, void* h, int vec, const LaunchCtx& c) {
  (void)vec;
  if (I % 8) return rc_fail(RC_ERR_UNSUPPORTED_OP, "swiglu pass: I %% 8 != 0");
  swiglu_pass_kernel<<<grid_for(M * I / 8, c), 256, 0, (cudaStream_t)c.stream>>>(
      (const __nv_bfloat16*)gu, M, I, (__nv_bfloat16*)h);
  return launched("swiglu pass");
}

rc_status rc_launch_bias_silu_pass(const void* y, const void* bias, int64_t rows, int64_t C, bool silu, void* out,
                                   int vec, const LaunchCtx& c) {
  (void)vec;
  if (C % 8) return rc_fail(RC_ERR_UNSUPPORTED_OP, "bias/SiLU pass: C %% 8 != 0");
  bias_silu_pass_kernel<<<grid_for(rows * C / 8, c), 256, 0, (cudaStream_t)c.stream>>>(
      (const __nv_bfloat16*)y, (const __nv_bfloat16*)bias, rows, C, silu ? 1 : 0, (__nv_bfloat16*)out);
  return launched("bias/SiLU pass");
}

rc_status rc_launch_splitk_reduce(const float* part, int splits, int64_t M, int64_t N, void* out, int vec,
                                  const LaunchCtx& c) {
  (void)vec;
  if (N % 4) return rc_fail(RC_ERR_UNSUPPORTED_OP, "split-K reduce: N %% 4 != 0");
  splitk_reduce_kernel<<<grid_for(M * N / 4, c), 256, 0, (cudaStream_t)c.stream>>>(part, splits, M * N,
                                                                                   (__nv_bfloat16*)out);
  return launched("split-K reduce");
}

rc_status rc_launch_f32_to_bf16(const float* in, int64_t n, void* out, const LaunchCtx& c) {
  if (n % 4) return rc_fail(RC_ERR_UNSUPPORTED_OP, "f32->bf16: n %% 4 != 0");
  f32_to_bf16_kernel<<<grid_for(n / 4, c), 256, 0, (cudaStream_t)c.stream>>>(in, n / 4, (__nv_bfloat16*)out);
  return launched("f32->bf16");
}

rc_status rc_launch_pad_nhwc(const void* x, int64_t N, int64_t H, int64_t W, int64_t C, int64_t pad, void* xp,
                              const LaunchCtx& c) {
  if (C % 8) return rc_fail(RC_ERR_UNSUPPORTED_OP, "pad: C %% 8 != 0");
  const int64_t total = N * (H + 2 * pad) * (W + 2 * pad) * (C / 8);
  pad_nhwc_kernel<<<grid_for(total, c), 256, 0, (cudaStream_t)c.stream>>>((const uint4*)x, N, H, W, C / 8, pad,
                                                                          (uint4*)xp);
  return launched("pad");
}

rc_status rc_launch_l2_flush(void* buf, size_t bytes, void* stream) {
  l2_flush_kernel<<<1024, 256, 0, (cudaStream_t)stream>>>((uint4*)buf, (int64_t)(bytes / 16));
  return launched("L2 flush");
}
