// Memory-bound passes that unfused schedules run after a GEMM, plus the L2
// flush used between timed runs. Each pass moves VB-byte vectors per thread
// access (the Vectorize knob: 4, 8 or 16 bytes, i.e. 2, 4 or 8 bf16) with a
// grid-stride loop sized to the SM count.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "rc_internal.h"

namespace {

__device__ __forceinline__ float silu_f(float x) { return x / (1.f + __expf(-x)); }

// VB bytes of bf16 elements, loaded and stored as one access.
template <int VB>
struct BVec;
template <>
struct BVec<16> {
  using T = uint4;
};
template <>
struct BVec<8> {
  using T = uint2;
};
template <>
struct BVec<4> {
  using T = uint32_t;
};
template <int VB>
union VecB {
  typename BVec<VB>::T u;
  __nv_bfloat16 h[VB / 2];
};

int grid_for(int64_t work, const LaunchCtx& c, int threads = 256) {
  int64_t g = (work + threads - 1) / threads;
  const int64_t cap = (int64_t)c.num_sms * 8;
  if (g > cap) g = cap;
  return (int)(g < 1 ? 1 : g);
}

// h[m, n] = silu(gu[m, n]) * gu[m, I + n]; I % 8 == 0.
template <int VB>
__global__ void swiglu_pass_kernel(const __nv_bfloat16* __restrict__ gu, int64_t M, int64_t I,
                                   __nv_bfloat16* __restrict__ h) {
  constexpr int E = VB / 2;
  const int64_t per_row = I / E;
  const int64_t total = M * per_row;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < total;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t m = v / per_row, c = (v % per_row) * E;
    VecB<VB> g, u, o;
    g.u = *reinterpret_cast<const typename BVec<VB>::T*>(gu + m * 2 * I + c);
    u.u = *reinterpret_cast<const typename BVec<VB>::T*>(gu + m * 2 * I + I + c);
#pragma unroll
    for (int i = 0; i < E; ++i) {
      const float gf = __bfloat162float(g.h[i]);
      o.h[i] = __float2bfloat16_rn(silu_f(gf) * __bfloat162float(u.h[i]));
    }
    *reinterpret_cast<typename BVec<VB>::T*>(h + m * I + c) = o.u;
  }
}

// out[r, c] = act(y[r, c] + bias[c]); C % 8 == 0.
template <int VB>
__global__ void bias_silu_pass_kernel(const __nv_bfloat16* __restrict__ y, const __nv_bfloat16* __restrict__ bias,
                                      int64_t rows, int64_t C, int silu, __nv_bfloat16* __restrict__ out) {
  constexpr int E = VB / 2;
  const int64_t per_row = C / E;
  const int64_t total = rows * per_row;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < total;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t c = (v % per_row) * E;
    VecB<VB> a, o;
    a.u = *reinterpret_cast<const typename BVec<VB>::T*>(y + v * E);
#pragma unroll
    for (int i = 0; i < E; ++i) {
      float f = __bfloat162float(a.h[i]) + (bias ? __bfloat162float(bias[c + i]) : 0.f);
      o.h[i] = __float2bfloat16_rn(silu ? silu_f(f) : f);
    }
    *reinterpret_cast<typename BVec<VB>::T*>(out + v * E) = o.u;
  }
}

// VB bytes of fp32 partials (VB / 4 floats) per access: load, sum, store as bf16.
template <int VB>
struct FVec;
template <>
struct FVec<16> {
  using T = float4;
};
template <>
struct FVec<8> {
  using T = float2;
};
template <>
struct FVec<4> {
  using T = float;
};
template <int VB>
union VecF {
  typename FVec<VB>::T v;
  float f[VB / 4];
};
template <int VB>
__device__ __forceinline__ void store_bf16(__nv_bfloat16* out, const float (&f)[VB / 4]) {
#pragma unroll
  for (int i = 0; i < VB / 4; ++i) out[i] = __float2bfloat16_rn(f[i]);
}
template <>
__device__ __forceinline__ void store_bf16<16>(__nv_bfloat16* out, const float (&f)[4]) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(f[0], f[1]), hi = __floats2bfloat162_rn(f[2], f[3]);
  uint2 pk;
  pk.x = *reinterpret_cast<uint32_t*>(&lo);
  pk.y = *reinterpret_cast<uint32_t*>(&hi);
  *reinterpret_cast<uint2*>(out) = pk;
}
template <>
__device__ __forceinline__ void store_bf16<8>(__nv_bfloat16* out, const float (&f)[2]) {
  *reinterpret_cast<__nv_bfloat162*>(out) = __floats2bfloat162_rn(f[0], f[1]);
}

// out[m, n] = bf16(sum_z part[z, m, n]); N % 4 == 0.
template <int VB>
__global__ void splitk_reduce_kernel(const float* __restrict__ part, int splits, int64_t MN,
                                     __nv_bfloat16* __restrict__ out) {
  constexpr int E = VB / 4;
  const int64_t total = MN / E;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < total;
       v += (int64_t)gridDim.x * blockDim.x) {
    VecF<VB> s;
    s.v = reinterpret_cast<const typename FVec<VB>::T*>(part)[v];
    for (int z = 1; z < splits; ++z) {
      VecF<VB> p;
      p.v = reinterpret_cast<const typename FVec<VB>::T*>(part + (int64_t)z * MN)[v];
#pragma unroll
      for (int i = 0; i < E; ++i) s.f[i] += p.f[i];
    }
    store_bf16<VB>(out + v * E, s.f);
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

template <int VB>
__global__ void f32_to_bf16_kernel(const float* __restrict__ in, int64_t n, __nv_bfloat16* __restrict__ out) {
  constexpr int E = VB / 4;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < n / E; v += (int64_t)gridDim.x * blockDim.x) {
    VecF<VB> s;
    s.v = reinterpret_cast<const typename FVec<VB>::T*>(in)[v];
    store_bf16<VB>(out + v * E, s.f);
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

// Bytes per access of the Vectorize knob: 4, 8 or 16.
static bool vec_ok(int vec) { return vec == 4 || vec == 8 || vec == 16; }

rc_status rc_launch_swiglu_pass(const void* gu, int64_t M, int64_t I, void* h, int vec, const LaunchCtx& c) {
  if (I % 8) return rc_fail(RC_ERR_UNSUPPORTED_OP, "swiglu pass: I %% 8 != 0");
  if (!vec_ok(vec)) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "swiglu pass: vector of %d bytes", vec);
  const int g = grid_for(M * I / (vec / 2), c);
  auto gp = (const __nv_bfloat16*)gu;
  auto hp = (__nv_bfloat16*)h;
  cudaStream_t st = (cudaStream_t)c.stream;
  if (vec == 16) swiglu_pass_kernel<16><<<g, 256, 0, st>>>(gp, M, I, hp);
  else if (vec == 8) swiglu_pass_kernel<8><<<g, 256, 0, st>>>(gp, M, I, hp);
  else swiglu_pass_kernel<4><<<g, 256, 0, st>>>(gp, M, I, hp);
  return launched("swiglu pass");
}

rc_status rc_launch_bias_silu_pass(const void* y, const void* bias, int64_t rows, int64_t C, bool silu, void* out,
                                   int vec, const LaunchCtx& c) {
  if (C % 8) return rc_fail(RC_ERR_UNSUPPORTED_OP, "bias/SiLU pass: C %% 8 != 0");
  if (!vec_ok(vec)) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "bias/SiLU pass: vector of %d bytes", vec);
  const int g = grid_for(rows * C / (vec / 2), c);
  auto yp = (const __nv_bfloat16*)y;
  auto bp = (const __nv_bfloat16*)bias;
  auto op = (__nv_bfloat16*)out;
  cudaStream_t st = (cudaStream_t)c.stream;
  if (vec == 16) bias_silu_pass_kernel<16><<<g, 256, 0, st>>>(yp, bp, rows, C, silu ? 1 : 0, op);
  else if (vec == 8) bias_silu_pass_kernel<8><<<g, 256, 0, st>>>(yp, bp, rows, C, silu ? 1 : 0, op);
  else bias_silu_pass_kernel<4><<<g, 256, 0, st>>>(yp, bp, rows, C, silu ? 1 : 0, op);
  return launched("bias/SiLU pass");
}

rc_status rc_launch_splitk_reduce(const float* part, int splits, int64_t M, int64_t N, void* out, int vec,
                                  const LaunchCtx& c) {
  if (N % 4) return rc_fail(RC_ERR_UNSUPPORTED_OP, "split-K reduce: N %% 4 != 0");
  if (!vec_ok(vec)) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "split-K reduce: vector of %d bytes", vec);
  const int g = grid_for(M * N / (vec / 4), c);
  auto op = (__nv_bfloat16*)out;
  cudaStream_t st = (cudaStream_t)c.stream;
  if (vec == 16) splitk_reduce_kernel<16><<<g, 256, 0, st>>>(part, splits, M * N, op);
  else if (vec == 8) splitk_reduce_kernel<8><<<g, 256, 0, st>>>(part, splits, M * N, op);
  else splitk_reduce_kernel<4><<<g, 256, 0, st>>>(part, splits, M * N, op);
  return launched("split-K reduce");
}

rc_status rc_launch_f32_to_bf16(const float* in, int64_t n, void* out, int vec, const LaunchCtx& c) {
  if (n % 4) return rc_fail(RC_ERR_UNSUPPORTED_OP, "f32->bf16: n %% 4 != 0");
  if (!vec_ok(vec)) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "f32->bf16: vector of %d bytes", vec);
  const int g = grid_for(n / (vec / 4), c);
  auto op = (__nv_bfloat16*)out;
  cudaStream_t st = (cudaStream_t)c.stream;
  if (vec == 16) f32_to_bf16_kernel<16><<<g, 256, 0, st>>>(in, n, op);
  else if (vec == 8) f32_to_bf16_kernel<8><<<g, 256, 0, st>>>(in, n, op);
  else f32_to_bf16_kernel<4><<<g, 256, 0, st>>>(in, n, op);
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
