// Memory-bound kernels of the decoder layer (RC_OP_DECODER_LAYER) around its
// GEMMs and attention: RMSNorm, and RoPE with the split of the fused QKV
// projection into contiguous Q, K, V heads. (The residual adds happen in the
// O and down GEMMs' epilogues.) Both read and write 16-byte vectors of bf16
// and compute in fp32.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>

#include "rc_internal.h"

namespace {

union V8 {
  uint4 u;
  __nv_bfloat16 h[8];
};

// One CTA per row; each thread loads up to kMaxVec 16-byte vectors (8
// elements each) at once and keeps them in registers between the sum of
// squares and the scaling: y = x / sqrt(mean(x^2) + eps) * g. H % 256 == 0,
// blockDim = the multiple of 32 that covers H / 8 in at most kMaxVec
// vectors per thread (128 threads at H = 4096).
constexpr int kMaxVec = 4;

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x / 32, nw = blockDim.x / 32;
  if (threadIdx.x % 32 == 0) red[w] = v;
  __syncthreads();
  float s = 0.f;
  for (int i = 0; i < nw; ++i) s += red[i];  // every thread sums the warp totals in the same order
  return s;
}

__global__ void rmsnorm_kernel(const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ g, int H,
                               float eps, __nv_bfloat16* __restrict__ y) {
  __shared__ float red[32];
  const int64_t off = (int64_t)blockIdx.x * H;
  const int nvec = H / 8;
  V8 a[kMaxVec];
#pragma unroll
  for (int i = 0; i < kMaxVec; ++i) {  // every load in flight before the first use
    const int v = threadIdx.x + i * blockDim.x;
    a[i].u = v < nvec ? reinterpret_cast<const uint4*>(x + off)[v] : make_uint4(0, 0, 0, 0);
  }
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxVec; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float f = __bfloat162float(a[i].h[j]);
      ss = fmaf(f, f, ss);
    }
  const float inv = rsqrtf(block_sum(ss, red) / (float)H + eps);
#pragma unroll
  for (int i = 0; i < kMaxVec; ++i) {
    const int v = threadIdx.x + i * blockDim.x;
    if (v >= nvec) break;
    V8 gg, o;
    gg.u = reinterpret_cast<const uint4*>(g)[v];
#pragma unroll
    for (int j = 0; j < 8; ++j)
      o.h[j] = __float2bfloat16_rn(__bfloat162float(a[i].h[j]) * inv * __bfloat162float(gg.h[j]));
    reinterpret_cast<uint4*>(y + off)[v] = o.u;
  }
}

// Inverse frequencies theta^(-2j/D) of the D/2 rotation pairs (computed in
// fp64 on the host, rounded once to fp32).
template <int D>
struct InvFreq {
  float v[D / 2];
};

// qkv[T][(Hq + 2 Hkv) D] -> Q[T][Hq][D], K[T][Hkv][D] rotated, V[T][Hkv][D] copied.
// Rotate-half pairing: element j and j + D/2 of a head turn by p * theta^(-2j/D).
// A CTA handles `per` (<= 8) consecutive tokens: their cos/sin are formed once
// in shared memory (fp32 angle p * inv_freq[j], at most ~2^-13 rad off at
// p = 2047, far below the bf16 rounding of the output), then each thread
// rotates 8 pairs per unit with 16-byte loads and stores, several units at a
// time.
template <int D>
__global__ void rope_split_kernel(const __nv_bfloat16* __restrict__ qkv, int T, int Hq, int Hkv,
                                  const InvFreq<D> invf, int per, __nv_bfloat16* __restrict__ Q,
                                  __nv_bfloat16* __restrict__ K, __nv_bfloat16* __restrict__ V) {
  __shared__ float cs[8][D / 2], sn[8][D / 2];
  const int t0 = blockIdx.x * per;
  const int nt = min(per, T - t0);
  for (int e = threadIdx.x; e < nt * (D / 2); e += blockDim.x) {
    const int tt = e / (D / 2), j = e % (D / 2);
    float s, c;
    sincosf((float)(t0 + tt) * invf.v[j], &s, &c);
    cs[tt][j] = c;
    sn[tt][j] = s;
  }
  __syncthreads();
  constexpr int G = D / 16;  // groups of 8 pairs per head
  const int width = (Hq + 2 * Hkv) * D;
  const int rot_units = (Hq + Hkv) * G;
  const int units = rot_units + Hkv * D / 8;
  // kUnits units in flight per thread: all their loads are issued before the first use
  constexpr int kUnits = 4;
  const int total = nt * units;
  for (int base = threadIdx.x; base < total; base += kUnits * blockDim.x) {
    V8 lo[kUnits], hi[kUnits];
#pragma unroll
    for (int q = 0; q < kUnits; ++q) {
      const int e = base + q * blockDim.x;
      if (e >= total) break;
      const int tt = e / units, u = e % units;
      const __nv_bfloat16* row = qkv + (int64_t)(t0 + tt) * width;
      if (u < rot_units) {
        const int hd = u / G, j0 = (u % G) * 8;
        lo[q].u = *reinterpret_cast<const uint4*>(row + hd * D + j0);
        hi[q].u = *reinterpret_cast<const uint4*>(row + hd * D + D / 2 + j0);
      } else {
        lo[q].u = *reinterpret_cast<const uint4*>(row + (Hq + Hkv) * D + (u - rot_units) * 8);
      }
    }
#pragma unroll
    for (int q = 0; q < kUnits; ++q) {
      const int e = base + q * blockDim.x;
      if (e >= total) break;
      const int tt = e / units, u = e % units;
      const int64_t t = t0 + tt;
      if (u < rot_units) {
        const int hd = u / G, j0 = (u % G) * 8;
        V8 olo, ohi;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float c = cs[tt][j0 + i], s = sn[tt][j0 + i];
          const float l = __bfloat162float(lo[q].h[i]), h = __bfloat162float(hi[q].h[i]);
          olo.h[i] = __float2bfloat16_rn(l * c - h * s);
          ohi.h[i] = __float2bfloat16_rn(h * c + l * s);
        }
        __nv_bfloat16* dst = hd < Hq ? Q + (t * Hq + hd) * D : K + (t * Hkv + (hd - Hq)) * D;
        *reinterpret_cast<uint4*>(dst + j0) = olo.u;
        *reinterpret_cast<uint4*>(dst + D / 2 + j0) = ohi.u;
      } else {
        reinterpret_cast<uint4*>(V + t * Hkv * D)[u - rot_units] = lo[q].u;
      }
    }
  }
}

rc_status launched(const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "%s launch: %s", what, cudaGetErrorString(e));
  return RC_OK;
}

}  // namespace

rc_status rc_launch_rmsnorm(const void* x, const void* g, int64_t rows, int64_t H, double eps, void* y,
                            const LaunchCtx& c) {
  if (H % 256 || H / 8 > 1024 * kMaxVec)
    return rc_fail(RC_ERR_UNSUPPORTED_OP, "rmsnorm: hidden must be a multiple of 256 and at most 32768");
  if (rows <= 0) return RC_OK;
  if (rows > 0x7fffffffLL) return rc_fail(RC_ERR_UNSUPPORTED_OP, "rmsnorm: too many rows");
  const int64_t per_thread = (H / 8 + kMaxVec - 1) / kMaxVec;
  const int threads = (int)std::min<int64_t>((per_thread + 31) / 32 * 32, 1024);
  rmsnorm_kernel<<<(unsigned)rows, threads, 0, (cudaStream_t)c.stream>>>(
      (const __nv_bfloat16*)x, (const __nv_bfloat16*)g, (int)H, (float)eps, (__nv_bfloat16*)y);
  return launched("rmsnorm");
}

rc_status rc_launch_rope_split(const rc_knobs& k, const void* qkv, int64_t T, int64_t Hq, int64_t Hkv, int64_t D,
                               double theta, void* Q, void* K, void* V, const LaunchCtx& c) {
  if (D != 128) return rc_fail(RC_ERR_UNSUPPORTED_OP, "rope: head_dim must be 128");
  const int per = k.tile_m;
  if (per < 1 || per > 8) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "rope: 1 to 8 tokens per CTA");
  if (T <= 0) return RC_OK;
  if (T > 0x7fffffffLL || (Hq + 2 * Hkv) * D * 8 > 0x7fffffffLL)
    return rc_fail(RC_ERR_UNSUPPORTED_OP, "rope: sizes out of range");
  InvFreq<128> f;
  for (int j = 0; j < 64; ++j) f.v[j] = (float)std::pow(theta, -2.0 * j / 128.0);
  const int64_t blocks = (T + per - 1) / per;
  rope_split_kernel<128><<<(unsigned)blocks, 256, 0, (cudaStream_t)c.stream>>>(
      (const __nv_bfloat16*)qkv, (int)T, (int)Hq, (int)Hkv, f, per, (__nv_bfloat16*)Q, (__nv_bfloat16*)K,
      (__nv_bfloat16*)V);
  return launched("rope");
}
