// fp32 GEMM + bias + ReLU on the CUDA cores (FFMA only; TF32 tensor cores
// would not hold a 1e-4 relative error).
//
// The loop nest is the one of the paper's App. A example, C[i,j] = 0 then
// C[i,j] += A[i,k] B[k,j], with a bias over j and a ReLU added. The schedule
// space is the CTA tile (BM, BN, BK) in {16, 32, 64}^3 times the unroll
// factor {1, 4} of the k loop over the shared-memory tile: 54 compiled
// kernels, selected at run time by the TileSize and Unroll knobs.
//
// Mapping: 256 threads as a 16 x 16 grid; thread (ty, tx) owns the
// (BM/16) x (BN/16) outputs at rows ty + 16 i and columns tx + 16 j, so
// shared-memory reads along a warp are broadcast (A) or consecutive (B).
// Ragged M, N and K are handled by zero-filled tile loads and guarded stores.
#include <cuda_runtime.h>

#include "rc_internal.h"

namespace {

template <int BM, int BN, int BK, int UNROLL>
__global__ void __launch_bounds__(256) gemm_f32_kernel(int M, int N, int K, const float* __restrict__ A,
                                                       const float* __restrict__ B,
                                                       const float* __restrict__ bias, float* __restrict__ C,
                                                       int relu) {
  constexpr int TM = BM / 16, TN = BN / 16;
  __shared__ float As[BK][BM + 1];  // As[k][m]: A tile transposed
  __shared__ float Bs[BK][BN];
  const int tid = threadIdx.x;
  const int tx = tid % 16, ty = tid / 16;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < K; k0 += BK) {
    for (int e = tid; e < BM * BK; e += 256) {
      const int m = e / BK, k = e % BK;  // consecutive threads walk along k (coalesced)
      const int gm = m0 + m, gk = k0 + k;
      As[k][m] = (gm < M && gk < K) ? A[(size_t)gm * K + gk] : 0.f;
    }
    for (int e = tid; e < BK * BN; e += 256) {
      const int k = e / BN, n = e % BN;
      const int gk = k0 + k, gn = n0 + n;
      Bs[k][n] = (gk < K && gn < N) ? B[(size_t)gk * N + gn] : 0.f;
    }
    __syncthreads();
#pragma unroll UNROLL
    for (int kk = 0; kk < BK; ++kk) {
      float a[TM], b[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < TN; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int gm = m0 + ty + 16 * i;
    if (gm >= M) continue;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int gn = n0 + tx + 16 * j;
      if (gn >= N) continue;
      float v = acc[i][j] + (bias ? bias[gn] : 0.f);
      if (relu) v = fmaxf(v, 0.f);
      C[(size_t)gm * N + gn] = v;
    }
  }
}

using KFn = void (*)(int, int, int, const float*, const float*, const float*, float*, int);

template <int BM, int BN, int BK>
KFn pick_unroll(int u) {
  return u == 4 ? gemm_f32_kernel<BM, BN, BK, 4> : gemm_f32_kernel<BM, BN, BK, 1>;
}
template <int BM, int BN>
KFn pick_bk(int bk, int u) {
  switch (bk) {
    case 16: return pick_unroll<BM, BN, 16>(u);
    case 32: return pick_unroll<BM, BN, 32>(u);
    case 64: return pick_unroll<BM, BN, 64>(u);
  }
  return nullptr;
}
template <int BM>
KFn pick_bn(int bn, int bk, int u) {
  switch (bn) {
    case 16: return pick_bk<BM, 16>(bk, u);
    case 32: return pick_bk<BM, 32>(bk, u);
    case 64: return pick_bk<BM, 64>(bk, u);
  }
  return nullptr;
}
KFn pick(int bm, int bn, int bk, int u) {
  if (u != 1 && u != 4) return nullptr;
  switch (bm) {
    case 16: return pick_bn<16>(bn, bk, u);
    case 32: return pick_bn<32>(bn, bk, u);
    case 64: return pick_bn<64>(bn, bk, u);
  }
  return nullptr;
}

}  // namespace

rc_status rc_launch_gemm_f32(const rc_knobs& k, int64_t M, int64_t N, int64_t K, const float* A,
                             const float* B, const float* bias, float* C, bool relu, const LaunchCtx& c) {
  KFn fn = pick(k.tile_m, k.tile_n, k.tile_k, k.unroll);
  if (!fn) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "gemm_f32: no kernel for tile %dx%dx%d unroll %d", k.tile_m,
                          k.tile_n, k.tile_k, k.unroll);
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return rc_fail(RC_ERR_UNSUPPORTED_OP, "gemm_f32: size");
  const int64_t gy = (M + k.tile_m - 1) / k.tile_m;
  if (gy > 65535) return rc_fail(RC_ERR_UNSUPPORTED_OP, "gemm_f32: M too large for the grid");
  dim3 grid((unsigned)((N + k.tile_n - 1) / k.tile_n), (unsigned)gy);
  fn<<<grid, 256, 0, (cudaStream_t)c.stream>>>((int)M, (int)N, (int)K, A, B, bias, C, relu ? 1 : 0);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "gemm_f32 launch: %s", cudaGetErrorString(e));
  return RC_OK;
}
