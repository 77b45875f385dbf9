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
// Tiles stream through a ring of shared-memory stages with cp.async, so
// several k blocks are in flight. Ragged M, N and K are handled by
// zero-filled tile loads and guarded stores.
#include <cuda_runtime.h>

#include "rc_internal.h"

namespace {

// Shared-memory ring depth: as many BK-deep stages as fit in 40 KB of static
// shared memory (at most 8), so that the global-memory latency of a k block is
// paid once per ring rather than once per block; a single stage (synchronous
// loads) when two do not fit.
template <int BM, int BN, int BK>
constexpr int k0_stages() {
  constexpr int bytes = (BM * (BK + 1) + BK * BN) * 4;
  constexpr int n = 40960 / bytes;
  return n >= 8 ? 8 : n >= 2 ? n : 1;
}

// 4-byte global -> shared copy (cp.async); src_bytes = 0 zero-fills.
__device__ __forceinline__ void cp_async4(float* dst, const float* src, uint32_t src_bytes) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(d), "l"(src), "r"(src_bytes) : "memory");
}

template <int BM, int BN, int BK, int UNROLL>
__global__ void __launch_bounds__(256) gemm_f32_kernel(int M, int N, int K, const float* __restrict__ A,
                                                       const float* __restrict__ B,
                                                       const float* __restrict__ bias, float* __restrict__ C,
                                                       int relu) {
  constexpr int TM = BM / 16, TN = BN / 16;
  constexpr int S = k0_stages<BM, BN, BK>();
  __shared__ float As[S][BM][BK + 1];  // As[s][m][k]
  __shared__ float Bs[S][BK][BN];
  const int tid = threadIdx.x;
  const int tx = tid % 16, ty = tid / 16;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const int nkb = (K + BK - 1) / BK;
  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

  // one k block into ring slot st (zero-filled outside M, N, K); consecutive threads walk along k for
  // A and along n for B (coalesced)
  auto load = [&](int st, int k0) {
    for (int e = tid; e < BM * BK; e += 256) {
      const int m = e / BK, k = e % BK;
      const int gm = m0 + m, gk = k0 + k;
      const bool v = gm < M && gk < K;
      cp_async4(&As[st][m][k], v ? A + (size_t)gm * K + gk : A, v ? 4u : 0u);
    }
    for (int e = tid; e < BK * BN; e += 256) {
      const int k = e / BN, n = e % BN;
      const int gk = k0 + k, gn = n0 + n;
      const bool v = gk < K && gn < N;
      cp_async4(&Bs[st][k][n], v ? B + (size_t)gk * N + gn : B, v ? 4u : 0u);
    }
  };
  // prologue: blocks 0 .. S - 2 (block 0 alone for a single stage)
#pragma unroll
  for (int st = 0; st < (S > 1 ? S - 1 : 1); ++st) {
    if (st < nkb) load(st, st * BK);
    asm volatile("cp.async.commit_group;" ::: "memory");
  }
  for (int kb = 0; kb < nkb; ++kb) {
    // block kb has landed (at most S - 2 younger groups pending)
    asm volatile("cp.async.wait_group %0;" ::"n"(S > 1 ? S - 2 : 0) : "memory");
    __syncthreads();
    // refill the slot every thread finished reading in iteration kb - 1
    if (S > 1 && kb + S - 1 < nkb) load((kb + S - 1) % S, (kb + S - 1) * BK);
    if (S > 1) asm volatile("cp.async.commit_group;" ::: "memory");
    const int st = kb % S;
#pragma unroll UNROLL
    for (int kk = 0; kk < BK; ++kk) {
      float a[TM], b[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i) a[i] = As[st][ty + 16 * i][kk];
#pragma unroll
      for (int j = 0; j < TN; ++j) b[j] = Bs[st][kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (S == 1) {  // synchronous: the next block overwrites this slot
      __syncthreads();
      if (kb + 1 < nkb) load(0, (kb + 1) * BK);
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
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
