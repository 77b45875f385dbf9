// MoE routing, gather and combine kernels.
//
// Routing (bit-exact ids / offsets / permutation):
//   1) route_topk: one warp per token. The E logits are widened exactly to
//      fp32, the softmax normaliser z = sum_e exp(l_e - max) is reduced over
//      the warp, and k arg-max rounds pick the experts in the order
//      (logit descending, expert id ascending) by comparing the widened
//      logits only. Weights w_j = exp(l_j - max) / z, renormalised over the k
//      picks when requested. A NaN logit is read as -inf: it ranks below every
//      number (ties by lower id) and gets probability 0, so every round picks
//      an id below E whatever the logits hold.
//   2) route_count: each CTA histograms 4096 slots' expert ids in shared
//      memory and adds its non-zero bins to the per-expert counts (integer
//      atomics: the totals do not depend on their order).
//   3) route_permute: one CTA per expert takes the exclusive prefix of the
//      counts as its offset and ranks the slots whose id is e in slot order
//      (coalesced striped loads, warp ballots, one block-wide scan of the
//      per-warp hit counts per chunk), so slot s = t*k + j lands at
//      perm[offset[e] + rank] - the (expert, token, j) order - with no
//      dependence on thread timing.
// Gather: Xp[pos] = X[perm[pos] / k], one warp per row, 4-, 8- or 16-byte
//   vectors (the Vectorize knob).
// Combine: out[t] = sum_{j<k} w[t,j] * Y[inv_perm[t*k+j]] in fp32, in j order,
//   rounded once to bf16, with the same choice of vector width.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "rc_internal.h"

namespace {

constexpr int kMaxE = 256;
constexpr int kMaxPerLane = kMaxE / 32;
constexpr int kMaxK = 16;

// (value, id) order of the selection: a beats b if larger, or equal and lower id.
__device__ __forceinline__ bool beats(float va, int ia, float vb, int ib) {
  return va > vb || (va == vb && ia < ib);
}

template <bool FP32>
__global__ void route_topk_kernel(const void* __restrict__ logits, int T, int E, int K, int renorm,
                                  int* __restrict__ ids, float* __restrict__ w) {
  const int warps = blockDim.x / 32;
  const int t = blockIdx.x * warps + threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  if (t >= T) return;
  float v[kMaxPerLane];
  bool taken[kMaxPerLane];
  float mx = -INFINITY;
#pragma unroll
  for (int i = 0; i < kMaxPerLane; ++i) {
    const int e = lane + 32 * i;
    taken[i] = false;
    if (e < E) {
      const float x = FP32 ? ((const float*)logits)[(size_t)t * E + e]
                           : __bfloat162float(((const __nv_bfloat16*)logits)[(size_t)t * E + e]);
      v[i] = x != x ? -INFINITY : x;  // NaN ranks last
      mx = fmaxf(mx, v[i]);
    } else {
      v[i] = -INFINITY;
      taken[i] = true;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  float z = 0.f;
#pragma unroll
  for (int i = 0; i < kMaxPerLane; ++i)
    if (lane + 32 * i < E) z += expf(v[i] - mx);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);

  float pk[kMaxK];
  int ik[kMaxK];
  float sel = 0.f;
  for (int j = 0; j < K; ++j) {
    // best untaken candidate of this lane
    float bv = -INFINITY;
    int bi = 0x7fffffff;
#pragma unroll
    for (int i = 0; i < kMaxPerLane; ++i) {
      const int e = lane + 32 * i;
      if (!taken[i] && beats(v[i], e, bv, bi)) {
        bv = v[i];
        bi = e;
      }
    }
    // warp arg-max under the same order
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (beats(ov, oi, bv, bi)) {
        bv = ov;
        bi = oi;
      }
    }
    // Each untaken expert beats the (-inf, INT_MAX) start and K <= E, so bi < E;
    // the guard keeps an out-of-range index from ever being written.
    bi = bi < E ? bi : 0;
    if ((bi & 31) == lane) taken[bi >> 5] = true;
    const float p = expf(bv - mx) / z;
    pk[j] = p;
    ik[j] = bi;
    sel += p;
  }
  if (lane < K) {
    float p = 0.f;
    int id = 0;
    for (int j = 0; j < K; ++j)
      if (j == lane) {
        p = pk[j];
        id = ik[j];
      }
    ids[(size_t)t * K + lane] = id;
    w[(size_t)t * K + lane] = renorm ? p / sel : p;
  }
}

constexpr int kCountThreads = 256;
constexpr int kCountSlots = 16;  // slots per thread

__global__ void __launch_bounds__(kCountThreads)
    route_count_kernel(const int* __restrict__ ids, int slots, int E, int* __restrict__ counts) {
  __shared__ int hist[kMaxE];
  for (int e = threadIdx.x; e < E; e += blockDim.x) hist[e] = 0;
  __syncthreads();
  const int s0 = blockIdx.x * (kCountThreads * kCountSlots);
  int id[kCountSlots];
#pragma unroll
  for (int q = 0; q < kCountSlots; ++q) {  // loads first, coalesced across the CTA
    const int s = s0 + q * kCountThreads + threadIdx.x;
    id[q] = s < slots ? ids[s] : -1;
  }
#pragma unroll
  for (int q = 0; q < kCountSlots; ++q)
    if (id[q] >= 0 && id[q] < E) atomicAdd(&hist[id[q]], 1);
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x)
    if (hist[e]) atomicAdd(&counts[e], hist[e]);
}

constexpr int kPermThreads = 1024;  // 32 warps
constexpr int kPermRounds = 16;     // slots per thread and chunk: a chunk is 16384 consecutive slots

// Slots are read striped (slot c0 + q*1024 + warp*32 + lane), so every load is
// coalesced. A slot is a hit when its id is e; since a token's k ids are
// distinct, ranking hits by slot index ranks them by token.
__global__ void __launch_bounds__(kPermThreads)
    route_permute_kernel(const int* __restrict__ ids, int T, int K, int E, const int* __restrict__ counts,
                         int* __restrict__ offsets, int* __restrict__ perm, int* __restrict__ inv_perm) {
  constexpr int NW = kPermThreads / 32;
  constexpr int NV = kPermRounds * NW;  // per-(round, warp) hit counts of a chunk
  const int e = blockIdx.x;
  __shared__ int base_s;
  __shared__ int scan[NV];
  __shared__ int warp_tot[NW];
  const int lane = threadIdx.x % 32, warp = threadIdx.x / 32;
  if (warp == 0) {  // offset of e = sum of the counts before it; all E counts loaded at once
    int before = 0, mine = 0;
#pragma unroll
    for (int r = 0; r < kMaxPerLane; ++r) {
      const int i = lane + 32 * r;
      const int c = i < E ? counts[i] : 0;
      before += i < e ? c : 0;
      mine += i == e ? c : 0;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      before += __shfl_xor_sync(0xffffffffu, before, o);
      mine += __shfl_xor_sync(0xffffffffu, mine, o);
    }
    if (lane == 0) {
      base_s = before;
      offsets[e] = before;
      if (e == E - 1) offsets[E] = before + mine;
    }
  }
  __syncthreads();
  int running = base_s;
  const int slots = T * K;
  for (int c0 = 0; c0 < slots; c0 += kPermThreads * kPermRounds) {
    int v[kPermRounds];
#pragma unroll
    for (int q = 0; q < kPermRounds; ++q) {  // every load of the chunk in flight before any use
      const int sl = c0 + q * kPermThreads + warp * 32 + lane;
      v[q] = sl < slots ? ids[sl] : -1;
    }
    unsigned bal[kPermRounds];
#pragma unroll
    for (int q = 0; q < kPermRounds; ++q) bal[q] = __ballot_sync(0xffffffffu, v[q] == e);
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < kPermRounds; ++q) scan[q * NW + warp] = __popc(bal[q]);
    }
    __syncthreads();
    // exclusive scan of the NV counts in (round, warp) order = slot order, one count per thread
    const int x = threadIdx.x < NV ? scan[threadIdx.x] : 0;
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    int before = 0, total = 0;
    for (int i = 0; i < NW; ++i) {
      const int c = warp_tot[i];
      before += i < warp ? c : 0;
      total += c;
    }
    __syncthreads();  // every thread has its count and the warp totals before scan[] is overwritten
    if (threadIdx.x < NV) scan[threadIdx.x] = before + incl - x;
    __syncthreads();
#pragma unroll
    for (int q = 0; q < kPermRounds; ++q) {
      if (!((bal[q] >> lane) & 1u)) continue;
      const int sl = c0 + q * kPermThreads + warp * 32 + lane;
      const int pos = running + scan[q * NW + warp] + __popc(bal[q] & ((1u << lane) - 1u));
      perm[pos] = sl;
      if (inv_perm) inv_perm[sl] = pos;
    }
    running += total;
    __syncthreads();  // scan[] and warp_tot[] are rewritten by the next chunk
  }
}

// VB-byte vectors of the Vectorize knob (4, 8 or 16 bytes per access).
template <int VB>
struct Vec;
template <>
struct Vec<16> {
  using T = uint4;
};
template <>
struct Vec<8> {
  using T = uint2;
};
template <>
struct Vec<4> {
  using T = uint32_t;
};

// One warp per grouped row: four vector loads in flight per lane before their stores. The source
// rows (each read by k slots) are left in L2; the grouped copy is written with the streaming hint.
template <int VB>
__global__ void gather_rows_kernel(const typename Vec<VB>::T* __restrict__ X, const int* __restrict__ perm, int rows,
                                   int HV, int K, typename Vec<VB>::T* __restrict__ Xp) {
  using V = typename Vec<VB>::T;
  const int warps = blockDim.x / 32;
  const int lane = threadIdx.x % 32;
  for (int r = blockIdx.x * warps + threadIdx.x / 32; r < rows; r += gridDim.x * warps) {
    const int t = perm[r] / K;
    const V* src = X + (size_t)t * HV;
    V* dst = Xp + (size_t)r * HV;
    int i = lane;
    for (; i + 96 < HV; i += 128) {
      const V a = src[i], b = src[i + 32], c = src[i + 64], d = src[i + 96];
      __stcs(dst + i, a);
      __stcs(dst + i + 32, b);
      __stcs(dst + i + 64, c);
      __stcs(dst + i + 96, d);
    }
    for (; i < HV; i += 32) __stcs(dst + i, src[i]);
  }
}

template <int VB>
union VecH {
  typename Vec<VB>::T u;
  __nv_bfloat162 h[VB / 4];
};

template <int VB>
__global__ void combine_kernel(const typename Vec<VB>::T* __restrict__ Y, const float* __restrict__ w,
                               const int* __restrict__ inv_perm, int T, int HV, int K,
                               typename Vec<VB>::T* __restrict__ out) {
  constexpr int P = VB / 4;  // bf16 pairs per vector
  const int warps = blockDim.x / 32;
  const int lane = threadIdx.x % 32;
  for (int t = blockIdx.x * warps + threadIdx.x / 32; t < T; t += gridDim.x * warps) {
    int rows[kMaxK];
    float ws[kMaxK];
    for (int j = 0; j < K; ++j) {
      rows[j] = inv_perm[(size_t)t * K + j];
      ws[j] = w[(size_t)t * K + j];
    }
    for (int i = lane; i < HV; i += 32) {
      float acc[2 * P];
#pragma unroll
      for (int q = 0; q < 2 * P; ++q) acc[q] = 0.f;
      for (int j = 0; j < K; ++j) {
        VecH<VB> y;
        y.u = Y[(size_t)rows[j] * HV + i];
#pragma unroll
        for (int q = 0; q < P; ++q) {
          const float2 f = __bfloat1622float2(y.h[q]);
          acc[2 * q] = fmaf(ws[j], f.x, acc[2 * q]);
          acc[2 * q + 1] = fmaf(ws[j], f.y, acc[2 * q + 1]);
        }
      }
      VecH<VB> o;
#pragma unroll
      for (int q = 0; q < P; ++q) o.h[q] = __floats2bfloat162_rn(acc[2 * q], acc[2 * q + 1]);
      out[(size_t)t * HV + i] = o.u;
    }
  }
}

rc_status launched(const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "%s launch: %s", what, cudaGetErrorString(e));
  return RC_OK;
}

}  // namespace

rc_status rc_launch_moe_route(const rc_knobs& k, const rc_op_desc& d, const void* logits, int* ids, float* w,
                              int* offsets, int* perm, int* inv_perm, int* counts, const LaunchCtx& c) {
  const int T = (int)d.tokens, E = (int)d.experts, K = (int)d.top_k;
  if (E > kMaxE || K > kMaxK || K > E) return rc_fail(RC_ERR_UNSUPPORTED_OP, "routing: E <= 256, k <= 16");
  if ((int64_t)T * K > 0x7fffffff - 32768) return rc_fail(RC_ERR_UNSUPPORTED_OP, "routing: too many slots");
  cudaStream_t st = (cudaStream_t)c.stream;
  const int warps = k.tile_m > 0 ? k.tile_m : 4;
  const int blocks = (T + warps - 1) / warps;
  cudaError_t me = cudaMemsetAsync(counts, 0, sizeof(int) * (size_t)E, st);
  if (me != cudaSuccess) return rc_fail(RC_ERR_CUDA, "routing counts memset: %s", cudaGetErrorString(me));
  if (d.logits_fp32)
    route_topk_kernel<true><<<blocks, 32 * warps, 0, st>>>(logits, T, E, K, d.renorm, ids, w);
  else
    route_topk_kernel<false><<<blocks, 32 * warps, 0, st>>>(logits, T, E, K, d.renorm, ids, w);
  RC_TRY(launched("route_topk"));
  const int slots = T * K;
  const int cblocks = (slots + kCountThreads * kCountSlots - 1) / (kCountThreads * kCountSlots);
  route_count_kernel<<<cblocks > 0 ? cblocks : 1, kCountThreads, 0, st>>>(ids, slots, E, counts);
  RC_TRY(launched("route_count"));
  route_permute_kernel<<<E, kPermThreads, 0, st>>>(ids, T, K, E, counts, offsets, perm, inv_perm);
  return launched("route_permute");
}

rc_status rc_launch_moe_gather(const void* X, const int* perm, int64_t rows, int64_t H, int topk, void* Xp, int vec,
                               const LaunchCtx& c) {
  if (H % 8) return rc_fail(RC_ERR_UNSUPPORTED_OP, "gather: H %% 8 != 0");
  if (vec != 4 && vec != 8 && vec != 16) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "gather: vector of %d bytes", vec);
  const int warps = 8;
  int64_t blocks = (rows + warps - 1) / warps;
  if (blocks > (int64_t)c.num_sms * 16) blocks = (int64_t)c.num_sms * 16;
  const int hv = (int)(H * 2 / vec);  // vectors per row
  cudaStream_t st = (cudaStream_t)c.stream;
  if (vec == 16)
    gather_rows_kernel<16><<<(unsigned)blocks, 32 * warps, 0, st>>>((const uint4*)X, perm, (int)rows, hv, topk,
                                                                     (uint4*)Xp);
  else if (vec == 8)
    gather_rows_kernel<8><<<(unsigned)blocks, 32 * warps, 0, st>>>((const uint2*)X, perm, (int)rows, hv, topk,
                                                                    (uint2*)Xp);
  else
    gather_rows_kernel<4><<<(unsigned)blocks, 32 * warps, 0, st>>>((const uint32_t*)X, perm, (int)rows, hv, topk,
                                                                    (uint32_t*)Xp);
  return launched("gather");
}

rc_status rc_launch_moe_combine(const void* Y, const float* w, const int* inv_perm, int64_t T, int64_t H, int topk,
                                void* out, int vec, const LaunchCtx& c) {
  if (H % 8 || topk > kMaxK) return rc_fail(RC_ERR_UNSUPPORTED_OP, "combine: H %% 8 != 0 or k > 16");
  if (vec != 4 && vec != 8 && vec != 16) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "combine: vector of %d bytes", vec);
  const int warps = 8;
  int64_t blocks = (T + warps - 1) / warps;
  if (blocks > (int64_t)c.num_sms * 16) blocks = (int64_t)c.num_sms * 16;
  const int hv = (int)(H * 2 / vec);
  cudaStream_t st = (cudaStream_t)c.stream;
  if (vec == 16)
    combine_kernel<16><<<(unsigned)blocks, 32 * warps, 0, st>>>((const uint4*)Y, w, inv_perm, (int)T, hv, topk,
                                                                 (uint4*)out);
  else if (vec == 8)
    combine_kernel<8><<<(unsigned)blocks, 32 * warps, 0, st>>>((const uint2*)Y, w, inv_perm, (int)T, hv, topk,
                                                                (uint2*)out);
  else
    combine_kernel<4><<<(unsigned)blocks, 32 * warps, 0, st>>>((const uint32_t*)Y, w, inv_perm, (int)T, hv, topk,
                                                                (uint32_t*)out);
  return launched("combine");
}
