// Fused attention core O = softmax(scale * Q K^T + mask) V with grouped-query
// heads, on the sm_103a tensor cores (tcgen05, TMEM accumulators, TMA).
//
// One CTA owns one (batch, query head h, block of 128 queries); the KV head is
// g = h / (Hq / Hkv). Per key block j of BN keys:
//   warp 0     : TMA producer - Q once, then K_j (2 x [BN][64] swizzled
//                halves of the head dimension) and V_j into a ring of stages.
//   warp 1     : one thread issues S = Q K_j^T into TMEM columns [0, BN)
//                (8 UMMAs of K = 16 over the 128-wide head dimension), then,
//                once P_j is in shared memory, O += P_j V_j into TMEM columns
//                [BN, BN + 128).
//   warps 2..5 : softmax, one query row per thread (TMEM lane = row). Pass 1
//                reads S and takes the masked row maximum; the running maximum
//                m and sum l follow the online softmax in the log2 domain
//                (p = 2^(s * scale * log2 e - m)); O is rescaled in TMEM by
//                2^(m_old - m_new) when the maximum moved; pass 2 writes P as
//                bf16 in the 128-byte-swizzled K-major layout the UMMA reads.
// The epilogue divides O by l, stores bf16 O and LSE = ln 2 * (m + log2 l).
//
// Schedule knobs: BN (template), ring depth (runtime), query-block order
// (natural or longest-first for the causal triangle), and the layout of V:
// as given ([keys][d], an MN-major UMMA B operand) or pre-transposed by a pass
// into [d][keys] (K-major). Masking: key j is visible to query i when j < S and
// (not causal or j <= i). Every wait is bounded as in the GEMM kernels.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstring>

#include "rc_internal.h"
#include "tc_common.cuh"

namespace tcg {
rc_status encode_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows);
}

namespace attn {

constexpr int BM = 128;
constexpr int D = 128;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 256;

struct Params {
  int B, S, Hq, Hkv, group;
  int q_blocks;
  int causal;
  float scale_log2;  // softmax scale * log2(e)
  int raster;
  __nv_bfloat16* O;
  float* lse;
  int* status;
};

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Packed fp32 pairs: two floats in one 64-bit register, for the f32x2
// add / fma instructions of sm_100+ (one issue slot for two lanes' worth;
// the FMA pipe still takes two cycles per warp, so they save issue slots,
// which is what the softmax runs short of, not FMA throughput).
__device__ __forceinline__ uint64_t f2(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void f2_split(uint64_t v, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Maximum of N raw scores (N even, >= 8): four independent chains of
// three-input maxima, then a combine.
template <int N>
__device__ __forceinline__ float row_max(const uint32_t* r) {
  float pm[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) pm[u] = __uint_as_float(r[u]);
#pragma unroll
  for (int i = 4; i < N; i += 2)
    pm[(i / 2) % 4] = max3(pm[(i / 2) % 4], __uint_as_float(r[i]), __uint_as_float(r[i + 1]));
  return fmaxf(max3(pm[0], pm[1], pm[2]), pm[3]);
}

// p_i = 2^(s_i * scale_log2 - mref) for N raw scores: bf16 pairs into pk and
// fp32 partial sums into ls2 (two packed accumulators). Masked scores are
// -inf and give +0.
template <int N>
__device__ __forceinline__ void exp_pack(const uint32_t* r, uint64_t sc2, uint64_t nm2, uint32_t* pk,
                                         uint64_t (&ls2)[2]) {
#pragma unroll
  for (int i = 0; i < N; i += 2) {
    const uint64_t x = f2_fma(f2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])), sc2, nm2);
    float x0, x1;
    f2_split(x, x0, x1);
    const float p0 = tc::ex2_approx(x0), p1 = tc::ex2_approx(x1);
    ls2[(i / 2) % 2] = f2_add(ls2[(i / 2) % 2], f2(p0, p1));
    pk[i / 2] = pack2(p0, p1);
  }
}

__device__ __forceinline__ float sum_pairs(const uint64_t (&ls2)[2]) {
  float a, b, c, d;
  f2_split(ls2[0], a, b);
  f2_split(ls2[1], c, d);
  return (a + b) + (c + d);
}

// One normalised output row: O (fp32 in this thread's TMEM lane, columns
// tO .. tO + D - 1) times 1/l, rounded to bf16, stored as 16-byte vectors.
// Each 64-column half is fetched with two loads and a single wait.
__device__ __forceinline__ void store_o_row(uint32_t tO, float inv_l, __nv_bfloat16* orow, bool row_ok) {
#pragma unroll
  for (int c = 0; c < D; c += 64) {
    uint32_t o[64];
    tc::tmem_ld32(tO + c, *reinterpret_cast<uint32_t(*)[32]>(&o[0]));
    tc::tmem_ld32(tO + c + 32, *reinterpret_cast<uint32_t(*)[32]>(&o[32]));
    tc::tmem_ld_wait();
    if (row_ok) {
#pragma unroll
      for (int i = 0; i < 64; i += 8) {
        uint32_t pk[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          pk[u] = pack2(__uint_as_float(o[i + 2 * u]) * inv_l, __uint_as_float(o[i + 2 * u + 1]) * inv_l);
        *reinterpret_cast<uint4*>(orow + c + i) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
      }
    }
  }
}


template <int BN, bool VT>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const Params p, const int stages) {
  static_assert(BN == 64 || BN == 128, "key block");
  constexpr int Q_BYTES = BM * D * 2;   // two [128][64] halves
  constexpr int KV_TILE = BN * D * 2;   // one K or V tile
  constexpr int P_BYTES = BM * BN * 2;  // BN/64 atoms of [128][64]

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;
  uint8_t* ring = smem + Q_BYTES;
  uint8_t* sP = ring + (size_t)stages * 2 * KV_TILE;
  uint64_t* q_full = (uint64_t*)(sP + P_BYTES);
  uint64_t* kv_full = q_full + 1;
  uint64_t* kv_empty = kv_full + stages;
  uint64_t* s_full = kv_empty + stages;
  uint64_t* s_free = s_full + 1;
  uint64_t* p_full = s_free + 1;
  uint64_t* pv_full = p_full + 1;
  uint64_t* drain = pv_full + 1;
  uint32_t* tmem_slot = (uint32_t*)(drain + 1);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);
  volatile int* status = p.status;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int BH = p.B * p.Hq;
  int qb, bh;
  if (p.raster == 0) {
    qb = blockIdx.x % p.q_blocks;
    bh = blockIdx.x / p.q_blocks;
  } else {  // longest causal rows first
    qb = p.q_blocks - 1 - (int)(blockIdx.x / BH);
    bh = blockIdx.x % BH;
  }
  const int b = bh / p.Hq, h = bh - b * p.Hq, g = h / p.group;
  const int q0 = qb * BM;
  const int kv_end = p.causal ? min(q0 + BM, p.S) : p.S;
  const int nkb = (kv_end + BN - 1) / BN;

  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    tc::mbar_init(q_full, 1);
    for (int s = 0; s < stages; ++s) {
      tc::mbar_init(&kv_full[s], 1);
      tc::mbar_init(&kv_empty[s], 1);
    }
    tc::mbar_init(s_full, 1);
    tc::mbar_init(s_free, 128);
    tc::mbar_init(p_full, 128);
    tc::mbar_init(pv_full, 1);
    tc::mbar_init(drain, 1);
    *abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc(tmem_slot, kTmemCols);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmK);
      tc::prefetch_tmap(&tmV);
      tc::mbar_expect_tx(q_full, Q_BYTES);
      const int qrow = b * p.S + q0;
      tc::tma_load_2d(sQ, &tmQ, q_full, h * D, qrow);
      tc::tma_load_2d(sQ + Q_BYTES / 2, &tmQ, q_full, h * D + 64, qrow);
      int j = 0;
      for (; j < nkb; ++j) {
        const int s = j % stages;
        const uint32_t ph = (uint32_t)(j / stages) & 1u;
        if (!tc::mbar_wait(&kv_empty[s], ph ^ 1u, abort_flag, status)) {
          fail(RC_DEV_TIMEOUT_EMPTY);
          break;
        }
        uint8_t* sk = ring + (size_t)s * 2 * KV_TILE;
        uint8_t* sv = sk + KV_TILE;
        tc::mbar_expect_tx(&kv_full[s], 2 * KV_TILE);
        const int krow = b * p.S + j * BN;
        tc::tma_load_2d(sk, &tmK, &kv_full[s], g * D, krow);
        tc::tma_load_2d(sk + BN * 128, &tmK, &kv_full[s], g * D + 64, krow);
        if constexpr (VT) {
#pragma unroll
          for (int a = 0; a < BN / 64; ++a)
            tc::tma_load_2d(sv + a * (BM * 128), &tmV, &kv_full[s], j * BN + a * 64, (b * p.Hkv + g) * D);
        } else {
          tc::tma_load_2d(sv, &tmV, &kv_full[s], g * D, krow);
          tc::tma_load_2d(sv + BN * 128, &tmV, &kv_full[s], g * D + 64, krow);
        }
      }
      if (!tc::mbar_wait_drain(q_full, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      for (int i = max(0, j - stages); i < j; ++i)
        if (!tc::mbar_wait_drain(&kv_full[i % stages], (uint32_t)(i / stages) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = tc::idesc_bf16_f32(BM, BN);
      constexpr uint32_t idO = tc::idesc_bf16_f32(BM, D, !VT);
      const uint32_t tS = tmem, tO = tmem + BN;
      bool ok = tc::mbar_wait(q_full, 0, abort_flag, status);
      if (!ok) fail(RC_DEV_TIMEOUT_FULL);
      const uint32_t sq = tc::smem_u32(sQ);
      for (int j = 0; ok && j < nkb; ++j) {
        const int s = j % stages;
        const uint32_t ph = (uint32_t)(j / stages) & 1u;
        if (!tc::mbar_wait(&kv_full[s], ph, abort_flag, status) ||
            (j > 0 && !tc::mbar_wait(s_free, (uint32_t)(j - 1) & 1u, abort_flag, status))) {
          fail(RC_DEV_TIMEOUT_FULL);
          ok = false;
          break;
        }
        tc::tc_fence_after();
        const uint32_t sk = tc::smem_u32(ring + (size_t)s * 2 * KV_TILE);
        const uint32_t sv = sk + KV_TILE;
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          tc::umma_bf16(tS, tc::sw128_desc(sq + (ks / 4) * (BM * 128) + off),
                        tc::sw128_desc(sk + (ks / 4) * (BN * 128) + off), idS, ks > 0 ? 1u : 0u);
        }
        tc::umma_commit(s_full);
        if (!tc::mbar_wait(p_full, (uint32_t)j & 1u, abort_flag, status)) {
          fail(RC_DEV_TIMEOUT_FULL);
          ok = false;
          break;
        }
        tc::tc_fence_after();
        const uint32_t sp = tc::smem_u32(sP);
#pragma unroll
        for (int ks = 0; ks < BN / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          const uint64_t da = tc::sw128_desc(sp + (ks / 4) * (BM * 128) + off);
          uint64_t db;
          if constexpr (VT)
            db = tc::sw128_desc(sv + (ks / 4) * (BM * 128) + off);
          else
            db = tc::sw128_desc_mn(sv + (uint32_t)ks * 16 * 128, BN * 128, 1024);
          tc::umma_bf16(tO, da, db, idO, (j > 0 || ks > 0) ? 1u : 0u);
        }
        tc::umma_commit(pv_full);
        tc::umma_commit(&kv_empty[s]);
      }
      if (!ok) {
        tc::umma_commit(drain);
        if (!tc::mbar_wait_drain(drain, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else {
    const int q = warp & 3;
    const int row = 32 * q + lane;
    const int qi = q0 + row;
    const uint32_t lane_base = (uint32_t)(32 * q) << 16;
    const uint32_t tS = tmem + lane_base, tO = tmem + lane_base + BN;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      if (!tc::mbar_wait(s_full, (uint32_t)j & 1u, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        ok = false;
        break;
      }
      tc::tc_fence_after();
      const int k0 = j * BN;
      // pass 1: masked row maximum
      float mx = -INFINITY;
#pragma unroll 1
      for (int c = 0; c < BN; c += 16) {
        uint32_t r[16];
        tc::tmem_ld16(tS + c, r);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int key = k0 + c + i;
          const bool vis = key < p.S && (!p.causal || key <= qi);
          mx = fmaxf(mx, vis ? __uint_as_float(r[i]) : -INFINITY);
        }
      }
      const float m_new = fmaxf(m, mx * p.scale_log2);
      const float alpha = (m == -INFINITY) ? 0.f : exp2f(m - m_new);
      const float m_use = (m_new == -INFINITY) ? 0.f : m_new;
      if (j > 0) {
        // O holds P_{j-1} V_{j-1}; P's buffer is free again; rescale O
        if (!tc::mbar_wait(pv_full, (uint32_t)(j - 1) & 1u, abort_flag, status)) {
          if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
          ok = false;
          break;
        }
        tc::tc_fence_after();
        if (__any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll 1
          for (int c = 0; c < D; c += 16) {
            uint32_t r[16];
            tc::tmem_ld16(tO + c, r);
            tc::tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
            tc::tmem_st16(tO + c, r);
          }
          tc::tmem_st_wait();
        }
      }
      // pass 2: probabilities -> P (bf16, swizzled K-major rows), row sum
      float lsum = 0.f;
      uint8_t* rowp0 = sP + (row / 8) * 1024 + (row % 8) * 128;
#pragma unroll 1
      for (int c = 0; c < BN; c += 16) {
        uint32_t r[16];
        tc::tmem_ld16(tS + c, r);
        tc::tmem_ld_wait();
        uint32_t pk[8];
#pragma unroll
        for (int i = 0; i < 16; i += 2) {
          const int key = k0 + c + i;
          const bool v0 = key < p.S && (!p.causal || key <= qi);
          const bool v1 = key + 1 < p.S && (!p.causal || key + 1 <= qi);
          const float p0 = v0 ? exp2f(__uint_as_float(r[i]) * p.scale_log2 - m_use) : 0.f;
          const float p1 = v1 ? exp2f(__uint_as_float(r[i + 1]) * p.scale_log2 - m_use) : 0.f;
          lsum += p0 + p1;
          pk[i / 2] = pack2(p0, p1);
        }
        uint8_t* rowp = rowp0 + (c / 64) * (BM * 128);
        const int ch = (c % 64) / 8;
        *reinterpret_cast<uint4*>(rowp + ((ch ^ (row % 8)) * 16)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        *reinterpret_cast<uint4*>(rowp + (((ch + 1) ^ (row % 8)) * 16)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
      }
      l = l * alpha + lsum;
      m = m_new;
      tc::tc_fence_before();
      tc::fence_proxy_async_smem();
      tc::mbar_arrive(s_free);
      tc::mbar_arrive(p_full);
    }
    if (ok) {
      if (tc::mbar_wait(pv_full, (uint32_t)(nkb - 1) & 1u, abort_flag, status)) {
        tc::tc_fence_after();
        const float inv_l = l > 0.f ? 1.f / l : 0.f;
        __nv_bfloat16* orow = p.O + ((size_t)(b * p.S + qi) * p.Hq + h) * D;
        const bool row_ok = qi < p.S;
#pragma unroll 1
        for (int c = 0; c < D; c += 16) {
          uint32_t r[16];
          tc::tmem_ld16(tO + c, r);
          tc::tmem_ld_wait();
          uint32_t pk[8];
#pragma unroll
          for (int i = 0; i < 16; i += 2)
            pk[i / 2] = pack2(__uint_as_float(r[i]) * inv_l, __uint_as_float(r[i + 1]) * inv_l);
          if (row_ok) {
            *reinterpret_cast<uint4*>(orow + c) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            *reinterpret_cast<uint4*>(orow + c + 8) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
          }
        }
        if (p.lse && row_ok) p.lse[((size_t)b * p.Hq + h) * p.S + qi] = 0.6931471805599453f * (m + log2f(l));
      } else if (!*abort_flag) {
        fail(RC_DEV_TIMEOUT_ACCUM);
      }
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// Two query tiles per CTA (TileSize M = 256), ping-pong between two softmax
// warpgroups: the MMA warp issues S_0 = Q_0 K^T, S_1 = Q_1 K^T, then
// O_0 += P_0 V as soon as P_0 is ready and the next S_0 right after it, so
// one tile's softmax overlaps the other tile's tensor-core work. TMEM holds
// S_0, S_1 (BN columns each) and O_0, O_1 (128 each). Each softmax thread
// loads its whole S row with one wait. O is rescaled only when the running
// maximum grows by more than 2^8 (kRescaleLog2); the exponents use that same
// reference maximum, and so does the row sum l, so the result is exact.
// S for key block j+1 is issued before block j's ring slot is released, so
// this kernel needs a ring of at least two stages.
constexpr int kThreads2 = 320;
constexpr float kRescaleLog2 = 8.0f;


// Softmax and output of one query tile in the two-tile kernels: one TMEM lane
// quadrant per warp (qd = warp % 4), one query row per thread. S of key block j
// sits in TMEM columns [(t * NSB + j % NSB) * BN, + BN) and O_t at o_base + t * D.
// Pass 1 takes the masked row maximum of the whole S row (one TMEM round trip);
// O is rescaled in TMEM when the reference maximum moves by more than 2^8; pass 2
// writes P = 2^(s * scale * log2 e - m) as bf16, over its own S columns (PT) or
// into the swizzled shared-memory P tile, and accumulates the row sum l.
template <int BN, bool PT, bool SDB>
__device__ __forceinline__ void softmax_tile(const Params& p, int t, int qd, int lane, int q0, int nkb, int b, int h,
                                             uint32_t tmem, uint32_t o_base, uint8_t* sP_tile, uint64_t* s_full,
                                             uint64_t* p_full, uint64_t* pv_full, volatile int* abort_flag,
                                             volatile int* status) {
  constexpr int NSB = SDB ? 2 : 1;
  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };
  const int row = 32 * qd + lane;
  const int qi = q0 + row;
  const uint32_t lane_base = (uint32_t)(32 * qd) << 16;
  const uint32_t tO = tmem + lane_base + o_base + t * D;
  uint8_t* rowp0 = sP_tile + (row / 8) * 1024 + (row % 8) * 128;
  float m_ref = -INFINITY, l = 0.f;
  bool ok = true;
  for (int j = 0; j < nkb; ++j) {
    const uint32_t tS = tmem + lane_base + (uint32_t)(t * NSB + (j % NSB)) * BN;
    if (!tc::mbar_wait(&s_full[j % NSB], (uint32_t)(j / NSB) & 1u, abort_flag, status)) {
      if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
      ok = false;
      break;
    }
    tc::tc_fence_after();
    const int k0 = j * BN;
    // keys [k0, k0 + nvis) of this block are visible to query qi
    int nvis = min(BN, p.S - k0);
    if (p.causal) nvis = min(nvis, max(0, qi - k0 + 1));
    // the whole S row in registers: one TMEM round trip
    uint32_t r[BN];
#pragma unroll
    for (int q = 0; q < BN; q += 16) tc::tmem_ld16(tS + q, *reinterpret_cast<uint32_t(*)[16]>(&r[q]));
    tc::tmem_ld_wait();
    if (nvis < BN) {
#pragma unroll
      for (int i = 0; i < BN; ++i)
        if (i >= nvis) r[i] = __float_as_uint(-INFINITY);
    }
    const float mxs = row_max<BN>(r) * p.scale_log2;
    float factor = 1.f;
    if (m_ref == -INFINITY) {
      m_ref = mxs;  // first visible scores: O and l are still zero
    } else if (mxs > m_ref + kRescaleLog2) {
      factor = exp2f(m_ref - mxs);
      m_ref = mxs;
    }
    const bool rescale = __any_sync(0xffffffffu, factor != 1.f);
    // pv_full completes once per key block (P_t V of that block). It is
    // observed phase by phase, so a parity wait never meets a barrier more
    // than one phase ahead: phase j-1 is awaited in iteration j, before the
    // O rescale when there is one (O must hold P_t V of block j-1), before
    // overwriting P's shared-memory buffer, or else after the probabilities
    // are written. P V of block j is only issued after this thread's p_full.
    bool pv_seen = j == 0;
    auto await_pv = [&]() -> bool {
      if (pv_seen) return true;
      pv_seen = true;
      if (!tc::mbar_wait(pv_full, (uint32_t)(j - 1) & 1u, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        return false;
      }
      tc::tc_fence_after();
      return true;
    };
    if (rescale || !PT) {
      if (!await_pv()) {
        ok = false;
        break;
      }
    }
    if (rescale) {
#pragma unroll 1
      for (int c = 0; c < D; c += 16) {
        uint32_t r[16];
        tc::tmem_ld16(tO + c, r);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * factor);
        tc::tmem_st16(tO + c, r);
      }
      tc::tmem_st_wait();
    }
    // pass 2: probabilities -> P (bf16) and the row sum
    const float mref = m_ref == -INFINITY ? 0.f : m_ref;
    const uint64_t sc2 = f2(p.scale_log2, p.scale_log2), nm2 = f2(-mref, -mref);
    uint64_t ls2[2] = {0ull, 0ull};
#pragma unroll
    for (int c = 0; c < BN; c += 32) {
      uint32_t pk[16];
      exp_pack<32>(r + c, sc2, nm2, pk, ls2);
      if constexpr (PT) {
        // P for keys [c, c + 32) goes to columns [c/2, c/2 + 16) of the S row (already in registers)
        tc::tmem_st16(tS + c / 2, pk);
      } else {
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          const int cc = c + 16 * h2;
          uint8_t* rowp = rowp0 + (cc / 64) * (BM * 128);
          const int ch = (cc % 64) / 8;
          *reinterpret_cast<uint4*>(rowp + ((ch ^ (row % 8)) * 16)) =
              make_uint4(pk[8 * h2], pk[8 * h2 + 1], pk[8 * h2 + 2], pk[8 * h2 + 3]);
          *reinterpret_cast<uint4*>(rowp + (((ch + 1) ^ (row % 8)) * 16)) =
              make_uint4(pk[8 * h2 + 4], pk[8 * h2 + 5], pk[8 * h2 + 6], pk[8 * h2 + 7]);
        }
      }
    }
    l = l * factor + sum_pairs(ls2);
    if constexpr (PT) tc::tmem_st_wait();
    if (!await_pv()) {
      ok = false;
      break;
    }
    tc::tc_fence_before();
    if constexpr (!PT) tc::fence_proxy_async_smem();
    tc::mbar_arrive(p_full);
  }
  if (ok && nkb > 0) {
    if (tc::mbar_wait(pv_full, (uint32_t)(nkb - 1) & 1u, abort_flag, status)) {
      tc::tc_fence_after();
      const float inv_l = l > 0.f ? 1.f / l : 0.f;
      const bool row_ok = qi < p.S;
      __nv_bfloat16* orow = p.O + ((size_t)(b * p.S + (row_ok ? qi : 0)) * p.Hq + h) * D;
      store_o_row(tO, inv_l, orow, row_ok);
      if (p.lse && row_ok) p.lse[((size_t)b * p.Hq + h) * p.S + qi] = 0.6931471805599453f * (m_ref + log2f(l));
    } else if (!*abort_flag) {
      fail(RC_DEV_TIMEOUT_ACCUM);
    }
  }
}

template <int BN, bool VT, bool PT, bool SDB>
__global__ void __launch_bounds__(kThreads2, 1)
    attn2_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                 const __grid_constant__ CUtensorMap tmV, const Params p, const int stages) {
  static_assert(BN == 64 || BN == 128, "key block");
  constexpr int Q_BYTES = BM * D * 2;   // one query tile: two [128][64] halves
  constexpr int KV_TILE = BN * D * 2;
  // P tiles live in shared memory (BN/64 atoms of [128][64]) or, when PT, in
  // the first BN/2 TMEM columns of their S tile (two bf16 per column).
  constexpr int P_BYTES = PT ? 0 : BM * BN * 2;
  // SDB: two S buffers per query tile, so S for key block j+1 is computed
  // while the softmax works on block j (two key blocks in flight per tile).
  static_assert(!SDB || (PT && BN == 64), "double-buffered S needs P in TMEM and BN = 64");
  // (SDB also needs >= 4 ring stages: S of block j+2 is issued while V of
  // block j is still in use, and the next block should already be loading.)
  constexpr int NSB = SDB ? 2 : 1;                     // S buffers per tile
  constexpr uint32_t O_BASE = (uint32_t)(2 * NSB * BN);  // TMEM column of O_0

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;                                   // [2] tiles
  uint8_t* ring = smem + 2 * Q_BYTES;
  uint8_t* sP = ring + (size_t)stages * 2 * KV_TILE;    // [2] tiles
  // separate K and V rings of `stages` slots each: K of a block is released
  // once both tiles' S products are issued, V once both P V products are
  uint64_t* q_full = (uint64_t*)(sP + 2 * P_BYTES);
  uint64_t* k_full = q_full + 1;
  uint64_t* k_empty = k_full + stages;
  uint64_t* v_full = k_empty + stages;
  uint64_t* v_empty = v_full + stages;
  uint64_t* s_full = v_empty + stages;  // [2 tiles][NSB buffers]
  uint64_t* p_full = s_full + 2 * NSB;   // [2]
  uint64_t* pv_full = p_full + 2;        // [2]
  uint64_t* drain = pv_full + 2;
  uint32_t* tmem_slot = (uint32_t*)(drain + 1);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);
  volatile int* status = p.status;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int pairs = (p.q_blocks + 1) / 2;
  const int BH = p.B * p.Hq;
  int pb, bh;
  if (p.raster == 0) {
    pb = blockIdx.x % pairs;
    bh = blockIdx.x / pairs;
  } else {
    pb = pairs - 1 - (int)(blockIdx.x / BH);
    bh = blockIdx.x % BH;
  }
  const int b = bh / p.Hq, h = bh - b * p.Hq, g = h / p.group;
  int q0[2], nkb[2];
#pragma unroll
  for (int t = 0; t < 2; ++t) {
    q0[t] = (2 * pb + t) * BM;
    const int end = p.causal ? min(q0[t] + BM, p.S) : p.S;
    nkb[t] = q0[t] < p.S ? (end + BN - 1) / BN : 0;
  }
  const int nblk = max(nkb[0], nkb[1]);

  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    tc::mbar_init(q_full, 1);
    for (int s = 0; s < stages; ++s) {
      tc::mbar_init(&k_full[s], 1);
      tc::mbar_init(&k_empty[s], 1);
      tc::mbar_init(&v_full[s], 1);
      tc::mbar_init(&v_empty[s], 1);
    }
    for (int t = 0; t < 2; ++t) {
      for (int b2 = 0; b2 < NSB; ++b2) tc::mbar_init(&s_full[t * NSB + b2], 1);
      tc::mbar_init(&p_full[t], 128);
      tc::mbar_init(&pv_full[t], 1);
    }
    tc::mbar_init(drain, 1);
    *abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc(tmem_slot, 512);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmK);
      tc::prefetch_tmap(&tmV);
      tc::mbar_expect_tx(q_full, 2 * Q_BYTES);
#pragma unroll
      for (int t = 0; t < 2; ++t) {
        const int qrow = b * p.S + q0[t];
        tc::tma_load_2d(sQ + t * Q_BYTES, &tmQ, q_full, h * D, qrow);
        tc::tma_load_2d(sQ + t * Q_BYTES + Q_BYTES / 2, &tmQ, q_full, h * D + 64, qrow);
      }
      int j = 0;
      for (; j < nblk; ++j) {
        const int s = j % stages;
        const uint32_t ph = (uint32_t)(j / stages) & 1u;
        uint8_t* sk = ring + (size_t)s * 2 * KV_TILE;
        uint8_t* sv = sk + KV_TILE;
        const int krow = b * p.S + j * BN;
        if (!tc::mbar_wait(&k_empty[s], ph ^ 1u, abort_flag, status)) {
          fail(RC_DEV_TIMEOUT_EMPTY);
          break;
        }
        tc::mbar_expect_tx(&k_full[s], KV_TILE);
        tc::tma_load_2d(sk, &tmK, &k_full[s], g * D, krow);
        tc::tma_load_2d(sk + BN * 128, &tmK, &k_full[s], g * D + 64, krow);
        if (!tc::mbar_wait(&v_empty[s], ph ^ 1u, abort_flag, status)) {
          fail(RC_DEV_TIMEOUT_EMPTY);
          // K of this block is in flight: let it land before exit
          if (!tc::mbar_wait_drain(&k_full[s], ph)) fail(RC_DEV_TIMEOUT_DRAIN);
          break;
        }
        tc::mbar_expect_tx(&v_full[s], KV_TILE);
        if constexpr (VT) {
#pragma unroll
          for (int a = 0; a < BN / 64; ++a)
            tc::tma_load_2d(sv + a * (BM * 128), &tmV, &v_full[s], j * BN + a * 64, (b * p.Hkv + g) * D);
        } else {
          tc::tma_load_2d(sv, &tmV, &v_full[s], g * D, krow);
          tc::tma_load_2d(sv + BN * 128, &tmV, &v_full[s], g * D + 64, krow);
        }
      }
      if (!tc::mbar_wait_drain(q_full, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      for (int i = max(0, j - stages); i < j; ++i) {
        if (!tc::mbar_wait_drain(&k_full[i % stages], (uint32_t)(i / stages) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
        if (!tc::mbar_wait_drain(&v_full[i % stages], (uint32_t)(i / stages) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = tc::idesc_bf16_f32(BM, BN);
      constexpr uint32_t idO = tc::idesc_bf16_f32(BM, D, !VT);
      bool ok = tc::mbar_wait(q_full, 0, abort_flag, status);
      if (!ok) fail(RC_DEV_TIMEOUT_FULL);
      int k_seen = -1, v_seen = -1;  // highest key block whose K / V arrival was awaited
      auto await_k = [&](int j) -> bool {
        if (j <= k_seen) return true;
        if (!tc::mbar_wait(&k_full[j % stages], (uint32_t)(j / stages) & 1u, abort_flag, status)) return false;
        k_seen = j;
        tc::tc_fence_after();
        return true;
      };
      auto await_v = [&](int j) -> bool {
        if (j <= v_seen) return true;
        if (!tc::mbar_wait(&v_full[j % stages], (uint32_t)(j / stages) & 1u, abort_flag, status)) return false;
        v_seen = j;
        tc::tc_fence_after();
        return true;
      };
      auto issue_s = [&](int t, int j) {
        const uint32_t sq = tc::smem_u32(sQ + t * Q_BYTES);
        const uint32_t sk = tc::smem_u32(ring + (size_t)(j % stages) * 2 * KV_TILE);
        const int sb = t * NSB + (j % NSB);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          tc::umma_bf16(tmem + (uint32_t)sb * BN, tc::sw128_desc(sq + (ks / 4) * (BM * 128) + off),
                        tc::sw128_desc(sk + (ks / 4) * (BN * 128) + off), idS, ks > 0 ? 1u : 0u);
        }
        tc::umma_commit(&s_full[sb]);
      };
      auto issue_pv = [&](int t, int j) {
        const uint32_t sp = tc::smem_u32(sP + t * P_BYTES);
        const uint32_t sv = tc::smem_u32(ring + (size_t)(j % stages) * 2 * KV_TILE) + KV_TILE;
        const uint32_t tO = tmem + O_BASE + t * D;
        const uint32_t tP = tmem + (uint32_t)(t * NSB + (j % NSB)) * BN;  // P aliases its S buffer
#pragma unroll
        for (int ks = 0; ks < BN / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          uint64_t db;
          if constexpr (VT)
            db = tc::sw128_desc(sv + (ks / 4) * (BM * 128) + off);
          else
            db = tc::sw128_desc_mn(sv + (uint32_t)ks * 16 * 128, BN * 128, 1024);
          if constexpr (PT)
            tc::umma_bf16_ts(tO, tP + (uint32_t)ks * 8, db, idO, (j > 0 || ks > 0) ? 1u : 0u);
          else
            tc::umma_bf16(tO, tc::sw128_desc(sp + (ks / 4) * (BM * 128) + off), db, idO,
                          (j > 0 || ks > 0) ? 1u : 0u);
        }
        tc::umma_commit(&pv_full[t]);
      };
      // prologue: S for the first NSB key blocks of both tiles; their K is then free
      for (int j0 = 0; ok && j0 < NSB && j0 < nblk; ++j0) {
        ok = await_k(j0);
        if (ok) {
          for (int t = 0; t < 2; ++t)
            if (j0 < nkb[t]) issue_s(t, j0);
          tc::umma_commit(&k_empty[j0 % stages]);
        }
      }
      for (int j = 0; ok && j < nblk; ++j) {
        for (int t = 0; t < 2; ++t) {
          if (j >= nkb[t]) continue;
          if (!tc::mbar_wait(&p_full[t], (uint32_t)j & 1u, abort_flag, status) || !await_v(j)) {
            ok = false;
            break;
          }
          tc::tc_fence_after();
          issue_pv(t, j);
          if (j + NSB < nkb[t]) {
            if (!await_k(j + NSB)) {
              ok = false;
              break;
            }
            issue_s(t, j + NSB);
          }
        }
        if (!ok) break;
        tc::umma_commit(&v_empty[j % stages]);  // both P V products of block j issued
        if (j + NSB < nblk) tc::umma_commit(&k_empty[(j + NSB) % stages]);  // both S products of block j+NSB
      }
      if (!ok) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(drain);
        if (!tc::mbar_wait_drain(drain, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else if (warp >= 2) {
    const int t = (warp - 2) / 4;  // query tile of this warpgroup
    softmax_tile<BN, PT, SDB>(p, t, warp & 3, lane, q0[t], nkb[t], b, h, tmem, O_BASE, sP + t * P_BYTES,
                              &s_full[t * NSB], &p_full[t], &pv_full[t], abort_flag, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, 512);
  }
}

// Compact softmax of one query tile for P in TMEM (one S buffer per tile): the
// S row is walked twice in chunks of 32 columns by loops that are not
// unrolled, first for the masked maximum (masked scores are written back as
// -inf, only in chunks that hold any), then for P and the row sum. It holds 32
// scores in registers instead of the whole row (68 registers per thread
// instead of 168) and measures as fast as the whole-row version in the
// two-issuer kernel, where the tensor pipe, not the softmax, sets the pace.
// P of keys [c, c + 32) goes to columns [c/2, c/2 + 16), which hold S values
// already consumed.
template <int BN>
__device__ __forceinline__ void softmax_tile_chunked(const Params& p, int t, int qd, int lane, int q0, int nkb, int b,
                                                     int h, uint32_t tmem, uint32_t o_base, uint64_t* s_full,
                                                     uint64_t* p_full, uint64_t* pv_full, volatile int* abort_flag,
                                                     volatile int* status) {
  constexpr int CH = 32;
  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };
  const int row = 32 * qd + lane;
  const int qi = q0 + row;
  const uint32_t lane_base = (uint32_t)(32 * qd) << 16;
  const uint32_t tO = tmem + lane_base + o_base + t * D;
  const uint32_t tS = tmem + lane_base + (uint32_t)(t * BN);
  float m_ref = -INFINITY, l = 0.f;
  bool ok = true;
  for (int j = 0; j < nkb; ++j) {
    if (!tc::mbar_wait(s_full, (uint32_t)j & 1u, abort_flag, status)) {
      if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
      ok = false;
      break;
    }
    tc::tc_fence_after();
    const int k0 = j * BN;
    // keys [k0, k0 + nvis) of this block are visible to query qi
    int nvis = min(BN, p.S - k0);
    if (p.causal) nvis = min(nvis, max(0, qi - k0 + 1));
    float mx = -INFINITY;
#pragma unroll 1
    for (int c = 0; c < BN; c += CH) {
      uint32_t r[CH];
      tc::tmem_ld32(tS + c, r);
      tc::tmem_ld_wait();
      if (__any_sync(0xffffffffu, nvis < c + CH)) {
#pragma unroll
        for (int i = 0; i < CH; ++i)
          if (c + i >= nvis) r[i] = __float_as_uint(-INFINITY);
        tc::tmem_st32(tS + c, r);
        tc::tmem_st_wait();
      }
      mx = fmaxf(mx, row_max<CH>(r));
    }
    const float mxs = mx * p.scale_log2;
    float factor = 1.f;
    if (m_ref == -INFINITY) {
      m_ref = mxs;  // first visible scores: O and l are still zero
    } else if (mxs > m_ref + kRescaleLog2) {
      factor = exp2f(m_ref - mxs);
      m_ref = mxs;
    }
    const bool rescale = __any_sync(0xffffffffu, factor != 1.f);
    // pv_full phase j-1 (P_t V of block j-1) is observed once per key block:
    // before the O rescale when there is one, else after P is written
    bool pv_seen = j == 0;
    auto await_pv = [&]() -> bool {
      if (pv_seen) return true;
      pv_seen = true;
      if (!tc::mbar_wait(pv_full, (uint32_t)(j - 1) & 1u, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        return false;
      }
      tc::tc_fence_after();
      return true;
    };
    if (rescale) {
      if (!await_pv()) {
        ok = false;
        break;
      }
#pragma unroll 1
      for (int c = 0; c < D; c += CH) {
        uint32_t r[CH];
        tc::tmem_ld32(tO + c, r);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < CH; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * factor);
        tc::tmem_st32(tO + c, r);
      }
      tc::tmem_st_wait();
    }
    const float mref = m_ref == -INFINITY ? 0.f : m_ref;
    const uint64_t sc2 = f2(p.scale_log2, p.scale_log2), nm2 = f2(-mref, -mref);
    uint64_t ls2[2] = {0ull, 0ull};
#pragma unroll 1
    for (int c = 0; c < BN; c += CH) {
      uint32_t r[CH];
      tc::tmem_ld32(tS + c, r);
      tc::tmem_ld_wait();
      uint32_t pk[CH / 2];
      exp_pack<CH>(r, sc2, nm2, pk, ls2);
      tc::tmem_st16(tS + c / 2, pk);
    }
    l = l * factor + sum_pairs(ls2);
    tc::tmem_st_wait();
    if (!await_pv()) {
      ok = false;
      break;
    }
    tc::tc_fence_before();
    tc::mbar_arrive(p_full);
  }
  if (ok && nkb > 0) {
    if (tc::mbar_wait(pv_full, (uint32_t)(nkb - 1) & 1u, abort_flag, status)) {
      tc::tc_fence_after();
      const float inv_l = l > 0.f ? 1.f / l : 0.f;
      const bool row_ok = qi < p.S;
      __nv_bfloat16* orow = p.O + ((size_t)(b * p.S + (row_ok ? qi : 0)) * p.Hq + h) * D;
      store_o_row(tO, inv_l, orow, row_ok);
      if (p.lse && row_ok) p.lse[((size_t)b * p.Hq + h) * p.S + qi] = 0.6931471805599453f * (m_ref + log2f(l));
    } else if (!*abort_flag) {
      fail(RC_DEV_TIMEOUT_ACCUM);
    }
  }
}

// Two query tiles per CTA with one UMMA-issuing warp per tile (Parallel = 1).
// One thread needs about as long to issue a 128 x 128 x 16 UMMA as the tensor
// pipe needs to execute it, and its barrier waits and commits come on top, so
// when a single thread issues both tiles' chains the pipe idles while that
// thread waits. Here each tile has its own issuer, which checks that V_j and
// K_{j+1} have landed while the softmax still works on S_j, and releases K_j
// once S_j is done and V_j once P_j V_j is done, through its own barriers; the
// producer refills a slot when every tile that read the block held there has
// released it (under the causal mask tile 0 stops before tile 1).
// The issuers take turns per chain (tile 0's chain c, then tile 1's chain c,
// then tile 0's chain c + 1), the UMMA order of the single-issuer kernel:
// this keeps the tiles half a period apart, so that one tile's softmax runs
// while the tensor pipe works on the other tile's products.
//   warp 0       : TMA producer (Q tiles once, then K_j and V_j)
//   warps 1, 2   : UMMA issue for query tile 0 / 1 (warp 1 also owns TMEM)
//   warps 3..6   : softmax of tile 0 (TMEM lane quadrant = warp % 4)
//   warps 7..10  : softmax of tile 1
// P is kept in TMEM over its S columns.
constexpr int kThreads3 = 352;

template <int BN, bool VT>
__global__ void __launch_bounds__(kThreads3, 1)
    attn3_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                 const __grid_constant__ CUtensorMap tmV, const Params p, const int stages) {
  static_assert(BN == 64 || BN == 128, "key block");
  constexpr int Q_BYTES = BM * D * 2;
  constexpr int KV_TILE = BN * D * 2;
  constexpr uint32_t O_BASE = (uint32_t)(2 * BN);  // TMEM: S_0, S_1, then O_0, O_1

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;  // [2] tiles
  uint8_t* ring = smem + 2 * Q_BYTES;
  uint64_t* q_full = (uint64_t*)(ring + (size_t)stages * 2 * KV_TILE);
  uint64_t* k_full = q_full + 1;              // [stages]
  uint64_t* v_full = k_full + stages;         // [stages]
  uint64_t* k_empty = v_full + stages;        // [2 tiles][stages]
  uint64_t* v_empty = k_empty + 2 * stages;   // [2 tiles][stages]
  uint64_t* s_full = v_empty + 2 * stages;    // [2]
  uint64_t* p_full = s_full + 2;              // [2]
  uint64_t* pv_full = p_full + 2;             // [2]
  uint64_t* drain = pv_full + 2;              // [2]
  uint32_t* tmem_slot = (uint32_t*)(drain + 2);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);
  volatile int* chains = (volatile int*)(tmem_slot + 2);  // [2] UMMA chains issued per tile
  volatile int* status = p.status;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int pairs = (p.q_blocks + 1) / 2;
  const int BH = p.B * p.Hq;
  int pb, bh;
  if (p.raster == 0) {
    pb = blockIdx.x % pairs;
    bh = blockIdx.x / pairs;
  } else {
    pb = pairs - 1 - (int)(blockIdx.x / BH);
    bh = blockIdx.x % BH;
  }
  const int b = bh / p.Hq, h = bh - b * p.Hq, g = h / p.group;
  int q0[2], nkb[2];
#pragma unroll
  for (int t = 0; t < 2; ++t) {
    q0[t] = (2 * pb + t) * BM;
    const int end = p.causal ? min(q0[t] + BM, p.S) : p.S;
    nkb[t] = q0[t] < p.S ? (end + BN - 1) / BN : 0;
  }
  const int nblk = max(nkb[0], nkb[1]);

  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    tc::mbar_init(q_full, 1);
    for (int s = 0; s < stages; ++s) {
      tc::mbar_init(&k_full[s], 1);
      tc::mbar_init(&v_full[s], 1);
    }
    for (int i = 0; i < 2 * stages; ++i) {
      tc::mbar_init(&k_empty[i], 1);
      tc::mbar_init(&v_empty[i], 1);
    }
    for (int t = 0; t < 2; ++t) {
      tc::mbar_init(&s_full[t], 1);
      tc::mbar_init(&p_full[t], 128);
      tc::mbar_init(&pv_full[t], 1);
      tc::mbar_init(&drain[t], 1);
    }
    *abort_flag = 0;
    chains[0] = chains[1] = 0;
    tc::fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc(tmem_slot, 512);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmK);
      tc::prefetch_tmap(&tmV);
      tc::mbar_expect_tx(q_full, 2 * Q_BYTES);
#pragma unroll
      for (int t = 0; t < 2; ++t) {
        const int qrow = b * p.S + q0[t];
        tc::tma_load_2d(sQ + t * Q_BYTES, &tmQ, q_full, h * D, qrow);
        tc::tma_load_2d(sQ + t * Q_BYTES + Q_BYTES / 2, &tmQ, q_full, h * D + 64, qrow);
      }
      // Slot s last held key block j - stages. Tile t read that block iff
      // j - stages < nkb[t]; its release is then the ((j - stages) / stages)-th
      // phase of its barrier for slot s, of parity ph ^ 1 (for j < stages the
      // fresh barrier passes that parity at once).
      auto released = [&](uint64_t* empty, int j, int s, uint32_t ph) -> bool {
        for (int t = 0; t < 2; ++t)
          if (j - stages < nkb[t] && !tc::mbar_wait(&empty[t * stages + s], ph ^ 1u, abort_flag, status))
            return false;
        return true;
      };
      int j = 0;
      for (; j < nblk; ++j) {
        const int s = j % stages;
        const uint32_t ph = (uint32_t)(j / stages) & 1u;
        uint8_t* sk = ring + (size_t)s * 2 * KV_TILE;
        uint8_t* sv = sk + KV_TILE;
        const int krow = b * p.S + j * BN;
        if (!released(k_empty, j, s, ph)) {
          fail(RC_DEV_TIMEOUT_EMPTY);
          break;
        }
        tc::mbar_expect_tx(&k_full[s], KV_TILE);
        tc::tma_load_2d(sk, &tmK, &k_full[s], g * D, krow);
        tc::tma_load_2d(sk + BN * 128, &tmK, &k_full[s], g * D + 64, krow);
        if (!released(v_empty, j, s, ph)) {
          fail(RC_DEV_TIMEOUT_EMPTY);
          if (!tc::mbar_wait_drain(&k_full[s], ph)) fail(RC_DEV_TIMEOUT_DRAIN);  // K of block j is in flight
          break;
        }
        tc::mbar_expect_tx(&v_full[s], KV_TILE);
        if constexpr (VT) {
#pragma unroll
          for (int a = 0; a < BN / 64; ++a)
            tc::tma_load_2d(sv + a * (BM * 128), &tmV, &v_full[s], j * BN + a * 64, (b * p.Hkv + g) * D);
        } else {
          tc::tma_load_2d(sv, &tmV, &v_full[s], g * D, krow);
          tc::tma_load_2d(sv + BN * 128, &tmV, &v_full[s], g * D + 64, krow);
        }
      }
      if (!tc::mbar_wait_drain(q_full, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      for (int i = max(0, j - stages); i < j; ++i) {
        if (!tc::mbar_wait_drain(&k_full[i % stages], (uint32_t)(i / stages) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
        if (!tc::mbar_wait_drain(&v_full[i % stages], (uint32_t)(i / stages) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp <= 2) {
    const int t = warp - 1;
    if (lane == 0 && nkb[t] > 0) {
      constexpr uint32_t idS = tc::idesc_bf16_f32(BM, BN);
      constexpr uint32_t idO = tc::idesc_bf16_f32(BM, D, !VT);
      const int nk = nkb[t];
      const int other_chains = nkb[1 - t] > 0 ? nkb[1 - t] + 1 : 0;
      const uint32_t sq = tc::smem_u32(sQ + t * Q_BYTES);
      const uint32_t tS = tmem + (uint32_t)(t * BN);
      const uint32_t tO = tmem + O_BASE + (uint32_t)(t * D);
      // this thread awaits every key block's K and V exactly once, in order;
      // a slot's next fill needs this tile's release of the current one
      auto await_full = [&](uint64_t* full, int j) -> bool {
        return tc::mbar_wait(&full[j % stages], (uint32_t)(j / stages) & 1u, abort_flag, status);
      };
      // chain c of this tile (c = 0: S_0; c = j + 1: P_j V_j and S_{j+1}) follows
      // chain c - 1 (tile 0) or chain c (tile 1) of the other tile
      auto await_turn = [&](int c) -> bool {
        const int need = min(t == 0 ? c : c + 1, other_chains);
        const uint64_t t0 = tc::globaltimer();
        for (uint32_t it = 1; chains[1 - t] < need; ++it)
          if ((it & 63) == 0 && (*abort_flag || tc::globaltimer() - t0 > tc::kWaitNs)) return false;
        return true;
      };
      auto issue_s = [&](int j) {
        const uint32_t sk = tc::smem_u32(ring + (size_t)(j % stages) * 2 * KV_TILE);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          tc::umma_bf16(tS, tc::sw128_desc(sq + (ks / 4) * (BM * 128) + off),
                        tc::sw128_desc(sk + (ks / 4) * (BN * 128) + off), idS, ks > 0 ? 1u : 0u);
        }
        tc::umma_commit(&s_full[t]);
        tc::umma_commit(&k_empty[t * stages + j % stages]);
      };
      auto issue_pv = [&](int j) {
        const int s = j % stages;
        const uint32_t sv = tc::smem_u32(ring + (size_t)s * 2 * KV_TILE) + KV_TILE;
#pragma unroll
        for (int ks = 0; ks < BN / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          uint64_t db;
          if constexpr (VT)
            db = tc::sw128_desc(sv + (ks / 4) * (BM * 128) + off);
          else
            db = tc::sw128_desc_mn(sv + (uint32_t)ks * 16 * 128, BN * 128, 1024);
          // P aliases S: two bf16 per TMEM column
          tc::umma_bf16_ts(tO, tS + (uint32_t)ks * 8, db, idO, (j > 0 || ks > 0) ? 1u : 0u);
        }
        tc::umma_commit(&pv_full[t]);
        tc::umma_commit(&v_empty[t * stages + s]);
      };
      bool ok = tc::mbar_wait(q_full, 0, abort_flag, status) && await_full(k_full, 0) && await_turn(0);
      if (ok) {
        tc::tc_fence_after();
        issue_s(0);
        chains[t] = 1;
      }
      for (int j = 0; ok && j < nk; ++j) {
        // V_j and K_{j+1} (landed long ago, normally) while the softmax works on S_j
        ok = await_full(v_full, j) && (j + 1 >= nk || await_full(k_full, j + 1)) &&
             tc::mbar_wait(&p_full[t], (uint32_t)j & 1u, abort_flag, status) && await_turn(j + 1);
        if (!ok) break;
        tc::tc_fence_after();
        issue_pv(j);  // O += P_j V_j
        if (j + 1 < nk) issue_s(j + 1);
        chains[t] = j + 2;
      }
      if (!ok) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[t]);
        if (!tc::mbar_wait_drain(&drain[t], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else {
    const int t = (warp - 3) / 4;
    softmax_tile_chunked<BN>(p, t, warp & 3, lane, q0[t], nkb[t], b, h, tmem, O_BASE, &s_full[t], &p_full[t],
                             &pv_full[t], abort_flag, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, 512);
  }
}

// One query tile per CTA with two S buffers and a P buffer of its own in TMEM
// (TileSize M = 128, Parallel = 1). TMEM: S_0, S_1 (BN columns each), O (128),
// P (BN/2 columns, two bf16 per column). S for key block j + 2 goes into the
// buffer of block j as soon as the softmax holds S_j in registers, so the
// tensor pipe computes S two key blocks ahead and the softmax of consecutive
// blocks runs back to back; the softmax keeps P_j in registers until
// P_{j-1} V_{j-1} has read the P buffer. The UMMAs come from two warps, one
// for the S products and one for the P V products (one thread needs about as
// long to issue a 128 x 128 x 16 UMMA as the pipe needs to run it), and K and
// V stream through rings of their own, each filled by its own producer warp.
//   warp 0     : TMA producer of Q and of the K ring
//   warp 1     : issues S_j = Q K_j^T (and owns TMEM)
//   warp 2     : issues O += P_j V_j
//   warp 3     : TMA producer of the V ring
//   warps 4..7 : softmax (TMEM lane quadrant = warp % 4), one query row per thread
constexpr int kThreads4 = 256;

template <int BN, int NSB>
// NSB S buffers at TMEM columns s_col + b * BN (block j in buffer j % NSB),
// O at o_col, P at p_col. g0: key blocks this CTA's softmax processed in
// earlier work items (persistent kernels; the barriers' phases run on across
// items). o_free (persistent kernels): arrived on once O has been read out.
__device__ __forceinline__ void softmax_sdb(const Params& p, int qd, int lane, int q0, int nkb, int b, int h,
                                            uint32_t tmem, uint32_t s_col, uint32_t o_col, uint32_t p_col,
                                            uint64_t* s_full, uint64_t* s_free, uint64_t* p_full, uint64_t* pv_full,
                                            volatile int* abort_flag, volatile int* status, int g0 = 0,
                                            uint64_t* o_free = nullptr) {
  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };
  const int row = 32 * qd + lane;
  const int qi = q0 + row;
  const uint32_t lane_base = (uint32_t)(32 * qd) << 16;
  const uint32_t tO = tmem + lane_base + o_col;
  const uint32_t tP = tmem + lane_base + p_col;
  float m_ref = -INFINITY, l = 0.f;
  // pv_full completes once per key block (P_j V_j done); its phases are
  // observed one by one, in order, never more than one behind: phase j - 1
  // in iteration j (before an O rescale, else before P_j overwrites P_{j-1}),
  // the last one before the output. Indices are global (g0 + j).
  int pv_seen = g0;
  auto await_pv = [&](int upto) -> bool {
    if (pv_seen > upto) return true;
    for (; pv_seen <= upto; ++pv_seen)
      if (!tc::mbar_wait(pv_full, (uint32_t)pv_seen & 1u, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        return false;
      }
    tc::tc_fence_after();
    return true;
  };
  bool ok = true;
  for (int j = 0; j < nkb; ++j) {
    const int gj = g0 + j;
    const int sb = gj % NSB;
    const uint32_t tS = tmem + lane_base + s_col + (uint32_t)(sb * BN);
    if (!tc::mbar_wait(&s_full[sb], (uint32_t)(gj / NSB) & 1u, abort_flag, status)) {
      if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
      ok = false;
      break;
    }
    tc::tc_fence_after();
    uint32_t r[BN];
#pragma unroll
    for (int c = 0; c < BN; c += 32) tc::tmem_ld32(tS + c, *reinterpret_cast<uint32_t(*)[32]>(&r[c]));
    tc::tmem_ld_wait();
    tc::tc_fence_before();
    tc::mbar_arrive(&s_free[sb]);  // S buffer sb may take S_{j+NSB}
    const int k0 = j * BN;
    int nvis = min(BN, p.S - k0);
    if (p.causal) nvis = min(nvis, max(0, qi - k0 + 1));
    if (nvis < BN) {
#pragma unroll
      for (int i = 0; i < BN; ++i)
        if (i >= nvis) r[i] = __float_as_uint(-INFINITY);
    }
    const float mxs = row_max<BN>(r) * p.scale_log2;
    float factor = 1.f;
    if (m_ref == -INFINITY) {
      m_ref = mxs;  // first visible scores: O and l are still zero
    } else if (mxs > m_ref + kRescaleLog2) {
      factor = exp2f(m_ref - mxs);
      m_ref = mxs;
    }
    if (__any_sync(0xffffffffu, factor != 1.f)) {
      if (!await_pv(gj - 1)) {  // O holds P_{j-1} V_{j-1}
        ok = false;
        break;
      }
#pragma unroll 1
      for (int c = 0; c < D; c += 32) {
        uint32_t o[32];
        tc::tmem_ld32(tO + c, o);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * factor);
        tc::tmem_st32(tO + c, o);
      }
      tc::tmem_st_wait();
    }
    const float mref = m_ref == -INFINITY ? 0.f : m_ref;
    const uint64_t sc2 = f2(p.scale_log2, p.scale_log2), nm2 = f2(-mref, -mref);
    uint64_t ls2[2] = {0ull, 0ull};
    uint32_t pk[BN / 2];
    exp_pack<BN>(r, sc2, nm2, pk, ls2);
    l = l * factor + sum_pairs(ls2);
    if (!await_pv(gj - 1)) {  // P_{j-1} V_{j-1} has read the P buffer
      ok = false;
      break;
    }
#pragma unroll
    for (int c = 0; c < BN / 2; c += 16) tc::tmem_st16(tP + c, *reinterpret_cast<uint32_t(*)[16]>(&pk[c]));
    tc::tmem_st_wait();
    tc::tc_fence_before();
    tc::mbar_arrive(p_full);
  }
  if (ok && nkb > 0) {
    if (await_pv(g0 + nkb - 1)) {
      const float inv_l = l > 0.f ? 1.f / l : 0.f;
      const bool row_ok = qi < p.S;
      __nv_bfloat16* orow = p.O + ((size_t)(b * p.S + (row_ok ? qi : 0)) * p.Hq + h) * D;
      store_o_row(tO, inv_l, orow, row_ok);
      if (p.lse && row_ok) p.lse[((size_t)b * p.Hq + h) * p.S + qi] = 0.6931471805599453f * (m_ref + log2f(l));
      if (o_free) {  // O has been read: the next item's first P V may overwrite it
        tc::tc_fence_before();
        tc::mbar_arrive(o_free);
      }
    }
  }
}

// TMEM layout of the one-tile kernel with NSB S buffers: S at 0 (and BN),
// then P and O. With one S buffer and BN = 64 the tile takes 256 columns
// (S 64, P 32, O 128 at column 128), so two CTAs share an SM: one CTA's
// softmax overlaps the other's tensor-core work, and a finishing CTA's tail
// overlaps its neighbour instead of idling the SM.
template <int BN, int NSB>
struct Attn4Cols {
  static constexpr uint32_t P = NSB == 2 ? 2 * BN + D : BN;
  static constexpr uint32_t O = NSB == 2 ? 2 * BN : (BN + BN / 2 + 127) / 128 * 128;
  static constexpr uint32_t END = NSB == 2 ? 2 * BN + D + BN / 2 : O + D;
  static constexpr uint32_t ALLOC = END <= 256 ? 256 : 512;
  static constexpr int CTAS_PER_SM = ALLOC == 256 ? 2 : 1;
};

// K ring depth = the schedule's stages; V ring depth. V_j is consumed one
// softmax period after K_j, so two-CTA-per-SM kernels keep at most two V
// slots and spend the shared memory on the K ring, whose refill latency (a
// K slot frees only when S_j completes) is what stalls S_{j+2}.
template <int BN, int NSB>
__host__ __device__ constexpr int attn4_vstages(int stages) {
  return Attn4Cols<BN, NSB>::CTAS_PER_SM == 2 && stages > 2 ? 2 : stages;
}
// Barrier words of attn4 after the rings: q_full, k_full/empty[stages],
// v_full/empty[vstages], s_full/s_free[2], p_full, pv_full, drain[2], then
// the TMEM address and the abort flag.
__host__ __device__ constexpr size_t attn4_bar_bytes(int stages, int vstages) {
  return (size_t)(9 + 2 * stages + 2 * vstages) * 8 + 8;
}
// Two CTAs per SM need the operands packed without alignment slack: the
// dynamic shared memory base is then required to be 1024-byte aligned (the
// kernel checks and reports RC_DEV_MISALIGNED otherwise).
template <int BN, int NSB>
size_t attn4_smem(int stages) {
  const int vst = attn4_vstages<BN, NSB>(stages);
  const size_t tiles = (size_t)BM * D * 2 + (size_t)(stages + vst) * BN * D * 2;
  return tiles + attn4_bar_bytes(stages, vst) + (Attn4Cols<BN, NSB>::CTAS_PER_SM == 2 ? 0 : 1024);
}

template <int BN, bool VT, int NSB>
__global__ void __launch_bounds__(kThreads4, (Attn4Cols<BN, NSB>::CTAS_PER_SM))
    attn4_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                 const __grid_constant__ CUtensorMap tmV, const Params p, const int stages) {
  static_assert(BN == 64 || BN == 128, "key block");
  static_assert(NSB == 1 || NSB == 2, "S buffers");
  constexpr int Q_BYTES = BM * D * 2;
  constexpr int KV_TILE = BN * D * 2;
  constexpr uint32_t O_COL = Attn4Cols<BN, NSB>::O, P_COL = Attn4Cols<BN, NSB>::P;
  constexpr uint32_t TMEM_COLS = Attn4Cols<BN, NSB>::ALLOC;

  extern __shared__ uint8_t smem_raw[];
  if constexpr (Attn4Cols<BN, NSB>::CTAS_PER_SM == 2) {
    // the operands are packed without alignment slack (two CTAs per SM)
    if (tc::smem_u32(smem_raw) & 1023u) {
      if (threadIdx.x == 0) tc::record_failure(p.status, RC_DEV_MISALIGNED);
      return;
    }
  }
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int vstages = attn4_vstages<BN, NSB>(stages);
  uint8_t* sQ = smem;
  uint8_t* kring = smem + Q_BYTES;
  uint8_t* vring = kring + (size_t)stages * KV_TILE;
  uint64_t* q_full = (uint64_t*)(vring + (size_t)vstages * KV_TILE);
  uint64_t* k_full = q_full + 1;      // [stages]
  uint64_t* k_empty = k_full + stages;
  uint64_t* v_full = k_empty + stages;  // [vstages]
  uint64_t* v_empty = v_full + vstages;
  uint64_t* s_full = v_empty + vstages;  // [2] S buffers
  uint64_t* s_free = s_full + 2;        // [2]
  uint64_t* p_full = s_free + 2;
  uint64_t* pv_full = p_full + 1;
  uint64_t* drain = pv_full + 1;        // [2] one per issuing warp
  uint32_t* tmem_slot = (uint32_t*)(drain + 2);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);
  volatile int* status = p.status;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int BH = p.B * p.Hq;
  int qb, bh;
  if (p.raster == 0) {
    qb = blockIdx.x % p.q_blocks;
    bh = blockIdx.x / p.q_blocks;
  } else {  // longest causal rows first
    qb = p.q_blocks - 1 - (int)(blockIdx.x / BH);
    bh = blockIdx.x % BH;
  }
  const int b = bh / p.Hq, h = bh - b * p.Hq, g = h / p.group;
  const int q0 = qb * BM;
  const int kv_end = p.causal ? min(q0 + BM, p.S) : p.S;
  const int nkb = (kv_end + BN - 1) / BN;

  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    tc::mbar_init(q_full, 1);
    for (int s = 0; s < stages; ++s) {
      tc::mbar_init(&k_full[s], 1);
      tc::mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < vstages; ++s) {
      tc::mbar_init(&v_full[s], 1);
      tc::mbar_init(&v_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&s_full[i], 1);
      tc::mbar_init(&s_free[i], 128);
      tc::mbar_init(&drain[i], 1);
    }
    tc::mbar_init(p_full, 128);
    tc::mbar_init(pv_full, 1);
    *abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc(tmem_slot, TMEM_COLS);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // slot s of a ring last held block j - stages; its release is the
  // ((j - stages) / stages)-th phase of empty[s], parity ph ^ 1 (a fresh
  // barrier passes that parity at once)
  auto produce = [&](uint64_t* full, uint64_t* empty, int depth, auto load) {
    int j = 0;
    for (; j < nkb; ++j) {
      const int s = j % depth;
      const uint32_t ph = (uint32_t)(j / depth) & 1u;
      if (!tc::mbar_wait(&empty[s], ph ^ 1u, abort_flag, status)) {
        fail(RC_DEV_TIMEOUT_EMPTY);
        break;
      }
      tc::mbar_expect_tx(&full[s], KV_TILE);
      load(s, j, &full[s]);
    }
    for (int i = max(0, j - depth); i < j; ++i)
      if (!tc::mbar_wait_drain(&full[i % depth], (uint32_t)(i / depth) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
  };

  if (warp == 0) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmK);
      tc::mbar_expect_tx(q_full, Q_BYTES);
      const int qrow = b * p.S + q0;
      tc::tma_load_2d(sQ, &tmQ, q_full, h * D, qrow);
      tc::tma_load_2d(sQ + Q_BYTES / 2, &tmQ, q_full, h * D + 64, qrow);
      produce(k_full, k_empty, stages, [&](int s, int j, uint64_t* bar) {
        uint8_t* sk = kring + (size_t)s * KV_TILE;
        const int krow = b * p.S + j * BN;
        tc::tma_load_2d(sk, &tmK, bar, g * D, krow);
        tc::tma_load_2d(sk + BN * 128, &tmK, bar, g * D + 64, krow);
      });
      if (!tc::mbar_wait_drain(q_full, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp == 3) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmV);
      produce(v_full, v_empty, vstages, [&](int s, int j, uint64_t* bar) {
        uint8_t* sv = vring + (size_t)s * KV_TILE;
        if constexpr (VT) {
#pragma unroll
          for (int a = 0; a < BN / 64; ++a)
            tc::tma_load_2d(sv + a * (BM * 128), &tmV, bar, j * BN + a * 64, (b * p.Hkv + g) * D);
        } else {
          const int krow = b * p.S + j * BN;
          tc::tma_load_2d(sv, &tmV, bar, g * D, krow);
          tc::tma_load_2d(sv + BN * 128, &tmV, bar, g * D + 64, krow);
        }
      });
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp == 1) {
    if (lane == 0 && nkb > 0) {
      constexpr uint32_t idS = tc::idesc_bf16_f32(BM, BN);
      const uint32_t sq = tc::smem_u32(sQ);
      auto issue_s = [&](int j) {
        const int s = j % stages;
        const uint32_t sk = tc::smem_u32(kring + (size_t)s * KV_TILE);
        const uint32_t tS = tmem + (uint32_t)((j % NSB) * BN);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          tc::umma_bf16(tS, tc::sw128_desc(sq + (ks / 4) * (BM * 128) + off),
                        tc::sw128_desc(sk + (ks / 4) * (BN * 128) + off), idS, ks > 0 ? 1u : 0u);
        }
        tc::umma_commit(&s_full[j % NSB]);
        tc::umma_commit(&k_empty[s]);
      };
      auto await_k = [&](int j) -> bool {
        return tc::mbar_wait(&k_full[j % stages], (uint32_t)(j / stages) & 1u, abort_flag, status);
      };
      bool ok = tc::mbar_wait(q_full, 0, abort_flag, status);
      for (int j = 0; ok && j < NSB && j < nkb; ++j) {
        if ((ok = await_k(j))) {
          tc::tc_fence_after();
          issue_s(j);
        }
      }
      for (int j = 0; ok && j + NSB < nkb; ++j) {
        // S buffer j % NSB is free once the softmax holds S_j in registers
        ok = tc::mbar_wait(&s_free[j % NSB], (uint32_t)(j / NSB) & 1u, abort_flag, status) && await_k(j + NSB);
        if (!ok) break;
        tc::tc_fence_after();
        issue_s(j + NSB);
      }
      if (!ok) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[0]);
        if (!tc::mbar_wait_drain(&drain[0], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else if (warp == 2) {
    if (lane == 0 && nkb > 0) {
      constexpr uint32_t idO = tc::idesc_bf16_f32(BM, D, !VT);
      const uint32_t tO = tmem + O_COL, tP = tmem + P_COL;
      bool ok = true;
      for (int j = 0; ok && j < nkb; ++j) {
        const int s = j % vstages;
        ok = tc::mbar_wait(&v_full[s], (uint32_t)(j / vstages) & 1u, abort_flag, status) &&
             tc::mbar_wait(p_full, (uint32_t)j & 1u, abort_flag, status);
        if (!ok) break;
        tc::tc_fence_after();
        const uint32_t sv = tc::smem_u32(vring + (size_t)s * KV_TILE);
#pragma unroll
        for (int ks = 0; ks < BN / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          uint64_t db;
          if constexpr (VT)
            db = tc::sw128_desc(sv + (ks / 4) * (BM * 128) + off);
          else
            db = tc::sw128_desc_mn(sv + (uint32_t)ks * 16 * 128, BN * 128, 1024);
          tc::umma_bf16_ts(tO, tP + (uint32_t)ks * 8, db, idO, (j > 0 || ks > 0) ? 1u : 0u);
        }
        tc::umma_commit(pv_full);
        tc::umma_commit(&v_empty[s]);
      }
      if (!ok) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[1]);
        if (!tc::mbar_wait_drain(&drain[1], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else {
    softmax_sdb<BN, NSB>(p, warp & 3, lane, q0, nkb, b, h, tmem, 0u, O_COL, P_COL, s_full, s_free, p_full, pv_full,
                         abort_flag, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, TMEM_COLS);
  }
}

// Persistent form of the one-tile, one-S-buffer kernel with 64-key blocks
// (Loop order 2). Two CTAs per SM stay resident and walk the query tiles,
// ordered longest first, in a zigzag over the CTAs (CTA c takes tiles c,
// 2G - 1 - c, 2G + c, ... of G CTAs), which pairs long causal tiles with
// short ones. TMEM, barriers and tensor maps are set up once; the K and V
// rings run on across tiles, so the next tile's keys stream in while the
// current one finishes; the next Q is loaded as soon as the current tile's
// last S UMMA has read Q (q_empty), and the next tile's first P V waits until
// the softmax warps have read O out (o_free). Every barrier's phase counts
// key blocks (or tiles) over the whole run of the CTA.
__host__ __device__ constexpr size_t attn4p_bar_bytes(int stages, int vstages) {
  return (size_t)(11 + 2 * stages + 2 * vstages) * 8 + 8;
}
size_t attn4p_smem(int stages) {
  const int vst = attn4_vstages<64, 1>(stages);
  return (size_t)BM * D * 2 + (size_t)(stages + vst) * 64 * D * 2 + attn4p_bar_bytes(stages, vst);
}

template <bool VT>
__global__ void __launch_bounds__(kThreads4, 2)
    attn4p_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, const Params p, const int stages) {
  constexpr int BN = 64;
  constexpr int Q_BYTES = BM * D * 2;
  constexpr int KV_TILE = BN * D * 2;
  constexpr uint32_t O_COL = Attn4Cols<BN, 1>::O, P_COL = Attn4Cols<BN, 1>::P;
  constexpr uint32_t TMEM_COLS = Attn4Cols<BN, 1>::ALLOC;
  static_assert(TMEM_COLS == 256, "two CTAs per SM");

  extern __shared__ uint8_t smem_raw[];
  if (tc::smem_u32(smem_raw) & 1023u) {  // operands packed without alignment slack
    if (threadIdx.x == 0) tc::record_failure(p.status, RC_DEV_MISALIGNED);
    return;
  }
  uint8_t* smem = smem_raw;
  const int vstages = attn4_vstages<BN, 1>(stages);
  uint8_t* sQ = smem;
  uint8_t* kring = smem + Q_BYTES;
  uint8_t* vring = kring + (size_t)stages * KV_TILE;
  uint64_t* q_full = (uint64_t*)(vring + (size_t)vstages * KV_TILE);
  uint64_t* q_empty = q_full + 1;
  uint64_t* k_full = q_empty + 1;  // [stages]
  uint64_t* k_empty = k_full + stages;
  uint64_t* v_full = k_empty + stages;  // [vstages]
  uint64_t* v_empty = v_full + vstages;
  uint64_t* s_full = v_empty + vstages;
  uint64_t* s_free = s_full + 1;
  uint64_t* p_full = s_free + 1;
  uint64_t* pv_full = p_full + 1;
  uint64_t* o_free = pv_full + 1;
  uint64_t* drain = o_free + 1;  // [2]
  uint32_t* tmem_slot = (uint32_t*)(drain + 2);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);
  volatile int* status = p.status;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int BH = p.B * p.Hq;
  const int n_tiles = p.q_blocks * BH;
  const int G = gridDim.x, c = blockIdx.x;
  // k-th work item of this CTA: a query tile in longest-first order, zigzag over the CTAs
  struct Work {
    bool valid;
    int q0, nkb, b, h, g;
  };
  auto work = [&](int k) -> Work {
    Work w;
    const long long t = (long long)k * G + ((k & 1) ? G - 1 - c : c);
    w.valid = t < n_tiles;
    if (!w.valid) return w;
    const int qb = p.q_blocks - 1 - (int)(t / BH), bh = (int)(t % BH);
    w.b = bh / p.Hq;
    w.h = bh - w.b * p.Hq;
    w.g = w.h / p.group;
    w.q0 = qb * BM;
    const int kv_end = p.causal ? min(w.q0 + BM, p.S) : p.S;
    w.nkb = (kv_end + BN - 1) / BN;
    return w;
  };
  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    tc::mbar_init(q_full, 1);
    tc::mbar_init(q_empty, 1);
    for (int s = 0; s < stages; ++s) {
      tc::mbar_init(&k_full[s], 1);
      tc::mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < vstages; ++s) {
      tc::mbar_init(&v_full[s], 1);
      tc::mbar_init(&v_empty[s], 1);
    }
    tc::mbar_init(s_full, 1);
    tc::mbar_init(s_free, 128);
    tc::mbar_init(p_full, 128);
    tc::mbar_init(pv_full, 1);
    tc::mbar_init(o_free, 128);
    tc::mbar_init(&drain[0], 1);
    tc::mbar_init(&drain[1], 1);
    *abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc(tmem_slot, TMEM_COLS);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // a ring of `depth` slots filled for blocks g = g0 .. g0 + n - 1 of the run
  auto produce = [&](uint64_t* full, uint64_t* empty, int depth, int g0, int n, auto load) -> bool {
    for (int j = 0; j < n; ++j) {
      const int g = g0 + j;
      const int s = g % depth;
      if (!tc::mbar_wait(&empty[s], ((uint32_t)(g / depth) & 1u) ^ 1u, abort_flag, status)) {
        fail(RC_DEV_TIMEOUT_EMPTY);
        return false;
      }
      tc::mbar_expect_tx(&full[s], KV_TILE);
      load(s, j, &full[s]);
    }
    return true;
  };
  auto drain_ring = [&](uint64_t* full, int depth, int g_end) {
    for (int g = max(0, g_end - depth); g < g_end; ++g)
      if (!tc::mbar_wait_drain(&full[g % depth], (uint32_t)(g / depth) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
  };

  if (warp == 0) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmK);
      int gk = 0, items = 0;
      bool ok = true;
      for (int k = 0; ok; ++k) {
        const Work w = work(k);
        if (!w.valid) break;
        if (k > 0 && !tc::mbar_wait(q_empty, (uint32_t)(k - 1) & 1u, abort_flag, status)) {
          fail(RC_DEV_TIMEOUT_EMPTY);
          break;
        }
        tc::mbar_expect_tx(q_full, Q_BYTES);
        const int qrow = w.b * p.S + w.q0;
        tc::tma_load_2d(sQ, &tmQ, q_full, w.h * D, qrow);
        tc::tma_load_2d(sQ + Q_BYTES / 2, &tmQ, q_full, w.h * D + 64, qrow);
        ++items;
        ok = produce(k_full, k_empty, stages, gk, w.nkb, [&](int s, int j, uint64_t* bar) {
          uint8_t* sk = kring + (size_t)s * KV_TILE;
          const int krow = w.b * p.S + j * BN;
          tc::tma_load_2d(sk, &tmK, bar, w.g * D, krow);
          tc::tma_load_2d(sk + BN * 128, &tmK, bar, w.g * D + 64, krow);
        });
        gk += w.nkb;
      }
      drain_ring(k_full, stages, gk);
      if (items > 0 && !tc::mbar_wait_drain(q_full, (uint32_t)(items - 1) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
    }
    __syncwarp();
  } else if (warp == 3) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmV);
      int gv = 0;
      bool ok = true;
      for (int k = 0; ok; ++k) {
        const Work w = work(k);
        if (!w.valid) break;
        ok = produce(v_full, v_empty, vstages, gv, w.nkb, [&](int s, int j, uint64_t* bar) {
          uint8_t* sv = vring + (size_t)s * KV_TILE;
          if constexpr (VT) {
            tc::tma_load_2d(sv, &tmV, bar, j * BN, (w.b * p.Hkv + w.g) * D);
          } else {
            const int krow = w.b * p.S + j * BN;
            tc::tma_load_2d(sv, &tmV, bar, w.g * D, krow);
            tc::tma_load_2d(sv + BN * 128, &tmV, bar, w.g * D + 64, krow);
          }
        });
        gv += w.nkb;
      }
      drain_ring(v_full, vstages, gv);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = tc::idesc_bf16_f32(BM, BN);
      const uint32_t sq = tc::smem_u32(sQ);
      int gs = 0;
      bool ok = true;
      for (int k = 0; ok; ++k) {
        const Work w = work(k);
        if (!w.valid) break;
        if (!tc::mbar_wait(q_full, (uint32_t)k & 1u, abort_flag, status)) {
          ok = false;
          break;
        }
        for (int j = 0; j < w.nkb; ++j) {
          const int g = gs + j;
          const int s = g % stages;
          // the S buffer is free once the softmax holds S_{g-1} in registers
          ok = (g == 0 || tc::mbar_wait(s_free, (uint32_t)(g - 1) & 1u, abort_flag, status)) &&
               tc::mbar_wait(&k_full[s], (uint32_t)(g / stages) & 1u, abort_flag, status);
          if (!ok) break;
          tc::tc_fence_after();
          const uint32_t sk = tc::smem_u32(kring + (size_t)s * KV_TILE);
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const uint32_t off = (uint32_t)(ks % 4) * 32;
            tc::umma_bf16(tmem, tc::sw128_desc(sq + (ks / 4) * (BM * 128) + off),
                          tc::sw128_desc(sk + (ks / 4) * (BN * 128) + off), idS, ks > 0 ? 1u : 0u);
          }
          tc::umma_commit(s_full);
          tc::umma_commit(&k_empty[s]);
        }
        if (!ok) break;
        tc::umma_commit(q_empty);  // Q may be replaced once this tile's S products are done
        gs += w.nkb;
      }
      if (!ok) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[0]);
        if (!tc::mbar_wait_drain(&drain[0], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else if (warp == 2) {
    if (lane == 0) {
      constexpr uint32_t idO = tc::idesc_bf16_f32(BM, D, !VT);
      const uint32_t tO = tmem + O_COL, tP = tmem + P_COL;
      int gp = 0;
      bool ok = true;
      for (int k = 0; ok; ++k) {
        const Work w = work(k);
        if (!w.valid) break;
        // O still holds the previous tile until its softmax warps have read it out
        if (k > 0 && !tc::mbar_wait(o_free, (uint32_t)(k - 1) & 1u, abort_flag, status)) {
          ok = false;
          break;
        }
        for (int j = 0; j < w.nkb; ++j) {
          const int g = gp + j;
          const int s = g % vstages;
          ok = tc::mbar_wait(&v_full[s], (uint32_t)(g / vstages) & 1u, abort_flag, status) &&
               tc::mbar_wait(p_full, (uint32_t)g & 1u, abort_flag, status);
          if (!ok) break;
          tc::tc_fence_after();
          const uint32_t sv = tc::smem_u32(vring + (size_t)s * KV_TILE);
#pragma unroll
          for (int ks = 0; ks < BN / 16; ++ks) {
            const uint32_t off = (uint32_t)(ks % 4) * 32;
            uint64_t db;
            if constexpr (VT)
              db = tc::sw128_desc(sv + (ks / 4) * (BM * 128) + off);
            else
              db = tc::sw128_desc_mn(sv + (uint32_t)ks * 16 * 128, BN * 128, 1024);
            tc::umma_bf16_ts(tO, tP + (uint32_t)ks * 8, db, idO, (j > 0 || ks > 0) ? 1u : 0u);
          }
          tc::umma_commit(pv_full);
          tc::umma_commit(&v_empty[s]);
        }
        gp += w.nkb;
      }
      if (!ok) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[1]);
        if (!tc::mbar_wait_drain(&drain[1], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else {
    int gsm = 0;
    for (int k = 0; !*abort_flag; ++k) {
      const Work w = work(k);
      if (!w.valid) break;
      softmax_sdb<BN, 1>(p, warp & 3, lane, w.q0, w.nkb, w.b, w.h, tmem, 0u, O_COL, P_COL, s_full, s_free, p_full,
                         pv_full, abort_flag, status, gsm, o_free);
      gsm += w.nkb;
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, TMEM_COLS);
  }
}

// Two query tiles per CTA with key blocks of 64 and a P buffer per tile
// (TileSize M = 256, N = 64, Parallel = 1). TMEM per tile t: S_t (64
// columns), P_t (32, two bf16 per column) and O_t (128): 448 columns. With P
// apart from S, S_{j+1} of a tile is issued as soon as its softmax holds S_j
// in registers, so the tensor pipe computes it while the softmax
// exponentiates, and the two tiles' softmax warpgroups run independently of
// each other. The UMMAs come from four warps (the S and the P V products of
// each tile), K and V from a producer warp each; a ring slot is refilled when
// every tile that read the block held there has released it.
//   warp 0      : TMA producer of Q (both tiles) and of the K ring
//   warp 1      : TMA producer of the V ring
//   warps 2, 3  : S_t = Q_t K_j^T issue for tile 0 / 1 (warp 2 also owns TMEM)
//   warps 4, 5  : O_t += P_t V_j issue for tile 0 / 1
//   warps 6..13 : softmax of tile (warp - 6) / 4, TMEM lane quadrant warp % 4
constexpr int kThreads5 = 448;

template <bool VT>
__global__ void __launch_bounds__(kThreads5, 1)
    attn5_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                 const __grid_constant__ CUtensorMap tmV, const Params p, const int stages) {
  constexpr int BN = 64;
  constexpr int Q_BYTES = BM * D * 2;
  constexpr int KV_TILE = BN * D * 2;
  constexpr uint32_t S_COL = 0, P_COL = 2 * BN, O_COL = 3 * BN;  // tile t: + t*BN, + t*BN/2, + t*D

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;  // [2] tiles
  uint8_t* kring = smem + 2 * Q_BYTES;
  uint8_t* vring = kring + (size_t)stages * KV_TILE;
  uint64_t* q_full = (uint64_t*)(vring + (size_t)stages * KV_TILE);
  uint64_t* k_full = q_full + 1;              // [stages]
  uint64_t* v_full = k_full + stages;         // [stages]
  uint64_t* k_empty = v_full + stages;        // [2 tiles][stages]
  uint64_t* v_empty = k_empty + 2 * stages;   // [2 tiles][stages]
  uint64_t* s_full = v_empty + 2 * stages;    // [2]
  uint64_t* s_free = s_full + 2;              // [2]
  uint64_t* p_full = s_free + 2;              // [2]
  uint64_t* pv_full = p_full + 2;             // [2]
  uint64_t* drain = pv_full + 2;              // [4] one per issuing warp
  uint32_t* tmem_slot = (uint32_t*)(drain + 4);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);
  volatile int* status = p.status;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int pairs = (p.q_blocks + 1) / 2;
  const int BH = p.B * p.Hq;
  int pb, bh;
  if (p.raster == 0) {
    pb = blockIdx.x % pairs;
    bh = blockIdx.x / pairs;
  } else {
    pb = pairs - 1 - (int)(blockIdx.x / BH);
    bh = blockIdx.x % BH;
  }
  const int b = bh / p.Hq, h = bh - b * p.Hq, g = h / p.group;
  int q0[2], nkb[2];
#pragma unroll
  for (int t = 0; t < 2; ++t) {
    q0[t] = (2 * pb + t) * BM;
    const int end = p.causal ? min(q0[t] + BM, p.S) : p.S;
    nkb[t] = q0[t] < p.S ? (end + BN - 1) / BN : 0;
  }
  const int nblk = max(nkb[0], nkb[1]);

  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    tc::mbar_init(q_full, 1);
    for (int s = 0; s < stages; ++s) {
      tc::mbar_init(&k_full[s], 1);
      tc::mbar_init(&v_full[s], 1);
    }
    for (int i = 0; i < 2 * stages; ++i) {
      tc::mbar_init(&k_empty[i], 1);
      tc::mbar_init(&v_empty[i], 1);
    }
    for (int t = 0; t < 2; ++t) {
      tc::mbar_init(&s_full[t], 1);
      tc::mbar_init(&s_free[t], 128);
      tc::mbar_init(&p_full[t], 128);
      tc::mbar_init(&pv_full[t], 1);
    }
    for (int i = 0; i < 4; ++i) tc::mbar_init(&drain[i], 1);
    *abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 2) tc::tmem_alloc(tmem_slot, 512);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Slot s of a ring last held key block j - stages; tile t read it iff
  // j - stages < nkb[t], and released it in the ((j - stages) / stages)-th
  // phase of its barrier for slot s (parity ph ^ 1; a fresh barrier passes).
  auto produce = [&](uint64_t* full, uint64_t* empty, auto load) {
    int j = 0;
    for (; j < nblk; ++j) {
      const int s = j % stages;
      const uint32_t ph = (uint32_t)(j / stages) & 1u;
      bool ok = true;
      for (int t = 0; t < 2 && ok; ++t)
        if (j - stages < nkb[t]) ok = tc::mbar_wait(&empty[t * stages + s], ph ^ 1u, abort_flag, status);
      if (!ok) {
        fail(RC_DEV_TIMEOUT_EMPTY);
        break;
      }
      tc::mbar_expect_tx(&full[s], KV_TILE);
      load(s, j, &full[s]);
    }
    for (int i = max(0, j - stages); i < j; ++i)
      if (!tc::mbar_wait_drain(&full[i % stages], (uint32_t)(i / stages) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
  };

  if (warp == 0) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmK);
      tc::mbar_expect_tx(q_full, 2 * Q_BYTES);
#pragma unroll
      for (int t = 0; t < 2; ++t) {
        const int qrow = b * p.S + q0[t];
        tc::tma_load_2d(sQ + t * Q_BYTES, &tmQ, q_full, h * D, qrow);
        tc::tma_load_2d(sQ + t * Q_BYTES + Q_BYTES / 2, &tmQ, q_full, h * D + 64, qrow);
      }
      produce(k_full, k_empty, [&](int s, int j, uint64_t* bar) {
        uint8_t* sk = kring + (size_t)s * KV_TILE;
        const int krow = b * p.S + j * BN;
        tc::tma_load_2d(sk, &tmK, bar, g * D, krow);
        tc::tma_load_2d(sk + BN * 128, &tmK, bar, g * D + 64, krow);
      });
      if (!tc::mbar_wait_drain(q_full, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp == 1) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmV);
      produce(v_full, v_empty, [&](int s, int j, uint64_t* bar) {
        uint8_t* sv = vring + (size_t)s * KV_TILE;
        if constexpr (VT) {
          tc::tma_load_2d(sv, &tmV, bar, j * BN, (b * p.Hkv + g) * D);
        } else {
          const int krow = b * p.S + j * BN;
          tc::tma_load_2d(sv, &tmV, bar, g * D, krow);
          tc::tma_load_2d(sv + BN * 128, &tmV, bar, g * D + 64, krow);
        }
      });
    }
    __syncwarp();
  } else if (warp <= 3) {  // S issue of tile warp - 2
    const int t = warp - 2;
    if (lane == 0 && nkb[t] > 0) {
      constexpr uint32_t idS = tc::idesc_bf16_f32(BM, BN);
      const uint32_t sq = tc::smem_u32(sQ + t * Q_BYTES);
      const uint32_t tS = tmem + S_COL + (uint32_t)(t * BN);
      bool ok = tc::mbar_wait(q_full, 0, abort_flag, status);
      for (int j = 0; ok && j < nkb[t]; ++j) {
        // the S buffer is free once the softmax holds S_{j-1} in registers
        if (j > 0) ok = tc::mbar_wait(&s_free[t], (uint32_t)(j - 1) & 1u, abort_flag, status);
        const int s = j % stages;
        ok = ok && tc::mbar_wait(&k_full[s], (uint32_t)(j / stages) & 1u, abort_flag, status);
        if (!ok) break;
        tc::tc_fence_after();
        const uint32_t sk = tc::smem_u32(kring + (size_t)s * KV_TILE);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t off = (uint32_t)(ks % 4) * 32;
          tc::umma_bf16(tS, tc::sw128_desc(sq + (ks / 4) * (BM * 128) + off),
                        tc::sw128_desc(sk + (ks / 4) * (BN * 128) + off), idS, ks > 0 ? 1u : 0u);
        }
        tc::umma_commit(&s_full[t]);
        tc::umma_commit(&k_empty[t * stages + s]);
      }
      if (!ok) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[t]);
        if (!tc::mbar_wait_drain(&drain[t], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else if (warp <= 5) {  // P V issue of tile warp - 4
    const int t = warp - 4;
    if (lane == 0 && nkb[t] > 0) {
      constexpr uint32_t idO = tc::idesc_bf16_f32(BM, D, !VT);
      const uint32_t tO = tmem + O_COL + (uint32_t)(t * D), tP = tmem + P_COL + (uint32_t)(t * BN / 2);
      bool ok = true;
      for (int j = 0; ok && j < nkb[t]; ++j) {
        const int s = j % stages;
        ok = tc::mbar_wait(&v_full[s], (uint32_t)(j / stages) & 1u, abort_flag, status) &&
             tc::mbar_wait(&p_full[t], (uint32_t)j & 1u, abort_flag, status);
        if (!ok) break;
        tc::tc_fence_after();
        const uint32_t sv = tc::smem_u32(vring + (size_t)s * KV_TILE);
#pragma unroll
        for (int ks = 0; ks < BN / 16; ++ks) {
          uint64_t db;
          if constexpr (VT)
            db = tc::sw128_desc(sv + (uint32_t)(ks % 4) * 32);
          else
            db = tc::sw128_desc_mn(sv + (uint32_t)ks * 16 * 128, BN * 128, 1024);
          tc::umma_bf16_ts(tO, tP + (uint32_t)ks * 8, db, idO, (j > 0 || ks > 0) ? 1u : 0u);
        }
        tc::umma_commit(&pv_full[t]);
        tc::umma_commit(&v_empty[t * stages + s]);
      }
      if (!ok) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[2 + t]);
        if (!tc::mbar_wait_drain(&drain[2 + t], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else {
    const int t = (warp - 6) / 4;
    softmax_sdb<BN, 1>(p, warp & 3, lane, q0[t], nkb[t], b, h, tmem, S_COL + (uint32_t)(t * BN),
                       O_COL + (uint32_t)(t * D), P_COL + (uint32_t)(t * BN / 2), &s_full[t], &s_free[t], &p_full[t],
                       &pv_full[t], abort_flag, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, 512);
  }
}

// Vt[(b*Hkv + g)*D + d][s] = V[b][s][g][d] (64 x 64 tiles through shared memory).
__global__ void transpose_v_kernel(const __nv_bfloat16* __restrict__ V, int S, int Hkv, __nv_bfloat16* __restrict__ Vt) {
  __shared__ __nv_bfloat16 tile[64][66];
  const int bg = blockIdx.z;  // b * Hkv + g
  const int b = bg / Hkv, g = bg - b * Hkv;
  const int s0 = blockIdx.x * 64, d0 = blockIdx.y * 64;
  for (int i = threadIdx.y; i < 64; i += blockDim.y) {
    const int s = s0 + i;
    for (int k = threadIdx.x; k < 64; k += blockDim.x)
      tile[i][k] = s < S ? V[(((size_t)b * S + s) * Hkv + g) * D + d0 + k] : __float2bfloat16_rn(0.f);
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 64; i += blockDim.y) {
    const int d = d0 + i;
    for (int k = threadIdx.x; k < 64; k += blockDim.x) {
      const int s = s0 + k;
      if (s < S) Vt[((size_t)bg * D + d) * S + s] = tile[k][i];
    }
  }
}

// Q tiles + K/V ring + P tiles + 1 KB alignment slack + barriers (at most
// 1 + 6 * stages + 8 of them, 8 B each, plus two words: 512 B for stages <= 5)
size_t smem_bytes(int bn, int stages, int qtiles) {
  return (size_t)qtiles * BM * D * 2 + (size_t)stages * 2 * bn * D * 2 + (size_t)qtiles * BM * bn * 2 + 1024 + 512;
}

template <int BN, bool VT, bool PINGPONG, bool PT = false, bool SDB = false, bool PAR = false>
rc_status launch(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V, void* O,
                 float* lse, const LaunchCtx& c) {
  static_assert(!PAR || (PT && !(SDB && PINGPONG)), "split UMMA issue: P in TMEM");
  // PAR: two query tiles with one issuing warp each (attn3), or one query tile
  // with one or two (SDB) S buffers and separate S and P V issuers (attn4)
  // (two tiles with BN = 64: P apart from S, four issuing warps, attn5)
  auto pick = []() {
    if constexpr (PAR && PINGPONG && BN == 64) return &attn5_kernel<VT>;
    else if constexpr (PAR && PINGPONG) return &attn3_kernel<BN, VT>;
    else if constexpr (PAR) return &attn4_kernel<BN, VT, SDB ? 2 : 1>;
    else if constexpr (PINGPONG) return &attn2_kernel<BN, VT, PT, SDB>;
    else return &attn_kernel<BN, VT>;
  };
  auto kern = pick();
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
    // the largest shared-memory carve-out, so that two 1-tile CTAs can share an SM
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "attention: smem attribute: %s", cudaGetErrorString(e));
    attr = true;
  }
  const uint64_t BS = (uint64_t)d.batch * d.seq;
  CUtensorMap tq, tk, tv;
  RC_TRY(tcg::encode_2d(&tq, Q, (uint64_t)d.heads_q * D, BS, BM));
  RC_TRY(tcg::encode_2d(&tk, K, (uint64_t)d.heads_kv * D, BS, BN));
  if (VT)
    RC_TRY(tcg::encode_2d(&tv, V, (uint64_t)d.seq, (uint64_t)d.batch * d.heads_kv * D, BM));
  else
    RC_TRY(tcg::encode_2d(&tv, V, (uint64_t)d.heads_kv * D, BS, BN));
  Params p;
  memset(&p, 0, sizeof p);
  p.B = (int)d.batch;
  p.S = (int)d.seq;
  p.Hq = (int)d.heads_q;
  p.Hkv = (int)d.heads_kv;
  p.group = (int)(d.heads_q / d.heads_kv);
  p.q_blocks = (int)((d.seq + BM - 1) / BM);
  p.causal = d.causal ? 1 : 0;
  p.scale_log2 = (float)(d.scale * 1.4426950408889634);
  p.raster = k.raster;
  p.O = (__nv_bfloat16*)O;
  p.lse = lse;
  p.status = c.status;
  const long long ctas = (long long)p.B * p.Hq * (PINGPONG ? (p.q_blocks + 1) / 2 : p.q_blocks);
  if (ctas > 0x7fffffffLL) return rc_fail(RC_ERR_UNSUPPORTED_OP, "attention: grid too large");
  const int qtiles = PINGPONG ? 2 : 1;
  size_t smem = smem_bytes(BN, k.stages, qtiles) - (PT ? (size_t)qtiles * BM * BN * 2 : 0);
  if constexpr (PAR && !PINGPONG) smem = attn4_smem<BN, SDB ? 2 : 1>(k.stages);
  const int threads = PAR ? (PINGPONG ? (BN == 64 ? kThreads5 : kThreads3) : kThreads4) : PINGPONG ? kThreads2 : kThreads;
  kern<<<(unsigned)ctas, threads, smem, (cudaStream_t)c.stream>>>(tq, tk, tv, p, k.stages);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    cudaFuncAttributes fa;
    memset(&fa, 0, sizeof fa);
    cudaFuncGetAttributes(&fa, kern);
    return rc_fail(RC_ERR_CUDA,
                   "attention launch: %s (%d threads, %zu B dynamic shared memory; kernel: %d registers, %zu B static "
                   "and at most %d B dynamic shared memory, at most %d threads)",
                   cudaGetErrorString(e), threads, smem, fa.numRegs, fa.sharedSizeBytes, fa.maxDynamicSharedSizeBytes,
                   fa.maxThreadsPerBlock);
  }
  return RC_OK;
}

// Persistent one-tile kernel (Loop order 2): grid = two CTAs per SM, at most one per tile.
template <bool VT>
rc_status launch_persistent(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V,
                            void* O, float* lse, const LaunchCtx& c) {
  auto kern = attn4p_kernel<VT>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "attention: smem attribute: %s", cudaGetErrorString(e));
    attr = true;
  }
  const uint64_t BS = (uint64_t)d.batch * d.seq;
  CUtensorMap tq, tk, tv;
  RC_TRY(tcg::encode_2d(&tq, Q, (uint64_t)d.heads_q * D, BS, BM));
  RC_TRY(tcg::encode_2d(&tk, K, (uint64_t)d.heads_kv * D, BS, 64));
  if (VT)
    RC_TRY(tcg::encode_2d(&tv, V, (uint64_t)d.seq, (uint64_t)d.batch * d.heads_kv * D, BM));
  else
    RC_TRY(tcg::encode_2d(&tv, V, (uint64_t)d.heads_kv * D, BS, 64));
  Params p;
  memset(&p, 0, sizeof p);
  p.B = (int)d.batch;
  p.S = (int)d.seq;
  p.Hq = (int)d.heads_q;
  p.Hkv = (int)d.heads_kv;
  p.group = (int)(d.heads_q / d.heads_kv);
  p.q_blocks = (int)((d.seq + BM - 1) / BM);
  p.causal = d.causal ? 1 : 0;
  p.scale_log2 = (float)(d.scale * 1.4426950408889634);
  p.raster = k.raster;
  p.O = (__nv_bfloat16*)O;
  p.lse = lse;
  p.status = c.status;
  const long long tiles = (long long)p.B * p.Hq * p.q_blocks;
  if (tiles > 0x7fffffffLL) return rc_fail(RC_ERR_UNSUPPORTED_OP, "attention: too many tiles");
  const int sms = c.num_sms > 0 ? c.num_sms : 1;
  const int grid = (int)std::min<long long>(tiles, 2LL * sms);
  kern<<<grid, kThreads4, attn4p_smem(k.stages), (cudaStream_t)c.stream>>>(tq, tk, tv, p, k.stages);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "attention (persistent) launch: %s", cudaGetErrorString(e));
  return RC_OK;
}

}  // namespace attn

rc_status rc_launch_attention(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V,
                              void* O, float* lse, void* workspace, const LaunchCtx& c) {
  if (d.head_dim != attn::D) return rc_fail(RC_ERR_UNSUPPORTED_OP, "attention: head_dim must be 128");
  if (d.batch * d.seq > 0x7fffffffLL) return rc_fail(RC_ERR_UNSUPPORTED_OP, "attention: B*S too large");
  const void* Vuse = V;
  if (k.layout == 1) {
    if (d.seq % 8) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: transposed V needs seq %% 8 == 0");
    dim3 grid((unsigned)((d.seq + 63) / 64), attn::D / 64, (unsigned)(d.batch * d.heads_kv));
    attn::transpose_v_kernel<<<grid, dim3(64, 8), 0, (cudaStream_t)c.stream>>>(
        (const __nv_bfloat16*)V, (int)d.seq, (int)d.heads_kv, (__nv_bfloat16*)workspace);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "V transpose launch: %s", cudaGetErrorString(e));
    Vuse = workspace;
  }
  const bool vt = k.layout == 1;
  const bool pp = k.tile_m == 256;  // two query tiles per CTA, ping-pong softmax
  if (pp && k.stages < 2) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: ping-pong needs >= 2 stages");
  const bool pt = k.location == 1;  // P kept in tensor memory
  if (pt && !pp && k.persistent != 1)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: P in TMEM needs two query tiles or split UMMA issue");
  const bool par = k.persistent == 1;  // UMMA issue split over several warps
  if (k.raster == 2) {  // persistent CTAs over longest-first tiles (one-tile kernel, one S buffer, BN 64)
    if (!(par && pt && !pp && k.tile_n == 64 && k.unroll == 1 && k.stages >= 2 && k.stages <= 3))
      return rc_fail(RC_ERR_ILLEGAL_SCHEDULE,
                     "attention: loop order 2 needs one query tile, split issue, P in TMEM, BN 64, unroll 1, 2-3 stages");
    return vt ? attn::launch_persistent<true>(k, d, Q, K, Vuse, O, lse, c)
              : attn::launch_persistent<false>(k, d, Q, K, Vuse, O, lse, c);
  }
  if (k.unroll == 2 && !(par && !pp)) {  // two key blocks in flight per query tile
    if (!(pp && pt && k.tile_n == 64 && k.stages >= 4) || k.persistent)
      return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: unroll 2 needs 2 query tiles, P in TMEM, BN 64, 4 stages");
    return vt ? attn::launch<64, true, true, true, true>(k, d, Q, K, Vuse, O, lse, c)
              : attn::launch<64, false, true, true, true>(k, d, Q, K, Vuse, O, lse, c);
  }
  const bool sdb = k.unroll == 2;  // one tile, split issue: two S buffers (two key blocks in flight)
  if (par && !pt) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: split UMMA issue needs P in TMEM");
  if (par && !pp && k.stages < 2)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: two S buffers need at least two K/V stages");
#define RC_ATT(BN)                                                                                  \
  if (k.tile_n == BN) {                                                                             \
    if (par && pp) return vt ? attn::launch<BN, true, true, true, false, true>(k, d, Q, K, Vuse, O, lse, c) \
                             : attn::launch<BN, false, true, true, false, true>(k, d, Q, K, Vuse, O, lse, c); \
    if (par && sdb) return vt ? attn::launch<BN, true, false, true, true, true>(k, d, Q, K, Vuse, O, lse, c) \
                              : attn::launch<BN, false, false, true, true, true>(k, d, Q, K, Vuse, O, lse, c); \
    if (par) return vt ? attn::launch<BN, true, false, true, false, true>(k, d, Q, K, Vuse, O, lse, c) \
                       : attn::launch<BN, false, false, true, false, true>(k, d, Q, K, Vuse, O, lse, c); \
    if (pp && pt) return vt ? attn::launch<BN, true, true, true>(k, d, Q, K, Vuse, O, lse, c)       \
                            : attn::launch<BN, false, true, true>(k, d, Q, K, Vuse, O, lse, c);     \
    if (pp) return vt ? attn::launch<BN, true, true>(k, d, Q, K, Vuse, O, lse, c)                   \
                      : attn::launch<BN, false, true>(k, d, Q, K, Vuse, O, lse, c);                 \
    return vt ? attn::launch<BN, true, false>(k, d, Q, K, Vuse, O, lse, c)                          \
              : attn::launch<BN, false, false>(k, d, Q, K, Vuse, O, lse, c);                        \
  }
  RC_ATT(64)
  RC_ATT(128)
#undef RC_ATT
  return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: key block %d", k.tile_n);
}
