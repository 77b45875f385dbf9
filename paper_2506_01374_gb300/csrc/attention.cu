// Fused attention core O = softmax(scale * Q K^T + mask) V with grouped-query
// heads, on the sm_103a tensor cores (tcgen05, TMEM accumulators, TMA).
//
// One CTA owns one (batch, query head h, block of 128 queries); the KV head is
// g = h / (Hq / Hkv). Per key block j of BN keys, S_j = Q K_j^T is computed
// into TMEM, the softmax threads read it (one query row per thread, or per
// two threads), keep the running row maximum m and sum l in the log2 domain
// (p = 2^(s * scale * log2 e - m)), rescale O in TMEM when m grows by more
// than 2^8, and write P_j as bf16; the tensor core then adds P_j V_j to O.
// The epilogue divides O by l and stores bf16 O and LSE = ln 2 * (m + log2 l).
//
// Three kernel families, chosen by the schedule's Parallel and TileSize M
// knobs:
//   Parallel 0: attn_kernel - one warp issues every UMMA, P goes through
//      shared memory (the unoptimised program P0);
//   Parallel 1, 2: attn4_kernel - S and P V issued by warps of their own, P
//      in TMEM, one or two S buffers (Unroll), one or two softmax threads per
//      row (Parallel 2), and optionally the row sums formed by the tensor
//      core (ComputeLocation 2);
//   TileSize M 256: attn2q_kernel - two 128-row query tiles per CTA sharing
//      each 128-key K and V block, one CTA per SM, the tensor core working on
//      one tile while the other's softmax runs.
// Other knobs: BN (TileSize N), ring depth (PipelineStages), query-block
// order (natural or longest causal rows first), and the layout of V: as given
// ([keys][d], an MN-major UMMA B operand) or pre-transposed by a pass into
// [d][keys] (K-major). Masking: key j is visible to query i when j < S and
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

// p_i = 2^(s_i * scale_log2 - mref) for N raw scores, two at a time: the
// exponent pair is formed in fp32 (packed FMA), rounded to bf16 and raised by
// one ex2.approx.ftz.bf16x2, which yields the packed bf16 pair the P V UMMA
// reads. No row sum is kept here: the tensor core forms it (a block of ones
// appended to V). Rounding the exponent to bf16 moves p by at most
// ln 2 * |x| * 2^-9 relative, i.e. at most about 2.7e-3 * 2^x absolutely,
// within about 1.4 times the bf16 rounding of p itself.
template <int N>
__device__ __forceinline__ void exp_pack_bf16(const uint32_t* r, uint64_t sc2, uint64_t nm2, uint32_t* pk) {
#pragma unroll
  for (int i = 0; i < N; i += 2) {
    const uint64_t x = f2_fma(f2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])), sc2, nm2);
    float x0, x1;
    f2_split(x, x0, x1);
    uint32_t e;
    asm("ex2.approx.ftz.bf16x2 %0, %1;" : "=r"(e) : "r"(pack2(x0, x1)));
    pk[i / 2] = e;
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

// One query tile per CTA with the UMMAs issued by warps of their own
// (Parallel 1 and 2). The S and the P V products come from two issuing warps
// (one thread needs about as long to issue a 128 x 128 x 16 UMMA as the pipe
// needs to run it), and K and V stream through rings of their own, each
// filled by its own producer warp.
//   warp 0          : TMA producer of Q and of the K ring
//   warp 1          : issues S_j = Q K_j^T (and owns TMEM)
//   warp 2          : issues O += P_j V_j
//   warp 3          : TMA producer of the V ring
//   warps 4..4+4S-1 : softmax (TMEM lane quadrant = warp % 4), S = 1 or 2 threads per query row
// With one S buffer (Unroll 1) S_{j+1} is issued as soon as the softmax holds
// S_j in registers and P has columns of its own; with two (Unroll 2) S_{j+1}
// is computed while the softmax works on S_j and P_j is written over its own
// S buffer, which takes S_{j+2} once P_j V_j has completed. At BN = 64 both
// fit 256 TMEM columns, so two CTAs share an SM and one CTA's softmax
// overlaps the other's UMMAs. ComputeLocation 2 lets the P V UMMA also form
// the row sums of P (a block of ones appended to V) and takes the
// exponentials in bf16 pairs.
constexpr float kRescaleLog2 = 8.0f;  // O is rescaled only when the row maximum grows by more than 2^8
constexpr int kThreads4 = 256;

// Normalised output columns [c0, c0 + NC) of one row, 32 columns per TMEM load.
template <int NC>
__device__ __forceinline__ void store_o_cols(uint32_t tO, float inv_l, __nv_bfloat16* orow, bool row_ok) {
#pragma unroll
  for (int c = 0; c < NC; c += 32) {
    uint32_t o[32];
    tc::tmem_ld32(tO + c, o);
    tc::tmem_ld_wait();
    if (row_ok) {
#pragma unroll
      for (int i = 0; i < 32; i += 8) {
        uint32_t pk[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          pk[u] = pack2(__uint_as_float(o[i + 2 * u]) * inv_l, __uint_as_float(o[i + 2 * u + 1]) * inv_l);
        *reinterpret_cast<uint4*>(orow + c + i) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
      }
    }
  }
}

// Row exchange between the two softmax threads of a row (SPLIT = 2): warps
// 4 + qd and 8 + qd read the same TMEM lanes, one half of the key columns
// each. Each block they swap their half-row maxima through `xch`
// ([2 parities][2 halves][128 rows] floats) and an mbarrier per lane
// quadrant and block parity (64 arrivals), whose waits are bounded like every
// other wait; at the end they swap their half-row sums the same way.
struct RowXchg {
  float* xch;
  uint64_t* xbar;  // [4 quadrants][2 parities]
  // Publish v for (row, half) in exchange number n and return the partner's.
  __device__ __forceinline__ bool swap(int n, int qd, int half, int row, float& v, volatile int* abort_flag,
                                       volatile int* status) const {
    float* slot = xch + (n & 1) * 256;
    slot[half * 128 + row] = v;
    uint64_t* bar = xbar + qd * 2 + (n & 1);
    tc::mbar_arrive(bar);  // release: the store above is visible to the partner after its wait
    if (!tc::mbar_wait(bar, (uint32_t)(n >> 1) & 1u, abort_flag, status)) return false;
    v = slot[(half ^ 1) * 128 + row];
    return true;
  }
};

// Softmax of the one-tile kernel. NSB S buffers at TMEM columns s_col + b * BN
// (block j in buffer j % NSB), O at o_col. With one S buffer P has columns of
// its own at p_col; with two, P_j is written over the first BN / 2 columns of
// its own S buffer (S_j is in registers by then), so the tile needs no P
// columns and S_{j+1} is computed while the softmax works on S_j. SPLIT
// threads share a row: thread `half` exponentiates keys
// [half * BN / SPLIT, + BN / SPLIT) of every block and owns O columns
// [half * D / SPLIT, + D / SPLIT); the row maximum is exchanged every block
// (both threads then take the same rescale decisions) and the row sum once at
// the end. p_full / pv_full: one barrier per S buffer with two buffers (block
// i completes phase i / 2 of barrier i % 2), else one. SUMC: the row sums of
// P come from the tensor core (O's columns D .. D + 15) and the exponentials
// are taken in bf16 pairs.
template <int BN, int NSB, int SPLIT, bool SUMC = false>
__device__ __forceinline__ void softmax_sdb(const Params& p, int qd, int half, int lane, int q0, int nkb, int b, int h,
                                            uint32_t tmem, uint32_t s_col, uint32_t o_col, uint32_t p_col,
                                            uint64_t* s_full, uint64_t* s_free, uint64_t* p_full, uint64_t* pv_full,
                                            RowXchg xc, volatile int* abort_flag, volatile int* status) {
  static_assert(SPLIT == 1 || SPLIT == 2, "threads per row");

  constexpr bool PA = NSB == 2;     // P written over its S buffer
  constexpr int NPV = PA ? 2 : 1;   // P and P V barriers
  constexpr int KN = BN / SPLIT;  // keys per block and thread
  constexpr int OC = D / SPLIT;   // O columns per thread
  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };
  const int row = 32 * qd + lane;
  const int qi = q0 + row;
  const uint32_t lane_base = (uint32_t)(32 * qd) << 16;
  const uint32_t tO = tmem + lane_base + o_col + (uint32_t)(half * OC);
  float m_ref = -INFINITY, l = 0.f;
  // P V of block i completes phase i / NPV of pv_full[i % NPV]; the phases are
  // observed one by one, in block order, never more than one behind on either
  // barrier: block j - 1 in iteration j (before an O rescale; with one S
  // buffer also before P_j overwrites P_{j-1}), the last one before the
  // output.
  int pv_seen = 0;
  auto await_pv = [&](int upto) -> bool {
    if (pv_seen > upto) return true;
    for (; pv_seen <= upto; ++pv_seen)
      if (!tc::mbar_wait(&pv_full[pv_seen % NPV], (uint32_t)(pv_seen / NPV) & 1u, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        return false;
      }
    tc::tc_fence_after();
    return true;
  };
  bool ok = true;
  for (int j = 0; j < nkb; ++j) {
    const int gj = j;
    const int sb = gj % NSB;
    const uint32_t tS = tmem + lane_base + s_col + (uint32_t)(sb * BN + half * KN);
    if (!tc::mbar_wait(&s_full[sb], (uint32_t)(gj / NSB) & 1u, abort_flag, status)) {
      if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
      ok = false;
      break;
    }
    tc::tc_fence_after();
    // two S buffers: S_j went into the buffer once P_{j-2} V_{j-2} had completed, so
    // observing that completion here never stalls and keeps the softmax at most one
    // phase behind on each P V barrier
    if (PA && !await_pv(gj - 2)) {
      ok = false;
      break;
    }
    uint32_t r[KN];
#pragma unroll
    for (int c = 0; c < KN; c += 32) tc::tmem_ld32(tS + c, *reinterpret_cast<uint32_t(*)[32]>(&r[c]));
    tc::tmem_ld_wait();
    if constexpr (!PA) {
      tc::tc_fence_before();
      tc::mbar_arrive(&s_free[sb]);  // S buffer sb may take S_{j+NSB}
    }
    const int k0 = j * BN + half * KN;
    int nvis = min(KN, p.S - k0);
    if (p.causal) nvis = min(nvis, max(0, qi - k0 + 1));
    if (nvis < KN) {
#pragma unroll
      for (int i = 0; i < KN; ++i)
        if (i >= nvis) r[i] = __float_as_uint(-INFINITY);
    }
    float mx = row_max<KN>(r);
    if constexpr (SPLIT == 2) {
      float other = mx;
      if (!xc.swap(gj, qd, half, row, other, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        ok = false;
        break;
      }
      mx = fmaxf(mx, other);  // the same row maximum in both threads of the row
    }
    const float mxs = mx * p.scale_log2;
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
      constexpr int RC = SPLIT == 1 ? 32 : 16;  // columns per TMEM round trip (registers)
      if (SUMC && half == 0) {  // the row-sum columns after O (rescaled once per row)
        uint32_t o[16];
        tc::tmem_ld16(tO + D, o);  // half 0: tO is the row's first O column
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * factor);
        tc::tmem_st16(tO + D, o);
      }
#pragma unroll 1
      for (int c = 0; c < OC; c += RC) {
        uint32_t o[RC];
        if constexpr (RC == 32) {
          tc::tmem_ld32(tO + c, o);
        } else {
          tc::tmem_ld16(tO + c, o);
        }
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < RC; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * factor);
        if constexpr (RC == 32) {
          tc::tmem_st32(tO + c, o);
        } else {
          tc::tmem_st16(tO + c, o);
        }
      }
      tc::tmem_st_wait();
    }
    const float mref = m_ref == -INFINITY ? 0.f : m_ref;
    const uint64_t sc2 = f2(p.scale_log2, p.scale_log2), nm2 = f2(-mref, -mref);
    uint32_t pk[KN / 2];
    if constexpr (SUMC) {
      exp_pack_bf16<KN>(r, sc2, nm2, pk);  // the sum of P accumulates in O's last columns
    } else {
      uint64_t ls2[2] = {0ull, 0ull};
      exp_pack<KN>(r, sc2, nm2, pk, ls2);
      l = l * factor + sum_pairs(ls2);
    }
    // P_j goes over S_j (already in registers; the P V that last read this
    // buffer completed before S_j was computed into it), else into the P
    // columns once P_{j-1} V_{j-1} has read them
    if (!PA && !await_pv(gj - 1)) {
      ok = false;
      break;
    }
    const uint32_t tP = tmem + lane_base + (PA ? s_col + (uint32_t)(sb * BN) : p_col) + (uint32_t)(half * KN / 2);
#pragma unroll
    for (int c = 0; c < KN / 2; c += 16) tc::tmem_st16(tP + c, *reinterpret_cast<uint32_t(*)[16]>(&pk[c]));
    tc::tmem_st_wait();
    tc::tc_fence_before();
    tc::mbar_arrive(&p_full[PA ? sb : 0]);
  }
  if (ok && nkb > 0) {
    if constexpr (SPLIT == 2 && !SUMC) {  // the row sum is the two halves' sums
      float lp = l;
      if (!xc.swap(nkb, qd, half, row, lp, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        ok = false;
      }
      l += lp;
    }
    if (ok && await_pv(nkb - 1)) {
      if constexpr (SUMC) {  // l = the row sum the P V UMMAs accumulated next to O
        uint32_t o[16];
        tc::tmem_ld16(tO - half * OC + D, o);
        tc::tmem_ld_wait();
        l = __uint_as_float(o[0]);
      }
      const float inv_l = l > 0.f ? 1.f / l : 0.f;
      const bool row_ok = qi < p.S;
      __nv_bfloat16* orow = p.O + ((size_t)(b * p.S + (row_ok ? qi : 0)) * p.Hq + h) * D + half * OC;
      if constexpr (SPLIT == 1) {
        store_o_row(tO, inv_l, orow, row_ok);
      } else {
        store_o_cols<OC>(tO, inv_l, orow, row_ok);
      }
      if (p.lse && row_ok && half == 0)
        p.lse[((size_t)b * p.Hq + h) * p.S + qi] = 0.6931471805599453f * (m_ref + log2f(l));
    }
  }
}

// TMEM layout of the one-tile kernel with NSB S buffers: S at 0 (and BN),
// then P (one S buffer) and O. With BN = 64 the tile takes 256 columns (one S
// buffer: S 64, P 32, O 128 at column 128; two: S 2 x 64, O 128), so two
// CTAs share an SM: one CTA's softmax overlaps the other's tensor-core work,
// and a finishing CTA's tail overlaps its neighbour instead of idling the SM.
template <int BN, int NSB, bool SUMC = false>
struct Attn4Cols {
  // SUMC (one S buffer): O has D + 16 columns, the last 16 holding the row
  // sums of P; S at 0, O at BN, P after O
  static constexpr uint32_t OW = SUMC ? D + 16 : D;
  static constexpr uint32_t P = NSB == 2 ? 0 : SUMC ? BN + OW : BN;  // two S buffers: P over its S buffer
  static constexpr uint32_t O = NSB == 2 ? 2 * BN : SUMC ? BN : (BN + BN / 2 + 127) / 128 * 128;
  static constexpr uint32_t END = NSB == 2 ? O + OW : SUMC ? P + BN / 2 : O + D;
  static constexpr uint32_t ALLOC = END <= 256 ? 256 : 512;
  static constexpr int CTAS_PER_SM = ALLOC == 256 ? 2 : 1;
};

// K ring depth = the schedule's stages; V ring depth. V_j is consumed one
// softmax period after K_j, so two-CTA-per-SM kernels keep at most two V
// slots and spend the shared memory on the K ring, whose refill latency (a
// K slot frees only when S_j completes) is what stalls S_{j+2}.
template <int BN, int NSB, bool SUMC = false>
__host__ __device__ constexpr int attn4_vstages(int stages) {
  return Attn4Cols<BN, NSB, SUMC>::CTAS_PER_SM == 2 && stages > 2 ? 2 : stages;
}
// Bytes of a V ring slot: the BN x 128 tile, and with row sums on the tensor
// core a third 64-column atom of ones (N = 128 + 16 for the P V UMMA).
template <int BN, bool SUMC>
__host__ __device__ constexpr size_t attn4_vslot() {
  return (size_t)BN * D * 2 + (SUMC ? (size_t)BN * 128 : 0);
}
// Barrier words of attn4 after the rings: q_full, k_full/empty[stages],
// v_full/empty[vstages], s_full/s_free[2], p_full[2], pv_full[2], drain[2],
// the row-exchange barriers [4][2] with two softmax threads per row, then the
// TMEM address and the abort flag.
__host__ __device__ constexpr size_t attn4_bar_bytes(int stages, int vstages, int split) {
  return (size_t)(11 + 2 * stages + 2 * vstages + (split == 2 ? 8 : 0)) * 8 + 8;
}
// Row-exchange area of the two-threads-per-row softmax: [2][2][128] floats.
__host__ __device__ constexpr size_t attn4_xch_bytes(int split) { return split == 2 ? 2048 : 0; }
// Two CTAs per SM need the operands packed without alignment slack: the
// dynamic shared memory base is then required to be 1024-byte aligned (the
// kernel checks and reports RC_DEV_MISALIGNED otherwise).
template <int BN, int NSB, int SPLIT = 1, bool SUMC = false>
size_t attn4_smem(int stages) {
  const int vst = attn4_vstages<BN, NSB, SUMC>(stages);
  const size_t tiles = (size_t)BM * D * 2 + (size_t)stages * BN * D * 2 + (size_t)vst * attn4_vslot<BN, SUMC>();
  return tiles + attn4_xch_bytes(SPLIT) + attn4_bar_bytes(stages, vst, SPLIT) +
         (Attn4Cols<BN, NSB, SUMC>::CTAS_PER_SM == 2 ? 0 : 1024);
}

// Threads of the one-tile kernel: four producer / UMMA warps and 4 * SPLIT softmax warps.
template <int SPLIT>
constexpr int attn4_threads() {
  return kThreads4 + 128 * (SPLIT - 1);
}

template <int BN, bool VT, int NSB, int SPLIT = 1, bool SUMC = false>
__global__ void __launch_bounds__(attn4_threads<SPLIT>(), (Attn4Cols<BN, NSB, SUMC>::CTAS_PER_SM))
    attn4_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                 const __grid_constant__ CUtensorMap tmV, const Params p, const int stages) {
  static_assert(BN == 64 || BN == 128, "key block");
  static_assert(NSB == 1 || NSB == 2, "S buffers");
  static_assert(SPLIT == 1 || SPLIT == 2, "softmax threads per row");
  static_assert(!SUMC || !VT, "row sums on the tensor core: V as given");
  constexpr int Q_BYTES = BM * D * 2;
  constexpr int KV_TILE = BN * D * 2;
  constexpr size_t VSLOT = attn4_vslot<BN, SUMC>();
  using Cols = Attn4Cols<BN, NSB, SUMC>;
  constexpr uint32_t O_COL = Cols::O, P_COL = Cols::P;
  constexpr uint32_t TMEM_COLS = Cols::ALLOC;

  extern __shared__ uint8_t smem_raw[];
  if constexpr (Cols::CTAS_PER_SM == 2) {
    // the operands are packed without alignment slack (two CTAs per SM)
    if (tc::smem_u32(smem_raw) & 1023u) {
      if (threadIdx.x == 0) tc::record_failure(p.status, RC_DEV_MISALIGNED);
      return;
    }
  }
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int vstages = attn4_vstages<BN, NSB, SUMC>(stages);
  uint8_t* sQ = smem;
  uint8_t* kring = smem + Q_BYTES;
  uint8_t* vring = kring + (size_t)stages * KV_TILE;
  float* xch = (float*)(vring + (size_t)vstages * VSLOT);  // SPLIT == 2: [2][2][128]
  uint64_t* q_full = (uint64_t*)((uint8_t*)xch + attn4_xch_bytes(SPLIT));
  uint64_t* k_full = q_full + 1;      // [stages]
  uint64_t* k_empty = k_full + stages;
  uint64_t* v_full = k_empty + stages;  // [vstages]
  uint64_t* v_empty = v_full + vstages;
  uint64_t* s_full = v_empty + vstages;  // [2] S buffers
  uint64_t* s_free = s_full + 2;        // [2]
  uint64_t* p_full = s_free + 2;        // [2] one per S buffer with two (P over S)
  uint64_t* pv_full = p_full + 2;       // [2]
  uint64_t* drain = pv_full + 2;        // [2] one per issuing warp
  uint64_t* xbar = drain + 2;           // SPLIT == 2: [4][2]
  uint32_t* tmem_slot = (uint32_t*)(xbar + (SPLIT == 2 ? 8 : 0));
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
      tc::mbar_init(&s_free[i], 128 * SPLIT);
      tc::mbar_init(&p_full[i], 128 * SPLIT);
      tc::mbar_init(&pv_full[i], 1);
      tc::mbar_init(&drain[i], 1);
    }
    if constexpr (SPLIT == 2)
      for (int i = 0; i < 8; ++i) tc::mbar_init(&xbar[i], 64);
    *abort_flag = 0;
    tc::fence_mbar_init();
  }
  if constexpr (SUMC) {
    // the ones atom of every V slot (bf16 1.0): P V then also accumulates sum_j P_j in O's
    // columns D .. D + 15; written once, through the generic proxy, before any UMMA reads it
    for (int s = 0; s < vstages; ++s) {
      uint4* ones = (uint4*)(vring + (size_t)s * VSLOT + (size_t)KV_TILE);
      for (int i = threadIdx.x; i < BN * 128 / 16; i += blockDim.x)
        ones[i] = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    }
    tc::fence_proxy_async_smem();
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
        uint8_t* sv = vring + (size_t)s * VSLOT;
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
    // S issuer. The whole warp runs the loop on warp-uniform values and one lane (elect.sync)
    // issues: a lane-0 branch spends far longer per UMMA forming its operands.
    if (nkb > 0) {
      const bool leader = tc::elect_one();
      auto all = [](bool x) { return __all_sync(0xffffffffu, x); };
      constexpr uint32_t idS = tc::idesc_bf16_f32(BM, BN);
      const uint64_t q_desc = tc::sw128_desc(tc::smem_u32(sQ));
      const uint64_t k_desc = tc::sw128_desc(tc::smem_u32(kring));
      auto issue_s = [&](int j) {
        const int s = j % stages;
        if (leader) {
          const uint64_t kd = k_desc + (uint64_t)(s * (KV_TILE >> 4));
          const uint32_t tS = tmem + (uint32_t)((j % NSB) * BN);
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            // 16-wide K steps: 32 B within a 64-wide swizzled half, halves [BM or BN][64] apart
            tc::umma_bf16(tS, q_desc + (uint64_t)((ks / 4) * ((BM * 128) >> 4) + (ks % 4) * 2),
                          kd + (uint64_t)((ks / 4) * ((BN * 128) >> 4) + (ks % 4) * 2), idS, ks > 0 ? 1u : 0u);
          }
          tc::umma_commit(&s_full[j % NSB]);
          tc::umma_commit(&k_empty[s]);
        }
        __syncwarp();
      };
      auto await_k = [&](int j) -> bool {
        return all(tc::mbar_wait(&k_full[j % stages], (uint32_t)(j / stages) & 1u, abort_flag, status));
      };
      bool ok = all(tc::mbar_wait(q_full, 0, abort_flag, status));
      for (int j = 0; ok && j < NSB && j < nkb; ++j) {
        if ((ok = await_k(j))) {
          tc::tc_fence_after();
          issue_s(j);
        }
      }
      for (int j = 0; ok && j + NSB < nkb; ++j) {
        // one S buffer: free once the softmax holds S_j in registers; two: S buffer j % 2
        // holds P_j, free once P_j V_j has completed
        if constexpr (NSB == 1)
          ok = all(tc::mbar_wait(&s_free[0], (uint32_t)j & 1u, abort_flag, status));
        else
          ok = all(tc::mbar_wait(&pv_full[j % 2], (uint32_t)(j / 2) & 1u, abort_flag, status));
        ok = ok && await_k(j + NSB);
        if (!ok) break;
        tc::tc_fence_after();
        issue_s(j + NSB);
      }
      if (!ok && leader) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[0]);
        if (!tc::mbar_wait_drain(&drain[0], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else if (warp == 2) {
    // P V issuer, warp-uniform like the S issuer
    if (nkb > 0) {
      const bool leader = tc::elect_one();
      auto all = [](bool x) { return __all_sync(0xffffffffu, x); };
      constexpr uint32_t idO = tc::idesc_bf16_f32(BM, (int)Cols::OW, !VT);
      const uint32_t tO = tmem + O_COL;
      const uint64_t v_desc = VT ? tc::sw128_desc(tc::smem_u32(vring))
                                 : tc::sw128_desc_mn(tc::smem_u32(vring), BN * 128, 1024);
      bool ok = true;
      for (int j = 0; ok && j < nkb; ++j) {
        const int s = j % vstages;
        const int pb = NSB == 2 ? j % 2 : 0;  // P over S buffer j % 2, or the P columns
        const uint32_t tP = tmem + (NSB == 2 ? (uint32_t)(pb * BN) : P_COL);
        ok = all(tc::mbar_wait(&v_full[s], (uint32_t)(j / vstages) & 1u, abort_flag, status) &&
                 tc::mbar_wait(&p_full[pb], (uint32_t)(j / (NSB == 2 ? 2 : 1)) & 1u, abort_flag, status));
        if (!ok) break;
        tc::tc_fence_after();
        if (leader) {
          const uint64_t vd = v_desc + (uint64_t)(s * (VSLOT >> 4));
#pragma unroll
          for (int ks = 0; ks < BN / 16; ++ks) {
            const uint64_t db = VT ? vd + (uint64_t)((ks / 4) * ((BM * 128) >> 4) + (ks % 4) * 2)
                                   : vd + (uint64_t)(ks * ((16 * 128) >> 4));
            tc::umma_bf16_ts(tO, tP + (uint32_t)ks * 8, db, idO, (j > 0 || ks > 0) ? 1u : 0u);
          }
          tc::umma_commit(&pv_full[pb]);
          tc::umma_commit(&v_empty[s]);
        }
        __syncwarp();
      }
      if (!ok && leader) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(&drain[1]);
        if (!tc::mbar_wait_drain(&drain[1], 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else {
    softmax_sdb<BN, NSB, SPLIT, SUMC>(p, warp & 3, (warp - 4) >> 2, lane, q0, nkb, b, h, tmem, 0u, O_COL, P_COL, s_full,
                                s_free, p_full, pv_full, RowXchg{xch, xbar}, abort_flag, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, TMEM_COLS);
  }
}

// Two query tiles per CTA (TileSize M = 256) with 128-key blocks. The CTA
// holds the whole SM: TMEM columns [0, 128) and [128, 256) are S_0 and S_1
// (fp32), [256, 384) and [384, 512) are O_0 and O_1; P_t (bf16 pairs) is
// written over the first 64 columns of S_t. One thread issues every UMMA in
// the order P_0 V_{j-1}, S_0(j), P_1 V_{j-1}, S_1(j): while tile t's softmax
// works on S_t(j), the tensor core runs the other tile's P V and S products,
// and K_j and V_j are loaded once for both tiles.
//   warps 0..7 : softmax, one thread per query row; warp w serves tile w / 4,
//                TMEM lane quadrant w % 4
//   warp 8     : TMA producer of Q and of the K ring; owns TMEM
//   warp 9     : TMA producer of the V ring
//   warp 10    : the UMMA issue loop, run by all 32 lanes on warp-uniform
//                descriptors, one elected lane issuing (a lane-0 branch
//                spends far longer per UMMA forming its operands)
// S_t(j) overwrites the columns P_t(j-1) V_{j-1} read as its A operand; both
// are issued by the same thread, and tcgen05.mma operations of one thread
// execute in issue order. The commit that signals S_t(j) also covers
// P_t(j-1) V_{j-1}, so the softmax may rescale O_t as soon as S_t(j) is
// ready. One commit per iteration (it_done) releases both rings: K_j's slot
// after S_1(j), V_{j-1}'s after P_1 V_{j-1}. A tile's key blocks: every
// block up to its diagonal when causal (the second tile has one more than
// the first), all blocks otherwise; a tile with no query row inside the
// sequence takes none.
constexpr int kBN2q = 128;
constexpr int kVStages2q = 2;
constexpr int kItRing2q = 4;  // it_done barriers: more than the K (<= 3) and V (2) ring depths
constexpr int kThreads2q = 32 * 11;

// Bytes of dynamic shared memory: two query tiles, the K ring (the schedule's
// stages), a two-slot V ring, barriers (q_full, k_full[stages], v_full[2],
// it_done[4], s_full[2], p_full[2], o_full[2], drain), the TMEM address and
// abort flag, and 1 KB of alignment slack.
__host__ __device__ constexpr size_t attn2q_smem(int stages) {
  return (size_t)2 * BM * D * 2 + (size_t)(stages + kVStages2q) * kBN2q * D * 2 + (size_t)(14 + stages) * 8 + 8 + 1024;
}

// Adds the two bf16 halves of v to a and b in fp32 (mixed-precision adds of sm_100+).
__device__ __forceinline__ void acc_bf16x2(float& a, float& b, uint32_t v) {
  asm("{\n\t.reg .b16 lo, hi;\n\t"
      "mov.b32 {lo, hi}, %2;\n\t"
      "add.rn.f32.bf16 %0, lo, %0;\n\t"
      "add.rn.f32.bf16 %1, hi, %1;\n\t}"
      : "+f"(a), "+f"(b)
      : "r"(v));
}

// exp_pack_bf16 in place: the bf16 pair of scores i, i + 1 goes to r[i / 2],
// which has been read by then, so P needs no registers of its own. Four
// pairs per volatile block: the compiler keeps the blocks in order, so at
// most four pairs' exponents are live at once (hoisting every packed FMA
// ahead of the exponentials would need 64 more registers).
template <int N>
__device__ __forceinline__ void exp_pack_bf16_inplace(uint32_t* r, uint64_t sc2, uint64_t nm2) {
  static_assert(N % 8 == 0, "four pairs per block");
#pragma unroll
  for (int i = 0; i < N; i += 8) {
    uint32_t e0, e1, e2, e3;
    asm volatile(
        "{\n\t.reg .b64 x0, x1, x2, x3;\n\t.reg .f32 a0, b0, a1, b1, a2, b2, a3, b3;\n\t"
        ".reg .b32 c0, c1, c2, c3;\n\t"
        "mov.b64 x0, {%4, %5};\n\tmov.b64 x1, {%6, %7};\n\tmov.b64 x2, {%8, %9};\n\tmov.b64 x3, {%10, %11};\n\t"
        "fma.rn.f32x2 x0, x0, %12, %13;\n\tfma.rn.f32x2 x1, x1, %12, %13;\n\t"
        "fma.rn.f32x2 x2, x2, %12, %13;\n\tfma.rn.f32x2 x3, x3, %12, %13;\n\t"
        "mov.b64 {a0, b0}, x0;\n\tmov.b64 {a1, b1}, x1;\n\tmov.b64 {a2, b2}, x2;\n\tmov.b64 {a3, b3}, x3;\n\t"
        "cvt.rn.bf16x2.f32 c0, b0, a0;\n\tcvt.rn.bf16x2.f32 c1, b1, a1;\n\t"
        "cvt.rn.bf16x2.f32 c2, b2, a2;\n\tcvt.rn.bf16x2.f32 c3, b3, a3;\n\t"
        "ex2.approx.ftz.bf16x2 %0, c0;\n\tex2.approx.ftz.bf16x2 %1, c1;\n\t"
        "ex2.approx.ftz.bf16x2 %2, c2;\n\tex2.approx.ftz.bf16x2 %3, c3;\n\t}"
        : "=r"(e0), "=r"(e1), "=r"(e2), "=r"(e3)
        : "r"(r[i]), "r"(r[i + 1]), "r"(r[i + 2]), "r"(r[i + 3]), "r"(r[i + 4]), "r"(r[i + 5]), "r"(r[i + 6]),
          "r"(r[i + 7]), "l"(sc2), "l"(nm2));
    r[i / 2] = e0;
    r[i / 2 + 1] = e1;
    r[i / 2 + 2] = e2;
    r[i / 2 + 3] = e3;
  }
}

// Softmax of query tile t (of the two) for TMEM lane quadrant qd, one
// thread per query row: the block's 128 scores in registers, the row
// maximum, the exponentials packed to bf16 pairs in place and written over
// S_t as P_t, the row sum of those bf16 values in fp32, and O_t rescaled when
// the maximum has grown by more than 2^8.
__device__ __forceinline__ void softmax_2q(const Params& p, int t, int qd, int lane, int q0, int nk, int b, int h,
                                           uint32_t tmem, uint64_t* s_full, uint64_t* p_full, uint64_t* o_full,
                                           volatile int* abort_flag, volatile int* status) {
  constexpr int BN = kBN2q;
  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };
  const int row = 32 * qd + lane;
  const int qi = q0 + t * BM + row;
  const uint32_t lane_base = (uint32_t)(32 * qd) << 16;
  const uint32_t tS = tmem + lane_base + (uint32_t)(t * 128);
  const uint32_t tO = tmem + lane_base + 256u + (uint32_t)(t * 128);
  float m_ref = -INFINITY, l = 0.f;
  for (int j = 0; j < nk; ++j) {
    if (!tc::mbar_wait(&s_full[t], (uint32_t)j & 1u, abort_flag, status)) {
      if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
      return;
    }
    tc::tc_fence_after();
    uint32_t r[BN];
#pragma unroll
    for (int c = 0; c < BN; c += 32) tc::tmem_ld32(tS + (uint32_t)c, *reinterpret_cast<uint32_t(*)[32]>(&r[c]));
    tc::tmem_ld_wait();
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
    const float mref = m_ref == -INFINITY ? 0.f : m_ref;
    const uint64_t sc2 = f2(p.scale_log2, p.scale_log2), nm2 = f2(-mref, -mref);
    float ls0 = 0.f, ls1 = 0.f, ls2 = 0.f, ls3 = 0.f;
#pragma unroll
    for (int hf = 0; hf < BN / 64; ++hf) {
      uint32_t* pk = r + hf * 64;  // the 32 bf16 pairs of scores [hf * 64, + 64), packed in place
      exp_pack_bf16_inplace<64>(pk, sc2, nm2);
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        acc_bf16x2(ls0, ls1, pk[i]);
        acc_bf16x2(ls2, ls3, pk[i + 1]);
      }
      // P_t(j) over S_t(j), whose scores are in registers
      tc::tmem_st32(tS + (uint32_t)(hf * 32), *reinterpret_cast<uint32_t(*)[32]>(pk));
    }
    l = l * factor + ((ls0 + ls1) + (ls2 + ls3));
    if (__any_sync(0xffffffffu, factor != 1.f)) {
      // O_t holds P_t V up to block j - 1 (complete: its UMMAs precede S_t(j)); rescaled here,
      // with the scores no longer live, before P_t V_j is released
#pragma unroll 1
      for (int c = 0; c < D; c += 32) {
        uint32_t o[32];
        tc::tmem_ld32(tO + (uint32_t)c, o);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * factor);
        tc::tmem_st32(tO + (uint32_t)c, o);
      }
    }
    tc::tmem_st_wait();
    tc::tc_fence_before();
    tc::mbar_arrive(&p_full[t]);
  }
  if (nk == 0) return;
  if (tc::mbar_wait(&o_full[t], 0, abort_flag, status)) {
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

template <bool VT>
__global__ void __launch_bounds__(kThreads2q, 1)
    attn2q_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, const Params p, const int stages) {
  constexpr int BN = kBN2q;
  constexpr int VS = kVStages2q;
  constexpr int QT = BM * D * 2;  // one query tile: two [128][64] swizzled halves
  constexpr int KV = BN * D * 2;  // one K or V tile
  constexpr int W_K = 8, W_V = 9, W_MMA = 10;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;
  uint8_t* kring = sQ + 2 * QT;
  uint8_t* vring = kring + (size_t)stages * KV;
  uint64_t* q_full = (uint64_t*)(vring + (size_t)VS * KV);
  uint64_t* k_full = q_full + 1;       // [stages]
  uint64_t* v_full = k_full + stages;  // [VS]
  uint64_t* it_done = v_full + VS;     // [kItRing2q]
  uint64_t* s_full = it_done + kItRing2q;  // [2] per tile
  uint64_t* p_full = s_full + 2;           // [2]
  uint64_t* o_full = p_full + 2;           // [2]
  uint64_t* drain = o_full + 2;
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
  const int q0 = qb * 2 * BM;
  auto blocks_of = [&](int t) {
    const int r0 = q0 + t * BM;
    const int kv_end = p.causal ? min(r0 + BM, p.S) : p.S;
    return r0 < p.S ? (kv_end + BN - 1) / BN : 0;
  };
  const int nkb0 = blocks_of(0), nkb1 = blocks_of(1);
  const int NK = max(nkb0, nkb1);

  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    tc::mbar_init(q_full, 1);
    for (int s = 0; s < stages; ++s) tc::mbar_init(&k_full[s], 1);
    for (int s = 0; s < VS; ++s) tc::mbar_init(&v_full[s], 1);
    for (int i = 0; i < kItRing2q; ++i) tc::mbar_init(&it_done[i], 1);
    for (int t = 0; t < 2; ++t) {
      tc::mbar_init(&s_full[t], 1);
      tc::mbar_init(&p_full[t], 128);
      tc::mbar_init(&o_full[t], 1);
    }
    tc::mbar_init(drain, 1);
    *abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == W_K) tc::tmem_alloc(tmem_slot, 512);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Block j goes into slot j % depth once iteration j - depth + lag has completed (that
  // iteration issued the last UMMA reading the slot's previous block: K lag 0, V lag 1).
  // A producer is never a full it_done ring behind: the UMMA issuer cannot finish
  // iteration i + kItRing2q before this producer has loaded a block that iteration reads.
  auto produce = [&](uint64_t* full, int depth, int lag, auto load) {
    int j = 0;
    for (; j < NK; ++j) {
      if (j >= depth) {
        const int it = j - depth + lag;
        if (!tc::mbar_wait(&it_done[it % kItRing2q], (uint32_t)(it / kItRing2q) & 1u, abort_flag, status)) {
          fail(RC_DEV_TIMEOUT_EMPTY);
          break;
        }
      }
      const int s = j % depth;
      tc::mbar_expect_tx(&full[s], KV);
      load(s, j, &full[s]);
    }
    for (int i = max(0, j - depth); i < j; ++i)
      if (!tc::mbar_wait_drain(&full[i % depth], (uint32_t)(i / depth) & 1u)) fail(RC_DEV_TIMEOUT_DRAIN);
  };

  if (warp == W_K) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmK);
      tc::mbar_expect_tx(q_full, (uint32_t)(((nkb0 > 0) + (nkb1 > 0)) * QT));
      for (int t = 0; t < 2; ++t) {
        if ((t == 0 ? nkb0 : nkb1) == 0) continue;
        const int qrow = b * p.S + q0 + t * BM;
        tc::tma_load_2d(sQ + t * QT, &tmQ, q_full, h * D, qrow);
        tc::tma_load_2d(sQ + t * QT + QT / 2, &tmQ, q_full, h * D + 64, qrow);
      }
      produce(k_full, stages, 0, [&](int s, int j, uint64_t* bar) {
        uint8_t* sk = kring + (size_t)s * KV;
        const int krow = b * p.S + j * BN;
        tc::tma_load_2d(sk, &tmK, bar, g * D, krow);
        tc::tma_load_2d(sk + BN * 128, &tmK, bar, g * D + 64, krow);
      });
      if (!tc::mbar_wait_drain(q_full, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp == W_V) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmV);
      produce(v_full, VS, 1, [&](int s, int j, uint64_t* bar) {
        uint8_t* sv = vring + (size_t)s * KV;
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
    __syncwarp();
  } else if (warp == W_MMA) {
    const bool leader = tc::elect_one();
    constexpr uint32_t idS = tc::idesc_bf16_f32(BM, BN);
    constexpr uint32_t idO = tc::idesc_bf16_f32(BM, D, !VT);
    // Descriptors of Q_0, the first K slot and the first V slot. Q_1, a ring slot and each
    // 16-wide K step add a constant to the 14-bit start-address field (addresses below
    // 256 KB: no carry out of it).
    const uint64_t q_desc = tc::sw128_desc(tc::smem_u32(sQ));
    const uint64_t k_desc = tc::sw128_desc(tc::smem_u32(kring));
    const uint64_t v_desc =
        VT ? tc::sw128_desc(tc::smem_u32(vring)) : tc::sw128_desc_mn(tc::smem_u32(vring), BN * 128, 1024);
    auto all = [](bool x) { return __all_sync(0xffffffffu, x); };
    bool ok = all(tc::mbar_wait(q_full, 0, abort_flag, status));
    // iteration j: P_t V_{j-1} then S_t(j) for t = 0, 1 (each where the tile has that block)
    for (int j = 0; ok && j <= NK; ++j) {
      const int jj = j - 1;
      bool v_ready = false, k_ready = false;
#pragma unroll
      for (int t = 0; t < 2; ++t) {
        const int nk = t == 0 ? nkb0 : nkb1;
        if (ok && jj >= 0 && jj < nk) {
          if (!v_ready) {
            ok = all(tc::mbar_wait(&v_full[jj % VS], (uint32_t)(jj / VS) & 1u, abort_flag, status));
            v_ready = true;
          }
          ok = ok && all(tc::mbar_wait(&p_full[t], (uint32_t)jj & 1u, abort_flag, status));
          if (ok) {
            tc::tc_fence_after();
            if (leader) {
              const uint64_t vd = v_desc + (uint64_t)((jj % VS) * (KV >> 4));
              const uint32_t tP = tmem + (uint32_t)(t * 128), tO = tmem + 256u + (uint32_t)(t * 128);
#pragma unroll
              for (int ks = 0; ks < BN / 16; ++ks) {
                const uint64_t db = VT ? vd + (uint64_t)((ks / 4) * ((BM * 128) >> 4) + (ks % 4) * 2)
                                       : vd + (uint64_t)(ks * ((16 * 128) >> 4));
                tc::umma_bf16_ts(tO, tP + (uint32_t)ks * 8, db, idO, (jj > 0 || ks > 0) ? 1u : 0u);
              }
              if (jj == nk - 1) tc::umma_commit(&o_full[t]);
            }
            __syncwarp();
          }
        }
        if (ok && j < nk) {
          if (!k_ready) {
            ok = all(tc::mbar_wait(&k_full[j % stages], (uint32_t)(j / stages) & 1u, abort_flag, status));
            k_ready = true;
            if (ok) tc::tc_fence_after();
          }
          if (ok) {
            if (leader) {
              const uint64_t kd = k_desc + (uint64_t)((j % stages) * (KV >> 4));
              const uint64_t qd = q_desc + (uint64_t)(t * (QT >> 4));
              const uint32_t tS = tmem + (uint32_t)(t * 128);
#pragma unroll
              for (int ks = 0; ks < D / 16; ++ks) {
                const uint64_t off = (uint64_t)((ks / 4) * ((BM * 128) >> 4) + (ks % 4) * 2);
                tc::umma_bf16(tS, qd + off, kd + off, idS, ks > 0 ? 1u : 0u);
              }
              tc::umma_commit(&s_full[t]);
            }
            __syncwarp();
          }
        }
      }
      if (ok) {
        if (leader) tc::umma_commit(&it_done[j % kItRing2q]);
        __syncwarp();
      }
    }
    if (!ok) {
      if (leader) {
        fail(RC_DEV_TIMEOUT_FULL);
        tc::umma_commit(drain);
        if (!tc::mbar_wait_drain(drain, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
      __syncwarp();
    }
  } else {
    const int t = warp / 4;
    softmax_2q(p, t, warp & 3, lane, q0, t == 0 ? nkb0 : nkb1, b, h, tmem, s_full, p_full, o_full, abort_flag, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == W_K) {
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

// P0 kernel: Q tile + K/V ring + P tile + 1 KB alignment slack + barriers
// (1 + 2 * stages + 4 of them, 8 B each, plus two words: 512 B for stages <= 5)
size_t smem_bytes(int bn, int stages) {
  return (size_t)BM * D * 2 + (size_t)stages * 2 * bn * D * 2 + (size_t)BM * bn * 2 + 1024 + 512;
}

template <typename Kern>
rc_status smem_attributes(Kern kern, bool& done) {
  if (done) return RC_OK;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
  // the largest shared-memory carve-out, so that two one-tile CTAs can share an SM
  if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "attention: smem attribute: %s", cudaGetErrorString(e));
  done = true;
  return RC_OK;
}

// Tensor maps and kernel parameters shared by both kernel families.
template <int BN, bool VT>
rc_status prepare(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V, void* O,
                  float* lse, const LaunchCtx& c, CUtensorMap* tq, CUtensorMap* tk, CUtensorMap* tv, Params* p) {
  const uint64_t BS = (uint64_t)d.batch * d.seq;
  RC_TRY(tcg::encode_2d(tq, Q, (uint64_t)d.heads_q * D, BS, BM));
  RC_TRY(tcg::encode_2d(tk, K, (uint64_t)d.heads_kv * D, BS, BN));
  if (VT)
    RC_TRY(tcg::encode_2d(tv, V, (uint64_t)d.seq, (uint64_t)d.batch * d.heads_kv * D, BM));
  else
    RC_TRY(tcg::encode_2d(tv, V, (uint64_t)d.heads_kv * D, BS, BN));
  memset(p, 0, sizeof *p);
  p->B = (int)d.batch;
  p->S = (int)d.seq;
  p->Hq = (int)d.heads_q;
  p->Hkv = (int)d.heads_kv;
  p->group = (int)(d.heads_q / d.heads_kv);
  p->q_blocks = (int)((d.seq + BM - 1) / BM);
  p->causal = d.causal ? 1 : 0;
  p->scale_log2 = (float)(d.scale * 1.4426950408889634);
  p->raster = k.raster;
  p->O = (__nv_bfloat16*)O;
  p->lse = lse;
  p->status = c.status;
  if ((long long)p->B * p->Hq * p->q_blocks > 0x7fffffffLL) return rc_fail(RC_ERR_UNSUPPORTED_OP, "attention: grid too large");
  return RC_OK;
}

template <typename Kern>
rc_status launched(Kern kern, int threads, size_t smem) {
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) return RC_OK;
  cudaFuncAttributes fa;
  memset(&fa, 0, sizeof fa);
  cudaFuncGetAttributes(&fa, kern);
  return rc_fail(RC_ERR_CUDA,
                 "attention launch: %s (%d threads, %zu B dynamic shared memory; kernel: %d registers, %zu B static "
                 "and at most %d B dynamic shared memory, at most %d threads)",
                 cudaGetErrorString(e), threads, smem, fa.numRegs, fa.sharedSizeBytes, fa.maxDynamicSharedSizeBytes,
                 fa.maxThreadsPerBlock);
}

// The P0 kernel: one UMMA-issuing warp, P in shared memory.
template <int BN, bool VT>
rc_status launch_basic(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V, void* O,
                       float* lse, const LaunchCtx& c) {
  auto kern = attn_kernel<BN, VT>;
  static bool attr = false;
  RC_TRY(smem_attributes(kern, attr));
  CUtensorMap tq, tk, tv;
  Params p;
  RC_TRY((prepare<BN, VT>(k, d, Q, K, V, O, lse, c, &tq, &tk, &tv, &p)));
  const size_t smem = smem_bytes(BN, k.stages);
  kern<<<(unsigned)(p.B * p.Hq * p.q_blocks), kThreads, smem, (cudaStream_t)c.stream>>>(tq, tk, tv, p, k.stages);
  return launched(kern, kThreads, smem);
}

// The split-issue kernel: NSB S buffers, SPLIT softmax threads per row, row sums on the tensor core.
template <int BN, bool VT, int NSB, int SPLIT, bool SUMC>
rc_status launch_split(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V, void* O,
                       float* lse, const LaunchCtx& c) {
  auto kern = attn4_kernel<BN, VT, NSB, SPLIT, SUMC>;
  static bool attr = false;
  RC_TRY(smem_attributes(kern, attr));
  CUtensorMap tq, tk, tv;
  Params p;
  RC_TRY((prepare<BN, VT>(k, d, Q, K, V, O, lse, c, &tq, &tk, &tv, &p)));
  const size_t smem = attn4_smem<BN, NSB, SPLIT, SUMC>(k.stages);
  constexpr int threads = attn4_threads<SPLIT>();
  kern<<<(unsigned)(p.B * p.Hq * p.q_blocks), threads, smem, (cudaStream_t)c.stream>>>(tq, tk, tv, p, k.stages);
  return launched(kern, threads, smem);
}

// The two-query-tile kernel (TileSize M = 256): 128-key blocks, one CTA per SM.
template <bool VT>
rc_status launch_2q(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V, void* O,
                    float* lse, const LaunchCtx& c) {
  auto kern = attn2q_kernel<VT>;
  static bool attr = false;
  RC_TRY(smem_attributes(kern, attr));
  CUtensorMap tq, tk, tv;
  Params p;
  RC_TRY((prepare<kBN2q, VT>(k, d, Q, K, V, O, lse, c, &tq, &tk, &tv, &p)));
  p.q_blocks = (int)((d.seq + 2 * BM - 1) / (2 * BM));
  const size_t smem = attn2q_smem(k.stages);
  kern<<<(unsigned)(p.B * p.Hq * p.q_blocks), kThreads2q, smem, (cudaStream_t)c.stream>>>(tq, tk, tv, p, k.stages);
  return launched(kern, kThreads2q, smem);
}

template <int BN, bool VT>
rc_status dispatch(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V, void* O,
                   float* lse, const LaunchCtx& c) {
  if (k.persistent == 0) return launch_basic<BN, VT>(k, d, Q, K, V, O, lse, c);
  const bool two_sb = k.unroll == 2, split = k.persistent == 2;
  if (k.location == 2) {
    if constexpr (!VT) {
      if (two_sb) return split ? launch_split<BN, false, 2, 2, true>(k, d, Q, K, V, O, lse, c)
                               : launch_split<BN, false, 2, 1, true>(k, d, Q, K, V, O, lse, c);
      return split ? launch_split<BN, false, 1, 2, true>(k, d, Q, K, V, O, lse, c)
                   : launch_split<BN, false, 1, 1, true>(k, d, Q, K, V, O, lse, c);
    }
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: row sums on the tensor core need V as given");
  }
  if (two_sb) return split ? launch_split<BN, VT, 2, 2, false>(k, d, Q, K, V, O, lse, c)
                           : launch_split<BN, VT, 2, 1, false>(k, d, Q, K, V, O, lse, c);
  return split ? launch_split<BN, VT, 1, 2, false>(k, d, Q, K, V, O, lse, c)
               : launch_split<BN, VT, 1, 1, false>(k, d, Q, K, V, O, lse, c);
}

}  // namespace attn

rc_status rc_launch_attention(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K, const void* V,
                              void* O, float* lse, void* workspace, const LaunchCtx& c) {
  if (d.head_dim != attn::D) return rc_fail(RC_ERR_UNSUPPORTED_OP, "attention: head_dim must be 128");
  if (d.batch * d.seq > 0x7fffffffLL) return rc_fail(RC_ERR_UNSUPPORTED_OP, "attention: B*S too large");
  // the same rules as the schedule legality check, so a launch never gets a kernel it cannot run
  if ((k.tile_m != attn::BM && k.tile_m != 2 * attn::BM) || k.raster > 1 || (k.tile_n != 64 && k.tile_n != 128))
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: 128- or 256-row query tiles, 64- or 128-key blocks, loop order 0 or 1");
  if (k.tile_m == 2 * attn::BM && (k.tile_n != attn::kBN2q || k.persistent != 1 || k.location != 1 || k.unroll != 1 ||
                                   k.stages < 1 || k.stages > 3))
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE,
                   "attention: two query tiles per CTA take 128-key blocks, P in tensor memory, one S buffer per tile, "
                   "one softmax thread per row and 1 to 3 K stages");
  if (k.persistent == 0 && (k.location != 0 || k.unroll != 1))
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: one issuing warp keeps P in shared memory, one S buffer");
  if (k.persistent > 0 && k.location == 0)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: split UMMA issue keeps P in TMEM");
  if (k.location == 2 && k.layout != 0)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "attention: row sums on the tensor core need V as given");
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
  if (k.tile_m == 2 * attn::BM)
    return vt ? attn::launch_2q<true>(k, d, Q, K, Vuse, O, lse, c) : attn::launch_2q<false>(k, d, Q, K, Vuse, O, lse, c);
  if (k.tile_n == 64)
    return vt ? attn::dispatch<64, true>(k, d, Q, K, Vuse, O, lse, c) : attn::dispatch<64, false>(k, d, Q, K, Vuse, O, lse, c);
  return vt ? attn::dispatch<128, true>(k, d, Q, K, Vuse, O, lse, c) : attn::dispatch<128, false>(k, d, Q, K, Vuse, O, lse, c);
}
