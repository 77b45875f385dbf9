// Tensor-core GEMM family for sm_103a: D = A B^T, A[M][K] and B[N][K] bf16
// K-major, fp32 accumulation in tensor memory (TMEM).
//
// One CTA computes one 128 x BN output tile (cta_group::1, UMMA M = 128):
//   warp 0     : TMA producer. One elected thread streams 128 x 64 A tiles and
//                BN x 64 B tiles (128-byte swizzle) into a ring of `stages`
//                shared-memory buffers, one or two such 64-wide K sub-blocks
//                per stage (TileSize K = 64 or 128), signalling a "full"
//                mbarrier per stage.
//   warp 1     : allocates TMEM; the whole warp runs the issue loop on
//                warp-uniform values and one lane (elect.sync) issues 4 UMMAs
//                (K = 16 each) per sub-block, releasing the stage through
//                tcgen05.commit onto its "empty" mbarrier; a final commit
//                signals the accumulator.
// Both control threads keep their ring slot, phase and (for convolutions)
// filter-tap position in counters: a single thread runs dependent integer
// code at a few cycles per instruction, so a division per k-block costs about
// as much as the k-block's UMMAs. A stage of two sub-blocks halves the barrier
// waits and commits per UMMA.
//   warps 2..5 : epilogue. Warp w reads TMEM lanes 32*(w%4) .. +31 with
//                tcgen05.ld (one output row per thread), applies the fused
//                epilogue and stores 16-byte vectors.
//
// Schedule knobs that select variants here: the N tile (template BN), the
// K sub-blocks per stage (runtime `ksub`), the ring depth (runtime
// `stages`), split-K (work items), tile raster order and
// group (runtime), and the fused epilogue (template EPI). The A operand is a
// plain matrix or, for convolutions, an implicit im2col view loaded with a
// 4-D TMA box whose out-of-range coordinates are zero-filled (the padding).
// Grouped mode (MoE) partitions A's rows into segments with their own B; its
// A rows may also be gathered from a source matrix by a row map inside the
// producer (TC_A_GATHER), which then uses the whole warp 0: each lane copies
// 16-byte chunks of 32 rows with cp.async, applying the 128-byte swizzle
// itself, and has the stage's "full" barrier count an arrival of its own once
// those copies land (cp.async.mbarrier.arrive); lane 0 still loads B by TMA.
// The MMA thread fences the generic-proxy copies for the tensor cores (async
// proxy) after the barrier wait.
#pragma once

#include <cstring>

#include "rc_internal.h"
#include "tc_common.cuh"

namespace tcg {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int kThreads = 192;

struct Params {
  int M, N, K;          // N: UMMA columns of the whole problem (2I for SwiGLU)
  int tiles_m, tiles_n;
  int kb_total, kb_per;
  int raster, group;
  void* D;
  long long ldd;
  const __nv_bfloat16* bias;
  int silu;
  int swiglu_I;         // SwiGLU: output width I (also the offset of the up rows)
  int out_cols;         // columns of D that exist (store bound)
  // implicit-GEMM convolution (pad = coordinate shift of the filter taps;
  // pad_rows = border width of an explicitly padded input)
  int img_hw, img_w, cblocks, ks, pad, pad_rows;
  // grouped rows (MoE)
  const int* offsets;
  int groups;
  int b_group_rows;
  int seg_mode;  // which rows of each segment: TcSegMode (all, the pair part, the short remainder)
  const float* row_scale;
  const int* row_map;
  int row_div;
  const __nv_bfloat16* a_src;  // TC_A_GATHER: source rows [..][K]
  int* status;
  int persistent;       // 1: grid-stride loop over tiles with two TMEM accumulators
  int splits;           // split-K factor (work items = tiles x splits)
  int ksub;             // 64-wide K sub-blocks per ring stage (1 or 2)
  const __nv_bfloat16* resid;  // STORE_BF16: residual [M][ldd] added before the rounding (NULL = none)
};

// Linear CTA index -> (m tile, n tile) under the raster order knob.
template <class P>
__device__ __forceinline__ void map_tile(const P& p, int t, int& mt, int& nt) {
  const int G = p.group;
  if (p.raster == 0) {  // M fastest within bands of G n-tiles
    const int band = t / (p.tiles_m * G), in = t - band * p.tiles_m * G;
    const int gw = min(G, p.tiles_n - band * G);
    mt = in / gw;
    nt = band * G + (in - (in / gw) * gw);
  } else {  // N fastest within bands of G m-tiles
    const int band = t / (p.tiles_n * G), in = t - band * p.tiles_n * G;
    const int gh = min(G, p.tiles_m - band * G);
    nt = in / gh;
    mt = band * G + (in - (in / gh) * gh);
  }
}

union Pack8 {
  uint4 u;
  __nv_bfloat162 h2[4];
};

__device__ __forceinline__ uint4 pack8(const float* v) {
  Pack8 p;
#pragma unroll
  for (int i = 0; i < 4; ++i) p.h2[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
  return p.u;
}

// Row pitch of an epilogue warp's staging area: BN bf16 plus 16 bytes, an odd number of 16-byte
// chunks (BN % 16 == 0), so that eight consecutive rows' chunks c fall on distinct bank groups.
template <int BN>
constexpr int stage_pitch() {
  return 2 * BN + 16;
}

// sbias: this warp's copy of the tile's bias (fp32, BN values; BIAS_SILU only). stage: NULL, or
// this warp's 32 x stage_pitch<BN>() bytes of idle operand ring (the plain bf16 store): the rows
// are converted into it, then stored as runs of whole rows, so that a warp store covers 512
// contiguous bytes instead of 16 bytes in each of 32 rows.
template <int BN, int EPI>
__device__ __forceinline__ void epilogue(const Params& p, uint32_t taddr, int r, int row_end, int nt, int split,
                                         bool have_acc, const float* sbias, uint8_t* stage = nullptr) {
  const bool row_ok = r < row_end;
  if constexpr (EPI == TC_EPI_SWIGLU) {
    constexpr int HALF = BN / 2;
    __nv_bfloat16* out = (__nv_bfloat16*)p.D + (long long)r * p.ldd;
    const int n0 = nt * HALF;
    // 16 columns per step, software-pipelined: the next step's TMEM loads are issued before this
    // step's math and stores, and waited for at the top of the next step
    uint32_t g[2][16], u[2][16];
    tc::tmem_ld16(taddr, g[0]);
    tc::tmem_ld16(taddr + HALF, u[0]);
#pragma unroll
    for (int c = 0; c < HALF; c += 16) {
      const int b = (c / 16) & 1;
      tc::tmem_ld_wait(g[b]);
      tc::tmem_ld_wait(u[b]);
      if (c + 16 < HALF) {
        tc::tmem_ld16(taddr + c + 16, g[b ^ 1]);
        tc::tmem_ld16(taddr + HALF + c + 16, u[b ^ 1]);
      }
      float v[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const float gv = have_acc ? __uint_as_float(g[b][j]) : 0.f;
        const float uv = have_acc ? __uint_as_float(u[b][j]) : 0.f;
        v[j] = tc::silu(gv) * uv;
      }
      const int col = n0 + c;
      if (row_ok) {
        if (col < p.out_cols) *reinterpret_cast<uint4*>(out + col) = pack8(v);
        if (col + 8 < p.out_cols) *reinterpret_cast<uint4*>(out + col + 8) = pack8(v + 8);
      }
    }
  } else {
    const int n0 = nt * BN;
    // MoE combine: the routed slot of this row and its weight, once per tile
    long long orow = 0;
    float scale = 0.f;
    if constexpr (EPI == TC_EPI_SCALE_ATOMIC) {
      if (row_ok) {
        const int slot = p.row_map[r];
        scale = p.row_scale[slot];
        orow = slot / p.row_div;
      }
    }
    // 16 columns per step, software-pipelined as in the SwiGLU epilogue
    uint32_t a[2][16];
    tc::tmem_ld16(taddr, a[0]);
#pragma unroll
    for (int c = 0; c < BN; c += 16) {
      const int b = (c / 16) & 1;
      const int col = n0 + c;
      tc::tmem_ld_wait(a[b]);
      if (c + 16 < BN) tc::tmem_ld16(taddr + c + 16, a[b ^ 1]);
      float v[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] = have_acc ? __uint_as_float(a[b][j]) : 0.f;
      if (!row_ok) continue;
      if constexpr (EPI == TC_EPI_STORE_BF16 || EPI == TC_EPI_BIAS_SILU) {
        if constexpr (EPI == TC_EPI_BIAS_SILU) {
          float bv[16];
#pragma unroll
          for (int j = 0; j < 16; j += 4) *reinterpret_cast<float4*>(&bv[j]) = *reinterpret_cast<const float4*>(&sbias[c + j]);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float x = v[j] + bv[j];
            v[j] = p.silu ? tc::silu(x) : x;
          }
        }
        if constexpr (EPI == TC_EPI_STORE_BF16) {
          if (p.resid) {  // residual connection: D = bf16(acc + resid), one rounding
            const __nv_bfloat16* rr = p.resid + (long long)r * p.ldd + col;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              if (col + 8 * h >= p.out_cols) break;
              union {
                uint4 u;
                __nv_bfloat162 b2[4];
              } x;
              x.u = *reinterpret_cast<const uint4*>(rr + 8 * h);
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const float2 f = __bfloat1622float2(x.b2[q]);
                v[8 * h + 2 * q] += f.x;
                v[8 * h + 2 * q + 1] += f.y;
              }
            }
          }
        }
        if (stage) {
          uint8_t* srow = stage + (threadIdx.x & 31) * stage_pitch<BN>() + c * 2;
          *reinterpret_cast<uint4*>(srow) = pack8(v);
          *reinterpret_cast<uint4*>(srow + 16) = pack8(v + 8);
        } else {
          __nv_bfloat16* out = (__nv_bfloat16*)p.D + (long long)r * p.ldd;
          if (col < p.out_cols) *reinterpret_cast<uint4*>(out + col) = pack8(v);
          if (col + 8 < p.out_cols) *reinterpret_cast<uint4*>(out + col + 8) = pack8(v + 8);
        }
      } else if constexpr (EPI == TC_EPI_PARTIAL_F32) {
        float* out = (float*)p.D + (long long)split * p.M * p.ldd + (long long)r * p.ldd;
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (col + 4 * q < p.out_cols)
            *reinterpret_cast<float4*>(out + col + 4 * q) = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      } else if constexpr (EPI == TC_EPI_SCALE_ATOMIC) {
        const float s = scale;
        float* out = (float*)p.D + orow * p.ldd;
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (col + 4 * q < p.out_cols)
            atomicAdd(reinterpret_cast<float4*>(out + col + 4 * q),
                      make_float4(s * v[4 * q], s * v[4 * q + 1], s * v[4 * q + 2], s * v[4 * q + 3]));
      }
    }
    if constexpr (EPI == TC_EPI_STORE_BF16) {
      if (stage) {  // the warp's 32 rows, 16-byte chunks in row order: lane l takes chunks l, l + 32, ...
        __syncwarp();
        constexpr int NCH = BN / 8;
        const int ln = threadIdx.x & 31, row0 = r - ln;
#pragma unroll 4
        for (int qc = ln; qc < 32 * NCH; qc += 32) {
          const int rr = qc / NCH, ch = qc - rr * NCH;
          const int row = row0 + rr, col = n0 + ch * 8;
          if (row < row_end && col < p.out_cols)
            *reinterpret_cast<uint4*>((__nv_bfloat16*)p.D + (long long)row * p.ldd + col) =
                *reinterpret_cast<const uint4*>(stage + rr * stage_pitch<BN>() + ch * 16);
        }
      }
    }
  }
}

// Work item -> (A rows, B rows, n tile, split, k-block range). Grouped mode
// maps the m tile onto the segment that owns it; `valid` is false for the
// spare m tiles launched beyond what the segments need.
struct Item {
  bool valid;
  int row0, row_end, brow0, nt, split, kb0, nkb;
};

// Grouped mode keeps, per CTA, the segment row ranges and the exclusive
// prefix of the segments' tile counts in shared memory (at most kSmemGroups
// segments, checked on the host), built once by one warp at CTA start, so
// that resolving an m tile is a binary search in shared memory instead of a
// scan over every segment in global memory (2.6 us per CTA for 64 segments).
constexpr int kSmemGroups = 256;
constexpr int kGroupTableBytes = 3 * (kSmemGroups + 1) * 4 + 8;

// Rows [lo, hi) of a segment of rows [s_lo, s_hi) that a grouped launch covers.
// TC_SEG_ALL: all of them. With kSegSplit-row CTA-pair tiles a segment whose
// last tile would hold 1 .. kSegSplit / 2 rows is split: TC_SEG_PAIRS takes
// everything before that remainder (whole pair tiles, or a last pair tile
// more than half full), TC_SEG_REST takes the remainder alone (one 128-row
// tile), so the padding of a ragged segment is at most 127 rows, not 255.
constexpr int kSegSplit = 256;
__device__ __forceinline__ void seg_rows(int mode, int s_lo, int s_hi, int& lo, int& hi) {
  const int rem = (s_hi - s_lo) % kSegSplit;
  const int rest = rem > 0 && rem <= kSegSplit / 2 ? rem : 0;
  lo = mode == TC_SEG_REST ? s_hi - rest : s_lo;
  hi = mode == TC_SEG_PAIRS ? s_hi - rest : s_hi;
}

// TR: rows of a tile (128, or 256 for a CTA pair). One warp, all lanes.
template <int TR>
__device__ __forceinline__ void build_group_table(const Params& p, int lane, int* s_goff, int* s_gend, int* s_gtile) {
  const int G = p.groups;
  const int per = (G + 31) / 32;  // segments per lane, lane-major
  const int g0 = min(G, lane * per), g1 = min(G, g0 + per);
  int sum = 0;
  for (int g = g0; g < g1; ++g) {
    int lo, hi;
    seg_rows(p.seg_mode, p.offsets[g], p.offsets[g + 1], lo, hi);
    s_goff[g] = lo;
    s_gend[g] = hi;
    sum += (hi - lo + TR - 1) / TR;
  }
  int incl = sum;  // inclusive scan of the lanes' tile counts
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, d);
    if (lane >= d) incl += v;
  }
  int acc = incl - sum;
  for (int g = g0; g < g1; ++g) {
    s_gtile[g] = acc;
    acc += (s_gend[g] - s_goff[g] + TR - 1) / TR;
  }
  if (lane == 31) s_gtile[G] = incl;
}

template <bool GROUPED, int TR>
__device__ __forceinline__ Item resolve_item(const Params& p, long long w, const int* s_goff, const int* s_gend,
                                             const int* s_gtile) {
  Item it;
  const long long tiles = (long long)p.tiles_m * p.tiles_n;
  it.split = (int)(w / tiles);
  int mt;
  map_tile(p, (int)(w - (long long)it.split * tiles), mt, it.nt);
  it.valid = true;
  it.brow0 = 0;
  if constexpr (GROUPED) {
    int g = 0;
    it.valid = false;
    // last segment whose first tile is <= mt (empty segments share their successor's start)
    if (mt < s_gtile[p.groups]) {
      int lo = 0, hi = p.groups - 1;
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (s_gtile[mid] <= mt)
          lo = mid;
        else
          hi = mid - 1;
      }
      g = lo;
      it.row0 = s_goff[g] + (mt - s_gtile[g]) * TR;
      it.row_end = s_gend[g];
      it.valid = true;
    }
    it.brow0 = g * p.b_group_rows;
  } else {
    it.row0 = mt * TR;
    it.row_end = p.M;
  }
  it.kb0 = it.split * p.kb_per;
  it.nkb = max(0, min(p.kb_total, it.kb0 + p.kb_per) - it.kb0);
  return it;
}

// PAIR (TileSize M = 256): a cluster of two CTAs computes a 256 x BN tile
// with cta_group::2 UMMAs. Each CTA loads its own 128 rows of A and half of
// the B tile (rows [0, BN/2) in the leader, [BN/2, BN) in the peer; for the
// fused SwiGLU the gate rows and the up rows), and both CTAs' copies complete
// on the leader's "full" barrier. The leader's MMA thread issues M = 256
// UMMAs and multicasts its commits to both CTAs' "empty" and "accumulator
// full" barriers; each CTA's epilogue drains its own TMEM rows and arrives
// on the leader's "accumulator empty" barrier (one arrival per warp).
//
// MC > 1 (TileSize M = 128 MC): a cluster of MC CTAs along M computes MC
// consecutive 128 x BN tiles of one N tile with cta_group::1 UMMAs. They
// need the same B tile, so each CTA loads 1 / MC of its rows and multicasts
// them into every CTA of the cluster: B is read from L2 once per cluster
// instead of once per CTA. A stage of a CTA is overwritten by its peers'
// copies, so every CTA's MMA thread releases a stage into all the cluster's
// "empty" barriers (a multicast commit; each counts MC arrivals) and a
// producer refills a stage only once every CTA has released it.
template <int BN, int EPI, int AMODE, bool GROUPED, bool PAIR = false, int MC = 1>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const Params p,
                const int stages) {
  constexpr int A_BYTES = BM * BK * 2;                    // one 64-wide K sub-block of A
  constexpr int B_BYTES = (PAIR ? BN / 2 : BN) * BK * 2;  // and this CTA's rows of B
  constexpr uint32_t ACC_COLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  constexpr bool CLUSTER = PAIR || MC > 1;
  static_assert(B_BYTES % 1024 == 0, "B tile must keep stage buffers 1024-byte aligned");
  static_assert(MC == 1 || MC == 2 || MC == 4 || MC == 8, "cluster size");
  static_assert(MC == 1 || (!PAIR && !GROUPED && EPI != TC_EPI_SWIGLU && AMODE != TC_A_GATHER &&
                            (BN / MC) % 8 == 0),
                "B multicast: one-CTA tiles of a dense or convolution GEMM, 8-row swizzle atoms per slice");
  constexpr uint16_t MC_MASK = (uint16_t)((1u << MC) - 1u);
  // stage layout: A sub-blocks [0, ksub), then B sub-blocks [0, ksub)
  const int ksub = p.ksub;
  const uint32_t STAGE_BYTES = (uint32_t)ksub * (A_BYTES + B_BYTES);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* full = (uint64_t*)(smem + (size_t)stages * STAGE_BYTES);
  uint64_t* empty = full + stages;
  uint64_t* acc_full = empty + stages;  // [2]
  uint64_t* acc_empty = acc_full + 2;   // [2]
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = (uint32_t*)(drain + 1);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);
  volatile int* status = p.status;
  // one copy of the tile's bias per epilogue warp (BN floats each, 16-byte aligned)
  float* sbias_all = (float*)(((uintptr_t)(abort_flag + 1) + 15) & ~(uintptr_t)15);
  // gathered A: source row of each of the tile's 128 rows (-1 = past the segment)
  int* s_src = (int*)(sbias_all + 4 * BN);
  // grouped: segment row ranges and tile prefix (kSmemGroups + 1 entries each)
  int* s_goff = s_src + BM;
  int* s_gend = s_goff + kSmemGroups + 1;
  int* s_gtile = s_gend + kSmemGroups + 1;


  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int n_acc = p.persistent ? 2 : 1;  // accumulator buffers in TMEM
  const uint32_t tmem_cols = ACC_COLS * (uint32_t)n_acc;
  const long long items = (long long)p.tiles_m * p.tiles_n * p.splits;  // tiles of 128 (PAIR: 256) rows
  const uint32_t rank = CLUSTER ? tc::cluster_ctarank() : 0u;  // PAIR: 0 = leader of the pair
  constexpr int PER_ITEM = PAIR ? 2 : MC;                        // CTAs per work item
  const long long w_first = blockIdx.x / PER_ITEM;
  const long long w_step = gridDim.x / PER_ITEM;
  auto item = [&](long long w) -> Item {
    Item it = resolve_item<GROUPED, PER_ITEM * BM>(p, w, s_goff, s_gend, s_gtile);
    it.row0 += (int)rank * BM;  // this CTA's 128 rows of the PER_ITEM x 128-row tile
    return it;
  };

  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      // gathered A: lane 0's arrival with the B bytes and one arrival per lane for its A copies
      tc::mbar_init(&full[s], AMODE == TC_A_GATHER ? 33 : 1);
      tc::mbar_init(&empty[s], MC);  // MC > 1: released by every CTA of the cluster
    }
    for (int b = 0; b < 2; ++b) {
      tc::mbar_init(&acc_full[b], 1);
      tc::mbar_init(&acc_empty[b], PAIR ? 8 : 128);  // PAIR: one arrival per epilogue warp of either CTA
    }
    tc::mbar_init(drain, 1);
    *abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 1) {
    if constexpr (PAIR)
      tc::tmem_alloc_pair(tmem_slot, tmem_cols);
    else
      tc::tmem_alloc(tmem_slot, tmem_cols);
  }
  if constexpr (GROUPED) {
    if (warp == 2) build_group_table<PAIR ? 2 * BM : BM>(p, lane, s_goff, s_gend, s_gtile);
  }
  tc::tc_fence_before();
  if constexpr (CLUSTER)
    tc::cluster_sync();  // every CTA's barriers exist before any copy or commit reaches them
  else
    __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && AMODE == TC_A_GATHER) {
    if constexpr (AMODE == TC_A_GATHER && !PAIR) {
      if (lane == 0) tc::prefetch_tmap(&tmB);
      const int chunk = lane & 7;          // this lane's 16-byte chunk of each 128-byte row segment
      const int rsub = lane >> 3;          // and its rows rsub + 4 i, i < 32
      uint32_t g = 0;                      // stages filled so far
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (long long w = w_first; ok && w < items; w += w_step) {
        const Item it = item(w);
        if (!it.valid) continue;
        __syncwarp();  // the previous tile's copies have all been issued
#pragma unroll
        for (int i = 0; i < BM / 32; ++i) {
          const int r = it.row0 + lane + 32 * i;
          s_src[lane + 32 * i] = r < it.row_end ? p.row_map[r] / p.row_div : -1;
        }
        __syncwarp();
        int kb = it.kb0;
        for (int i = 0; i < it.nkb; i += ksub, ++g) {
          const int nsub = min(ksub, it.nkb - i);
          int okl = 1;
          if (lane == 0) okl = tc::mbar_wait(&empty[s], ph ^ 1u, abort_flag, status) ? 1 : 0;
          okl = __shfl_sync(0xffffffffu, okl, 0);
          if (!okl) {
            if (lane == 0) fail(RC_DEV_TIMEOUT_EMPTY);
            ok = false;
            break;
          }
          uint8_t* stage = smem + (size_t)s * STAGE_BYTES;
          if (lane == 0) {
            tc::mbar_expect_tx(&full[s], (uint32_t)nsub * B_BYTES);
            for (int q = 0; q < nsub; ++q) {
              uint8_t* sb = stage + ksub * A_BYTES + q * B_BYTES;
              const int nh = it.nt * (BN / 2);
              tc::tma_load_2d(sb, &tmB, &full[s], (kb + q) * BK, it.brow0 + nh);
              tc::tma_load_2d(sb + (BN / 2) * 128, &tmB, &full[s], (kb + q) * BK, it.brow0 + p.swiglu_I + nh);
            }
          }
          for (int q = 0; q < nsub; ++q) {
            const uint32_t sa = tc::smem_u32(stage + q * A_BYTES);
            const int col = (kb + q) * BK + chunk * 8;
            const bool col_ok = col < p.K;
#pragma unroll 8
            for (int ii = 0; ii < 32; ++ii) {
              const int row = rsub + 4 * ii;
              const int src = s_src[row];
              const uint32_t dst = sa + (uint32_t)row * 128u + ((uint32_t)(chunk ^ (row & 7)) << 4);
              const bool v = src >= 0 && col_ok;
              tc::cp_async16(dst, v ? (const void*)(p.a_src + (size_t)src * p.K + col) : (const void*)p.a_src,
                             v ? 16u : 0u);
            }
          }
          kb += nsub;
          tc::cp_async_mbar_arrive(&full[s]);  // this lane's arrival, when its copies of the stage land
          if (++s == stages) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      tc::cp_async_wait(0);  // no copy of this lane is in flight at exit
      if (lane == 0) {  // let the B copies of the last stages land before exit
        const uint32_t first = g > (uint32_t)stages ? g - (uint32_t)stages : 0u;
        for (uint32_t j = first; j < g; ++j)
          if (!tc::mbar_wait_drain(&full[j % (uint32_t)stages], (j / (uint32_t)stages) & 1u))
            fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp == 0) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmA);
      tc::prefetch_tmap(&tmB);
      uint32_t g = 0;   // stages filled so far
      int s = 0;        // ring slot g % stages
      uint32_t ph = 0;  // its phase parity (g / stages) & 1
      bool ok = true;
      for (long long w = w_first; ok && w < items; w += w_step) {
        const Item it = item(w);
        if (!it.valid) continue;
        // convolutions: image and first output row of the tile; filter tap
        // (rr, ss) and channel block cb of the current k sub-block
        int img = 0, prow = 0, rr = 0, ss = 0, cb = 0;
        if constexpr (AMODE == TC_A_CONV || AMODE == TC_A_CONV_ROWS) {
          img = it.row0 / p.img_hw;
          prow = (it.row0 - img * p.img_hw) / p.img_w;
          const int rs = it.kb0 / p.cblocks;
          cb = it.kb0 - rs * p.cblocks;
          rr = rs / p.ks;
          ss = rs - rr * p.ks;
        }
        int kb = it.kb0;
        for (int i = 0; i < it.nkb; i += ksub, ++g) {
          const int nsub = min(ksub, it.nkb - i);
          if (!tc::mbar_wait(&empty[s], ph ^ 1u, abort_flag, status)) {
            fail(RC_DEV_TIMEOUT_EMPTY);
            ok = false;
            break;
          }
          uint8_t* stage = smem + (size_t)s * STAGE_BYTES;
          // PAIR: the leader's barrier counts both CTAs' bytes
          const uint32_t cbar = PAIR ? tc::mapa_shared(tc::smem_u32(&full[s]), 0) : 0u;
          // MC > 1: every CTA's barrier counts its own A and the whole B tile (all the slices)
          if (rank == 0 || !PAIR)
            tc::mbar_expect_tx(&full[s], (uint32_t)nsub * (PAIR ? 2 : 1) * (A_BYTES + B_BYTES));
          auto ld2 = [&](void* dst, const CUtensorMap* m, int x, int y) {
            if constexpr (PAIR)
              tc::tma_load_2d_pair(dst, m, cbar, x, y);
            else
              tc::tma_load_2d(dst, m, &full[s], x, y);
          };
          for (int q = 0; q < nsub; ++q, ++kb) {
            uint8_t* sa = stage + q * A_BYTES;
            uint8_t* sb = stage + ksub * A_BYTES + q * B_BYTES;
            if constexpr (AMODE == TC_A_CONV) {
              if constexpr (PAIR)
                tc::tma_load_4d_pair(sa, &tmA, cbar, cb * 64, ss - p.pad, prow + rr - p.pad, img);
              else
                tc::tma_load_4d(sa, &tmA, &full[s], cb * 64, ss - p.pad, prow + rr - p.pad, img);
            } else if constexpr (AMODE == TC_A_CONV_ROWS) {
              // padded input [N][Hp][Wp][C] as rows of pixels: image row r of the tile, shifted by (rr, ss)
              const int wp = p.img_w + 2 * p.pad_rows, hp = p.img_hw / p.img_w + 2 * p.pad_rows;
              for (int r = 0; r < BM / p.img_w; ++r)
                ld2(sa + r * p.img_w * 128, &tmA, cb * 64, (img * hp + prow + r + rr) * wp + ss);
            } else {
              ld2(sa, &tmA, kb * BK, it.row0);
            }
            if constexpr (AMODE == TC_A_CONV || AMODE == TC_A_CONV_ROWS) {
              if (++cb == p.cblocks) {
                cb = 0;
                if (++ss == p.ks) {
                  ss = 0;
                  ++rr;
                }
              }
            }
            if constexpr (EPI == TC_EPI_SWIGLU) {
              const int nh = it.nt * (BN / 2);
              if constexpr (PAIR) {  // gate rows in the leader, up rows in the peer
                ld2(sb, &tmB, kb * BK, it.brow0 + (rank ? p.swiglu_I : 0) + nh);
              } else {
                ld2(sb, &tmB, kb * BK, it.brow0 + nh);
                ld2(sb + (BN / 2) * 128, &tmB, kb * BK, it.brow0 + p.swiglu_I + nh);
              }
            } else if constexpr (MC > 1) {
              // this CTA's 1 / MC of the B tile's rows, into every CTA of the cluster
              tc::tma_load_2d_mc(sb + rank * (BN / MC) * 128, &tmB, &full[s], kb * BK,
                                 it.brow0 + it.nt * BN + (int)rank * (BN / MC), MC_MASK);
            } else {
              ld2(sb, &tmB, kb * BK, it.brow0 + it.nt * BN + (int)rank * (BN / 2));
            }
          }
          if (++s == stages) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      // let the copies issued in the last `stages` ring slots land before exit
      // (PAIR peer: its copies complete on the leader's barrier; it waits
      // instead, bounded, for the leader's release of those slots)
      const uint32_t first = g > (uint32_t)stages ? g - (uint32_t)stages : 0u;
      for (uint32_t j = first; j < g; ++j) {
        if (rank == 0 || !PAIR) {
          if (!tc::mbar_wait_drain(&full[j % (uint32_t)stages], (j / (uint32_t)stages) & 1u))
            fail(RC_DEV_TIMEOUT_DRAIN);
        } else {
          tc::mbar_wait_drain(&empty[j % (uint32_t)stages], (j / (uint32_t)stages) & 1u);
        }
      }
    }
    __syncwarp();  // reconverge before the final block barrier
  } else if (warp == 1) {
    // the whole warp runs the issue loop on warp-uniform values and one elected lane issues (a lane-0
    // branch spends far longer per UMMA forming its operands); in a pair only the leader CTA issues
    if (rank == 0 || !PAIR) {
      const bool leader = tc::elect_one();
      auto all = [](bool x) { return __all_sync(0xffffffffu, x); };
      constexpr uint32_t idesc = tc::idesc_bf16_f32(PAIR ? 2 * BM : BM, BN);
      const uint32_t sbase = tc::smem_u32(smem);
      uint32_t li = 0;
      int s = 0;        // ring slot, advanced in step with the producer
      uint32_t ph = 0;  // its phase parity
      bool ok = true;
      for (long long w = w_first; ok && w < items; w += w_step) {
        const Item it = item(w);
        if (!it.valid) continue;
        const uint32_t buf = li % (uint32_t)n_acc;
        const uint32_t aph = (li / (uint32_t)n_acc) & 1u;
        if (!all(tc::mbar_wait(&acc_empty[buf], aph ^ 1u, abort_flag, status))) {
          if (leader) fail(RC_DEV_TIMEOUT_ACCUM);
          ok = false;
          break;
        }
        tc::tc_fence_after();
        const uint32_t dacc = tmem + buf * ACC_COLS;
        for (int i = 0; i < it.nkb; i += ksub) {
          const int nsub = min(ksub, it.nkb - i);
          if (!all(tc::mbar_wait(&full[s], ph, abort_flag, status))) {
            if (leader) fail(RC_DEV_TIMEOUT_FULL);
            ok = false;
            break;
          }
          // gathered A: cp.async wrote the rows through the generic proxy; order them before the UMMA reads
          if constexpr (AMODE == TC_A_GATHER) tc::fence_proxy_async_smem();
          tc::tc_fence_after();
          if (leader) {
            const uint32_t sa = sbase + (uint32_t)s * (uint32_t)STAGE_BYTES;
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              if (q >= nsub) break;
              const uint64_t da = tc::sw128_desc(sa + q * A_BYTES);
              const uint64_t db = tc::sw128_desc(sa + ksub * A_BYTES + q * B_BYTES);
#pragma unroll
              for (int k = 0; k < BK / 16; ++k) {
                const uint32_t acc = (i > 0 || q > 0 || k > 0) ? 1u : 0u;
                if constexpr (PAIR)
                  tc::umma_bf16_pair(dacc, da + 2 * k, db + 2 * k, idesc, acc);
                else
                  tc::umma_bf16(dacc, da + 2 * k, db + 2 * k, idesc, acc);
              }
            }
            if constexpr (PAIR)
              tc::umma_commit_pair(&empty[s], 3);  // the slot is free in both CTAs
            else if constexpr (MC > 1)
              tc::umma_commit_mc(&empty[s], MC_MASK);  // this CTA has read the slot: every producer may refill it
            else
              tc::umma_commit(&empty[s]);
          }
          __syncwarp();
          if (++s == stages) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        if (leader) {
          if constexpr (PAIR)
            tc::umma_commit_pair(&acc_full[buf], 3);
          else
            tc::umma_commit(&acc_full[buf]);  // accumulator ready (also when nkb == 0)
        }
        __syncwarp();
        ++li;
      }
      if (!ok && leader) {
        if constexpr (PAIR)
          tc::umma_commit_pair(drain, 1);
        else
          tc::umma_commit(drain);  // wait for the MMAs already issued before TMEM is freed
        if (!tc::mbar_wait_drain(drain, 0)) fail(RC_DEV_TIMEOUT_DRAIN);
      }
    }
    __syncwarp();
  } else {
    const int q = warp & 3;
    float* sbias = sbias_all + (warp - 2) * BN;
    uint32_t li = 0;
    for (long long w = w_first; w < items; w += w_step) {
      const Item it = item(w);
      if (!it.valid) continue;
      if constexpr (EPI == TC_EPI_BIAS_SILU) {
        // the tile's bias, loaded while the accumulator is being computed
        __syncwarp();  // the previous tile's reads of this copy are done
        for (int j = lane; j < BN; j += 32) {
          const int col = it.nt * BN + j;
          sbias[j] = p.bias && col < p.out_cols ? __bfloat162float(p.bias[col]) : 0.f;
        }
        __syncwarp();
      }
      const uint32_t buf = li % (uint32_t)n_acc;
      const uint32_t aph = (li / (uint32_t)n_acc) & 1u;
      if (!tc::mbar_wait(&acc_full[buf], aph, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        break;
      }
      tc::tc_fence_after();
      // one tile per CTA: every ring stage has been read by the tensor core and none is refilled,
      // so the ring can stage the rows of the plain bf16 store, whose time is all in its stores (not
      // with B multicast, whose peers write into the ring; the bias/SiLU epilogue's arithmetic
      // already overlaps its stores, and staging only added to it: conv pair tiles 641 -> 614
      // TFLOP/s, where the plain store gained 1-3% on the down-projection GEMM)
      uint8_t* stg = nullptr;
      if constexpr (MC == 1 && EPI == TC_EPI_STORE_BF16) {
        if (!p.persistent && (size_t)stages * STAGE_BYTES >= (size_t)4 * 32 * stage_pitch<BN>())
          stg = smem + (size_t)(warp - 2) * 32 * stage_pitch<BN>();
      }
      epilogue<BN, EPI>(p, tmem + buf * ACC_COLS + ((uint32_t)(32 * q) << 16), it.row0 + 32 * q + lane,
                        it.row_end, it.nt, it.split, it.nkb > 0, sbias, stg);
      tc::tc_fence_before();
      if constexpr (PAIR) {
        __syncwarp();
        if (lane == 0) tc::mbar_arrive_cluster(tc::mapa_shared(tc::smem_u32(&acc_empty[buf]), 0));
      } else {
        tc::mbar_arrive(&acc_empty[buf]);
      }
      ++li;
    }
  }
  tc::tc_fence_before();
  if constexpr (CLUSTER)
    tc::cluster_sync();  // no copy, commit or arrival may reach a CTA that has exited
  else
    __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    if constexpr (PAIR)
      tc::tmem_dealloc_pair(tmem, tmem_cols);
    else
      tc::tmem_dealloc(tmem, tmem_cols);
  }
}

// ------------------------------------------------------------------ host --
rc_status encode_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows);
rc_status encode_conv(CUtensorMap* m, const void* x, uint64_t c, uint64_t w, uint64_t h, uint64_t n,
                      uint64_t box_w, uint64_t box_h);

template <typename Kern>
rc_status launch_kernel(Kern kern, const CUtensorMap& tmA, const CUtensorMap& tmB, const Params& p, int stages,
                        int acc_cols, size_t smem, int per_item, const LaunchCtx& c) {
  const long long items = (long long)p.tiles_m * p.tiles_n * p.splits;
  if (items <= 0 || items > 0x3fffffffLL) return rc_fail(RC_ERR_UNSUPPORTED_OP, "tc_gemm: %lld work items", items);
  // per_item: CTAs per work item (the cluster: 2 for a CTA pair, MC for B multicast)
  long long ctas = items * per_item;
  if (p.persistent) {
    // as many CTAs as fit on the SMs at once (shared memory and 512 TMEM columns)
    long long per_sm = 233472 / (long long)(smem + 1024);
    const long long by_tmem = 512 / (2LL * acc_cols);
    if (by_tmem < per_sm) per_sm = by_tmem;
    if (per_sm < 1) per_sm = 1;
    long long resident = per_sm * (c.num_sms > 0 ? c.num_sms : 1);
    resident -= resident % per_item;
    if (resident < ctas) ctas = resident;
  }
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)ctas, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = (cudaStream_t)c.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)per_item;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = per_item > 1 ? 1 : 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, tmA, tmB, p, stages);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "tc_gemm launch: %s", cudaGetErrorString(e));
  return RC_OK;
}

// Dynamic shared memory above which two CTAs cannot share an SM (228 KB per SM, 1 KB reserved per CTA).
constexpr size_t kSmemHalfPlus = 233472 / 2 - 1024 + 16;

// ring of A (128 rows) and this CTA's B rows (bn, or bn / 2 for a CTA pair)
// per sub-block + 1 KB alignment slack + barriers and flags (256 B) + four
// fp32 bias copies of the bn-column tile + the gathered-A row table (512 B)
// + the grouped segment tables
inline size_t smem_bytes(int bn, int stages, int ksub, bool pair = false) {
  const size_t b_rows = pair ? (size_t)bn / 2 : (size_t)bn;
  return (size_t)stages * ksub * (BM * BK * 2 + b_rows * BK * 2) + 1024 + 256 + 4 * (size_t)bn * 4 + BM * 4 +
         kGroupTableBytes;
}

template <int BN, int EPI, int AMODE, bool GROUPED, bool PAIR = false, int MC = 1>
rc_status launch(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  auto kern = gemm_kernel<BN, EPI, AMODE, GROUPED, PAIR, MC>;
  if (k.tile_k != 64 && k.tile_k != 128) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm: K tile %d", k.tile_k);
  constexpr int acc_cols_tile = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  const int tmem_cols = (k.persistent ? 2 : 1) * acc_cols_tile;
  const int ksub = k.tile_k / 64;
  size_t smem = smem_bytes(BN, k.stages, ksub, PAIR);
  // A CTA pair taking all 512 TMEM columns of each of its SMs must not share an SM with a CTA of
  // another pair: their allocations could then wait on each other across SMs. Asking for more than
  // half of an SM's shared memory keeps one such CTA per SM, so its allocation never waits.
  if (PAIR && tmem_cols > 256 && smem < kSmemHalfPlus) smem = kSmemHalfPlus;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
    if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "tc_gemm: smem attribute: %s", cudaGetErrorString(e));
    attr_set = true;
  }
  CUtensorMap tmA, tmB;
  if constexpr (AMODE == TC_A_CONV) {
    const uint64_t extra = a.padded ? 2 * (uint64_t)a.pad : 0;  // padded copy: no out-of-range coordinates
    RC_TRY(encode_conv(&tmA, a.A, a.c_in, a.img_w + extra, a.img_h + extra, a.img_n, a.img_w, 128 / a.img_w));
  } else if constexpr (AMODE == TC_A_CONV_ROWS) {
    const uint64_t rows = (uint64_t)a.img_n * (a.img_h + 2 * a.pad) * (a.img_w + 2 * a.pad);
    RC_TRY(encode_2d(&tmA, a.A, a.c_in, rows, (uint32_t)a.img_w));
  } else if constexpr (AMODE == TC_A_GATHER) {
    static_assert(GROUPED && !PAIR && EPI == TC_EPI_SWIGLU, "gathered A: grouped SwiGLU on one CTA");
    if (a.a_rows <= 0 || !a.row_map || (uintptr_t)a.A % 16 || a.K % 8)
      return rc_fail(RC_ERR_INVALID_ARG, "tc_gemm: gathered A needs a row map, rows and 16-byte rows");
    memset(&tmA, 0, sizeof tmA);  // A is copied with cp.async; the map is unused
  } else {
    RC_TRY(encode_2d(&tmA, a.A, a.K, a.M, BM));
  }
  if (GROUPED && (a.groups < 1 || a.groups > kSmemGroups))
    return rc_fail(RC_ERR_UNSUPPORTED_OP, "tc_gemm: grouped GEMM with %d segments (1 .. %d)", a.groups, kSmemGroups);
  const int64_t b_rows = GROUPED ? (int64_t)a.groups * a.b_group_rows : a.N;
  RC_TRY(encode_2d(&tmB, a.B, a.K, b_rows, (PAIR || EPI == TC_EPI_SWIGLU) ? BN / 2 : BN / MC));
  Params p;
  memset(&p, 0, sizeof p);
  p.M = (int)a.M;
  p.N = (int)a.N;
  p.K = (int)a.K;
  const int out_w = EPI == TC_EPI_SWIGLU ? (int)(a.N / 2) : (int)a.N;
  const int tile_out = EPI == TC_EPI_SWIGLU ? BN / 2 : BN;
  p.tiles_n = (out_w + tile_out - 1) / tile_out;
  const int64_t tile_rows = (PAIR ? 2 : MC) * BM;
  // grouped: an upper bound of the tiles the segments need (spare tiles are skipped)
  // (the remainder launch needs at most one tile per segment)
  p.tiles_m = GROUPED ? (int)(a.seg_mode == TC_SEG_REST ? a.groups : PAIR ? a.M / tile_rows + a.groups : a.max_tiles_m)
                      : (int)((a.M + tile_rows - 1) / tile_rows);
  p.kb_total = (int)((a.K + BK - 1) / BK);
  const int splits = EPI == TC_EPI_PARTIAL_F32 ? k.split_k : 1;
  p.kb_per = (p.kb_total + splits - 1) / splits;
  p.splits = splits;
  p.persistent = k.persistent ? 1 : 0;
  p.ksub = ksub;
  p.raster = k.raster;
  p.group = k.group > 0 ? k.group : 1;
  p.D = a.D;
  p.ldd = a.ldd;
  if (a.resid && (EPI != TC_EPI_STORE_BF16 || ((uintptr_t)a.resid % 16) || a.ldd % 8))
    return rc_fail(RC_ERR_INVALID_ARG, "tc_gemm: a residual needs the bf16 store epilogue and 16-byte rows");
  p.resid = (const __nv_bfloat16*)a.resid;
  p.bias = (const __nv_bfloat16*)a.bias;
  p.silu = a.silu;
  p.swiglu_I = (int)(a.N / 2);
  p.out_cols = out_w;
  if constexpr (AMODE == TC_A_CONV || AMODE == TC_A_CONV_ROWS) {
    p.img_hw = (int)(a.img_h * a.img_w);
    p.img_w = (int)a.img_w;
    p.cblocks = (int)(a.c_in / 64);
    p.ks = (int)a.ks;
    p.pad = a.padded ? 0 : (int)a.pad;
    p.pad_rows = (int)a.pad;
  }
  p.offsets = a.offsets;
  p.groups = a.groups;
  p.seg_mode = a.seg_mode;
  p.b_group_rows = (int)a.b_group_rows;
  p.row_scale = a.row_scale;
  p.row_map = a.row_map;
  p.row_div = a.row_div > 0 ? a.row_div : 1;
  p.a_src = (const __nv_bfloat16*)a.A;
  p.status = c.status;
  constexpr int acc_cols = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  return launch_kernel(kern, tmA, tmB, p, k.stages, acc_cols, smem, PAIR ? 2 : MC, c);
}

}  // namespace tcg
