// Grouped (MoE) GEMM with the operand roles exchanged (Layout 2 of the MoE
// GEMM stages): per expert segment g it computes D_g^T = W_g X_g^T, so the
// expert's weight rows stream as the UMMA M operand (128 rows per UMMA) and
// the segment's token rows as the N operand. UMMA N may be any multiple of 16
// up to 256, so a ragged segment of n tokens is cut into ceil(n / TN) token
// tiles of nearly equal size, each a whole number of 16-row units: at most 15
// rows of padding per segment, where 128- or 256-row M tiles of tokens pad
// 12-23% of the routed rows at 64 experts.
//
// One CTA computes 256 weight rows x one token tile with two UMMAs per K step
// into two TMEM accumulators of TN columns each:
//   SwiGLU (gate/up): the gate rows f .. f+127 and the up rows I+f .. I+f+127,
//     so a thread of the epilogue holds a feature's gate and up values for
//     the same tokens: H[token][f + lane] = silu(gate) * up;
//   bf16 store (down): the output features f .. f+255, two halves of 128.
// Warp roles as in tc_gemm.cuh: warp 0 the TMA producer (two 128 x 64 weight
// boxes and the token tile in 64-row boxes per 64-wide K sub-block), warp 1
// TMEM allocation and the warp-uniform issue loop (one elected lane issues),
// warps 2..5 the epilogue. The accumulator holds the output transposed (TMEM
// lane = feature, column = token), so each epilogue warp turns 16 tokens x 32
// features around through a 1 KB shared-memory buffer and stores 16-byte runs
// of a token row's features.
//
// PAIR (TileSize M = 256): a cluster of two CTAs issues cta_group::2 UMMAs of
// M = 256 weight rows, 128 in each CTA, so a pair tile covers 512 weight rows
// (SwiGLU: 256 gate and 256 up features; store: 512 output features) x one
// token tile, and each CTA holds half of the token tile's rows (the UMMA's N
// split in two). An SM then loads 48 KB per 1024 tensor cycles (256-row token
// tiles) instead of 64 KB: the one-CTA form is bound by L2-to-SM bandwidth.
// Token tiles are whole 32-row units here, so that each CTA's half is whole
// 16-row blocks. Barriers and commits follow the CTA pairs of tc_gemm.cuh.
#include "tc_gemm.cuh"

namespace tcg {
namespace {

constexpr int kWRows = 128;                  // weight rows per UMMA
constexpr int kWBytes = kWRows * BK * 2;     // one weight box: 128 rows x 64 K (16 KB)
// token rows per TMA box: 64, or fewer where a CTA holds fewer rows of the token tile
constexpr int x_box(int tn, bool pair) { return (pair ? tn / 2 : tn) < 64 ? (pair ? tn / 2 : tn) : 64; }

struct TParams {
  int K, kb_total, ksub;
  int unit;              // token rows per unit of a token tile (16, or 32 for a CTA pair)
  int tiles_m, tiles_n;  // token tiles (an upper bound; spare ones are skipped) x weight tiles
  int raster, group;
  int persistent;
  int groups;
  const int* offsets;
  int w_group_rows;  // weight rows per expert (2I for gate/up, H for down)
  int f_step;        // output features per weight tile (one CTA: 128 for SwiGLU, 256 for the store; x 2 for a pair)
  int half_off;      // weight-row offset of the second UMMA's rows (I for SwiGLU, f_step / 2 for the store)
  int out_cols;      // output columns (I or H)
  long long ldd;
  void* D;
  int* status;
};

struct TItem {
  bool valid;
  int g, ft, row0, row_end, units;  // token rows [row0, row0 + unit x units) clipped to row_end
};

// Token tiles of a segment of n rows: ceil(ceil(n / unit) / U) with U = TN / unit.
__device__ __forceinline__ int seg_tiles(int n, int unit, int U) {
  return n > 0 ? ((n + unit - 1) / unit + U - 1) / U : 0;
}

// One warp: segment bounds and the exclusive prefix of their token-tile counts.
__device__ __forceinline__ void build_table(const TParams& p, int U, int lane, int* s_goff, int* s_gend,
                                            int* s_gtile) {
  const int G = p.groups;
  const int per = (G + 31) / 32;
  const int g0 = min(G, lane * per), g1 = min(G, g0 + per);
  int sum = 0;
  for (int g = g0; g < g1; ++g) {
    s_goff[g] = p.offsets[g];
    s_gend[g] = p.offsets[g + 1];
    sum += seg_tiles(s_gend[g] - s_goff[g], p.unit, U);
  }
  int incl = sum;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, d);
    if (lane >= d) incl += v;
  }
  int acc = incl - sum;
  for (int g = g0; g < g1; ++g) {
    s_gtile[g] = acc;
    acc += seg_tiles(s_gend[g] - s_goff[g], p.unit, U);
  }
  if (lane == 31) s_gtile[G] = incl;
}

// The segment's u = ceil(n / unit) units are spread over its nt tiles: the first u % nt tiles take
// u / nt + 1 units, the others u / nt (each at most U).
__device__ __forceinline__ TItem resolve(const TParams& p, int U, long long w, const int* s_goff, const int* s_gend,
                                         const int* s_gtile) {
  TItem it;
  int mt;
  map_tile(p, (int)w, mt, it.ft);
  it.valid = mt < s_gtile[p.groups];
  it.g = 0;
  it.row0 = it.row_end = it.units = 0;
  if (!it.valid) return it;
  int lo = 0, hi = p.groups - 1;  // last segment whose first tile is <= mt
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_gtile[mid] <= mt)
      lo = mid;
    else
      hi = mid - 1;
  }
  const int g = lo, tt = mt - s_gtile[g];
  const int n = s_gend[g] - s_goff[g];
  const int u = (n + p.unit - 1) / p.unit, nt = seg_tiles(n, p.unit, U);
  const int base = u / nt, extra = u - base * nt;
  it.g = g;
  it.units = base + (tt < extra ? 1 : 0);
  it.row0 = s_goff[g] + p.unit * (tt * base + min(tt, extra));
  it.row_end = s_gend[g];
  return it;
}

template <int TN, int EPI, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_t_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, const TParams p,
                  const int stages) {
  static_assert(TN == 64 || TN == 128 || TN == 256, "token tile");
  static_assert(EPI == TC_EPI_SWIGLU || EPI == TC_EPI_STORE_BF16, "epilogue");
  constexpr int CT = PAIR ? 2 : 1;             // CTAs per work item
  constexpr int X_BYTES = TN / CT * BK * 2;    // this CTA's token rows of one sub-block
  constexpr int XB = x_box(TN, PAIR), XB_BYTES = XB * BK * 2;
  constexpr int UNIT = PAIR ? 32 : 16;
  constexpr int U = TN / UNIT;
  constexpr uint32_t ACC = 2 * TN;  // one accumulator: two 128-row halves of TN columns
  const int ksub = p.ksub;
  const uint32_t STAGE_BYTES = (uint32_t)ksub * (2 * kWBytes + X_BYTES);

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
  // per epilogue warp: 16 tokens x 32 features of bf16 (1 KB)
  __nv_bfloat16* s_t = (__nv_bfloat16*)(((uintptr_t)(abort_flag + 1) + 15) & ~(uintptr_t)15);
  int* s_goff = (int*)(s_t + 4 * 16 * 32);
  int* s_gend = s_goff + kSmemGroups + 1;
  int* s_gtile = s_gend + kSmemGroups + 1;

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  // persistent CTAs double-buffer the accumulator where two fit in 512 columns
  const int n_acc = p.persistent && 2 * ACC <= 512 ? 2 : 1;
  const uint32_t tmem_cols = ACC * (uint32_t)n_acc;
  const long long items = (long long)p.tiles_m * p.tiles_n;
  const uint32_t rank = PAIR ? tc::cluster_ctarank() : 0u;  // PAIR: 0 = the leader, which issues the UMMAs
  const long long w_first = blockIdx.x / CT, w_step = gridDim.x / CT;
  auto item = [&](long long w) { return resolve(p, U, w, s_goff, s_gend, s_gtile); };
  auto fail = [&](int code) {
    *abort_flag = 1;
    tc::record_failure(status, code);
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
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
  if (warp == 2) build_table(p, U, lane, s_goff, s_gend, s_gtile);
  tc::tc_fence_before();
  if constexpr (PAIR)
    tc::cluster_sync();  // both CTAs' barriers exist before any copy or commit reaches them
  else
    __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      tc::prefetch_tmap(&tmW);
      tc::prefetch_tmap(&tmX);
      uint32_t g = 0;  // stages filled so far
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (long long w = w_first; ok && w < items; w += w_step) {
        const TItem it = item(w);
        if (!it.valid) continue;
        // this CTA's first weight row of each half, and its rows of the token tile
        const int w0 = it.g * p.w_group_rows + it.ft * p.f_step + (int)rank * kWRows;
        const int xrows = p.unit * it.units / CT;
        const int x0 = it.row0 + (int)rank * xrows;
        const int nbox = (xrows + XB - 1) / XB;  // token boxes this CTA loads (within its TN / CT rows)
        for (int kb = 0; kb < p.kb_total; kb += ksub, ++g) {
          const int nsub = min(ksub, p.kb_total - kb);
          if (!tc::mbar_wait(&empty[s], ph ^ 1u, abort_flag, status)) {
            fail(RC_DEV_TIMEOUT_EMPTY);
            ok = false;
            break;
          }
          uint8_t* stage = smem + (size_t)s * STAGE_BYTES;
          // PAIR: both CTAs' copies complete on the leader's barrier, which counts both CTAs' bytes
          const uint32_t cbar = PAIR ? tc::mapa_shared(tc::smem_u32(&full[s]), 0) : 0u;
          if (rank == 0)
            tc::mbar_expect_tx(&full[s], (uint32_t)(CT * nsub) * (2u * kWBytes + (uint32_t)nbox * XB_BYTES));
          auto ld = [&](void* dst, const CUtensorMap* m, int x, int y) {
            if constexpr (PAIR)
              tc::tma_load_2d_pair(dst, m, cbar, x, y);
            else
              tc::tma_load_2d(dst, m, &full[s], x, y);
          };
          for (int q = 0; q < nsub; ++q) {
            const int x = (kb + q) * BK;
            uint8_t* sw = stage + q * 2 * kWBytes;
            uint8_t* sx = stage + ksub * 2 * kWBytes + q * X_BYTES;
            ld(sw, &tmW, x, w0);
            ld(sw + kWBytes, &tmW, x, w0 + p.half_off);
            for (int j = 0; j < nbox; ++j) ld(sx + j * XB_BYTES, &tmX, x, x0 + j * XB);
          }
          if (++s == stages) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      // let the copies issued in the last `stages` ring slots land before exit (PAIR peer: its copies
      // complete on the leader's barrier; it waits instead, bounded, for the leader's release of the slots)
      const uint32_t first = g > (uint32_t)stages ? g - (uint32_t)stages : 0u;
      for (uint32_t j = first; j < g; ++j) {
        if (rank == 0) {
          if (!tc::mbar_wait_drain(&full[j % (uint32_t)stages], (j / (uint32_t)stages) & 1u))
            fail(RC_DEV_TIMEOUT_DRAIN);
        } else {
          tc::mbar_wait_drain(&empty[j % (uint32_t)stages], (j / (uint32_t)stages) & 1u);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (!PAIR || rank == 0) {  // the leader issues the pair's UMMAs
    const bool leader = tc::elect_one();
    auto all = [](bool x) { return __all_sync(0xffffffffu, x); };
    const uint32_t sbase = tc::smem_u32(smem);
    uint32_t li = 0;
    int s = 0;
    uint32_t ph = 0;
    bool ok = true;
    for (long long w = w_first; ok && w < items; w += w_step) {
      const TItem it = item(w);
      if (!it.valid) continue;
      // N = the tile's tokens in whole units (M = 256 over a CTA pair)
      const uint32_t idesc = tc::idesc_bf16_f32(CT * kWRows, p.unit * it.units);
      const uint32_t buf = li % (uint32_t)n_acc;
      const uint32_t aph = (li / (uint32_t)n_acc) & 1u;
      if (!all(tc::mbar_wait(&acc_empty[buf], aph ^ 1u, abort_flag, status))) {
        if (leader) fail(RC_DEV_TIMEOUT_ACCUM);
        ok = false;
        break;
      }
      tc::tc_fence_after();
      const uint32_t d0 = tmem + buf * ACC, d1 = d0 + TN;
      for (int kb = 0; kb < p.kb_total; kb += ksub) {
        const int nsub = min(ksub, p.kb_total - kb);
        if (!all(tc::mbar_wait(&full[s], ph, abort_flag, status))) {
          if (leader) fail(RC_DEV_TIMEOUT_FULL);
          ok = false;
          break;
        }
        tc::tc_fence_after();
        if (leader) {
          const uint32_t sa = sbase + (uint32_t)s * STAGE_BYTES;
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            if (q >= nsub) break;
            const uint64_t dw0 = tc::sw128_desc(sa + q * 2 * kWBytes);
            const uint64_t dw1 = tc::sw128_desc(sa + q * 2 * kWBytes + kWBytes);
            const uint64_t dx = tc::sw128_desc(sa + ksub * 2 * kWBytes + q * X_BYTES);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              const uint32_t acc = (kb > 0 || q > 0 || k > 0) ? 1u : 0u;
              if constexpr (PAIR) {
                tc::umma_bf16_pair(d0, dw0 + 2 * k, dx + 2 * k, idesc, acc);
                tc::umma_bf16_pair(d1, dw1 + 2 * k, dx + 2 * k, idesc, acc);
              } else {
                tc::umma_bf16(d0, dw0 + 2 * k, dx + 2 * k, idesc, acc);
                tc::umma_bf16(d1, dw1 + 2 * k, dx + 2 * k, idesc, acc);
              }
            }
          }
          if constexpr (PAIR)
            tc::umma_commit_pair(&empty[s], 3);  // the slot is free in both CTAs
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
          tc::umma_commit(&acc_full[buf]);
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
    const int q = warp & 3;  // TMEM lanes 32 q .. 32 q + 31: this warp's 32 features of each half
    __nv_bfloat16* st = s_t + (warp - 2) * 16 * 32;
    __nv_bfloat16* D = (__nv_bfloat16*)p.D;
    uint32_t li = 0;
    for (long long w = w_first; w < items; w += w_step) {
      const TItem it = item(w);
      if (!it.valid) continue;
      const uint32_t buf = li % (uint32_t)n_acc;
      const uint32_t aph = (li / (uint32_t)n_acc) & 1u;
      if (!tc::mbar_wait(&acc_full[buf], aph, abort_flag, status)) {
        if (!*abort_flag) fail(RC_DEV_TIMEOUT_ACCUM);
        break;
      }
      tc::tc_fence_after();
      const uint32_t tl = tmem + buf * ACC + ((uint32_t)(32 * q) << 16);
      // chunks of 16 tokens: nch per half, the halves one after the other (SwiGLU: one, gate with up)
      const int nch = p.unit * it.units / 16;
      constexpr int HALVES = EPI == TC_EPI_SWIGLU ? 1 : 2;
      const int total = HALVES * nch;
      // after the transposition lane l stores features 8 (l % 4) .. +7 of tokens l / 4 and l / 4 + 8
      const int tq = lane >> 2, fq = 8 * (lane & 3);
      auto load = [&](int i, uint32_t(&a)[16], uint32_t(&u)[16]) {
        const int h = i >= nch ? 1 : 0, c = 16 * (i - h * nch);
        if constexpr (EPI == TC_EPI_SWIGLU) {
          tc::tmem_ld16(tl + c, a);       // gate
          tc::tmem_ld16(tl + TN + c, u);  // up
        } else {
          tc::tmem_ld16(tl + h * TN + c, a);
        }
      };
      auto wait = [&](uint32_t(&a)[16], uint32_t(&u)[16]) {
        tc::tmem_ld_wait(a);
        if constexpr (EPI == TC_EPI_SWIGLU) tc::tmem_ld_wait(u);
      };
      auto store = [&](int i, const uint32_t(&a)[16], const uint32_t(&u)[16]) {
        const int h = i >= nch ? 1 : 0, c = 16 * (i - h * nch);
        float v[16];
#pragma unroll
        for (int j = 0; j < 16; ++j)
          v[j] = EPI == TC_EPI_SWIGLU ? tc::silu(__uint_as_float(a[j])) * __uint_as_float(u[j]) : __uint_as_float(a[j]);
        __syncwarp();  // the previous chunk's reads of the buffer are done
#pragma unroll
        for (int j = 0; j < 16; ++j) st[j * 32 + lane] = __float2bfloat16_rn(v[j]);
        __syncwarp();
        const int col = it.ft * p.f_step + h * CT * kWRows + (int)rank * kWRows + 32 * q + fq;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int t = tq + 8 * r;
          const int row = it.row0 + c + t;
          const uint4 val = *reinterpret_cast<const uint4*>(st + t * 32 + fq);
          if (row < it.row_end && col < p.out_cols) *reinterpret_cast<uint4*>(D + (long long)row * p.ldd + col) = val;
        }
      };
      // software-pipelined: the next chunk's TMEM loads are in flight while this chunk is stored
      // (tcgen05.wait::ld waits for every earlier load, so a chunk's wait comes before the next issue)
      uint32_t a0[16], u0[16], a1[16], u1[16];
      load(0, a0, u0);
#pragma unroll 1
      for (int i = 0; i < total; i += 2) {
        wait(a0, u0);
        if (i + 1 < total) load(i + 1, a1, u1);
        store(i, a0, u0);
        if (i + 1 >= total) break;
        wait(a1, u1);
        if (i + 2 < total) load(i + 2, a0, u0);
        store(i + 1, a1, u1);
      }
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
  if constexpr (PAIR)
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

template <int TN, int EPI, bool PAIR>
rc_status launch_t(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  auto kern = gemm_t_kernel<TN, EPI, PAIR>;
  constexpr int CT = PAIR ? 2 : 1;
  if (k.tile_k != 64 && k.tile_k != 128) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm_t: K tile %d", k.tile_k);
  const int n_acc = k.persistent && 4 * TN <= 512 ? 2 : 1;  // as in the kernel
  const int tmem_cols = 2 * TN * n_acc;
  if (a.groups < 1 || a.groups > kSmemGroups)
    return rc_fail(RC_ERR_UNSUPPORTED_OP, "tc_gemm_t: %d segments (1 .. %d)", a.groups, kSmemGroups);
  const int64_t out_w = EPI == TC_EPI_SWIGLU ? a.N / 2 : a.N;
  if (out_w % 8 || a.ldd % 8 || (uintptr_t)a.D % 16 || a.ldd < out_w)
    return rc_fail(RC_ERR_INVALID_ARG, "tc_gemm_t: output rows of whole 16-byte runs");
  const size_t smem = tc_t_smem_bytes(TN, k.stages, k.tile_k, PAIR);
  if (smem > 232448) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm_t: %zu bytes of shared memory", smem);
  // all 512 TMEM columns: keep other CTAs off the SM so that no allocation waits (for a CTA pair,
  // on an allocation of a CTA of another pair on the peer's SM)
  const size_t smem_launch = tmem_cols > 256 && smem < kSmemHalfPlus ? kSmemHalfPlus : smem;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
    if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "tc_gemm_t: smem attribute: %s", cudaGetErrorString(e));
    attr_set = true;
  }
  CUtensorMap tmW, tmX;
  RC_TRY(encode_2d(&tmW, a.B, a.K, (uint64_t)a.groups * a.b_group_rows, kWRows));
  RC_TRY(encode_2d(&tmX, a.A, a.K, a.M, x_box(TN, PAIR)));
  TParams p;
  memset(&p, 0, sizeof p);
  p.K = (int)a.K;
  p.kb_total = (int)((a.K + BK - 1) / BK);
  p.ksub = k.tile_k / 64;
  p.unit = PAIR ? 32 : 16;
  // per segment at most n / TN + 2 tiles (see seg_tiles)
  p.tiles_m = (int)(a.M / TN + 2 * a.groups);
  p.f_step = (EPI == TC_EPI_SWIGLU ? kWRows : 2 * kWRows) * CT;
  p.tiles_n = (int)((out_w + p.f_step - 1) / p.f_step);
  p.raster = k.raster;
  p.group = k.group > 0 ? k.group : 1;
  p.persistent = k.persistent ? 1 : 0;
  p.groups = a.groups;
  p.offsets = a.offsets;
  p.w_group_rows = (int)a.b_group_rows;
  p.half_off = EPI == TC_EPI_SWIGLU ? (int)(a.N / 2) : CT * kWRows;
  p.out_cols = (int)out_w;
  p.ldd = a.ldd;
  p.D = a.D;
  p.status = c.status;
  const long long items = (long long)p.tiles_m * p.tiles_n;
  if (items <= 0 || items > 0x3fffffffLL) return rc_fail(RC_ERR_UNSUPPORTED_OP, "tc_gemm_t: %lld work items", items);
  long long ctas = items * CT;
  if (p.persistent) {
    long long per_sm = 233472 / (long long)(smem_launch + 1024);
    const long long by_tmem = 512 / tmem_cols;
    if (by_tmem < per_sm) per_sm = by_tmem;
    if (per_sm < 1) per_sm = 1;
    long long resident = per_sm * (c.num_sms > 0 ? c.num_sms : 1);
    resident -= resident % CT;
    if (resident < ctas) ctas = resident;
  }
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)ctas, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem_launch;
  cfg.stream = (cudaStream_t)c.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)CT;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = PAIR ? 1 : 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, tmW, tmX, p, k.stages);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "tc_gemm_t launch: %s", cudaGetErrorString(e));
  return RC_OK;
}

}  // namespace
}  // namespace tcg

// ring of two 128-row weight boxes and this CTA's token rows (tn, or tn / 2 in a CTA pair) per 64-wide
// K sub-block + 1 KB alignment slack + barriers and flags (256 B) + four 1 KB transposition buffers +
// the segment tables
int64_t tc_t_smem_bytes(int tn, int stages, int tile_k, bool pair) {
  const int64_t x_rows = pair ? tn / 2 : tn;
  return (int64_t)stages * (tile_k / 64) * (2 * tcg::kWBytes + x_rows * tcg::BK * 2) + 1024 + 256 + 16 + 4 * 1024 +
         tcg::kGroupTableBytes;
}

rc_status tc_dispatch_grouped_t(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  using namespace tcg;
  if (k.tile_m != 128 && k.tile_m != 256)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm_t: M tile 128 (one CTA) or 256 (a CTA pair)");
  if (a.a_mode != TC_A_2D) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm_t: A rows as a plain matrix");
  const int tn = a.epilogue == TC_EPI_SWIGLU ? 2 * k.tile_n : k.tile_n;
  const bool pair = k.tile_m == 256;
#define RC_T_CASES(EPI)                                                               \
  switch (tn) {                                                                       \
    case 64: return pair ? launch_t<64, EPI, true>(k, a, c) : launch_t<64, EPI, false>(k, a, c);    \
    case 128: return pair ? launch_t<128, EPI, true>(k, a, c) : launch_t<128, EPI, false>(k, a, c); \
    case 256: return pair ? launch_t<256, EPI, true>(k, a, c) : launch_t<256, EPI, false>(k, a, c); \
  }
  if (a.epilogue == TC_EPI_SWIGLU) {
    RC_T_CASES(TC_EPI_SWIGLU)
  } else if (a.epilogue == TC_EPI_STORE_BF16) {
    RC_T_CASES(TC_EPI_STORE_BF16)
  }
#undef RC_T_CASES
  return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm_t: no variant for token tile %d epilogue %d", tn, a.epilogue);
}
