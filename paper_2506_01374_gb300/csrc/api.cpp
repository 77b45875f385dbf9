// Host-side C ABI: operators (programs P0), schedules (transformed
// programs) and their legality. The problem statement (Sec. 2, Eq. 1)
// defines a program transformed by a sequence of semantics-preserving
// transformations; here a schedule is the canonical knob vector that such a
// sequence produces, one vector per stage (kernel) of the op.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>

#include "rc_internal.h"

// Tensor-core GEMM shared-memory footprint per CTA: a ring of `stages`
// stages of tile_k / 64 sub-blocks, each an A (128 x 64) and a B (bn x 64,
// or bn/2 x 64 in each CTA of a pair) bf16 tile, plus 1 KB alignment slack,
// barriers, four fp32 copies of a bias tile, a 128-entry row table and the
// grouped segment tables (3 x 257 entries + 8 B).
int64_t tc_smem_bytes(int bn_mma, int stages, int tile_k, int tile_m) {
  const int64_t b_rows = tile_m == 256 ? bn_mma / 2 : bn_mma;
  return (int64_t)stages * (tile_k / 64) * (128 * 64 * 2 + b_rows * 64 * 2) + 1024 + 256 + 4 * (int64_t)bn_mma * 4 +
         128 * 4 + 3 * 257 * 4 + 8;
}

namespace {
thread_local std::string g_err;

constexpr int64_t kSmemLimit = 232448;  // 227 KB opt-in shared memory per CTA

bool tc_gemm_ok(int bn_mma, int stages, int tile_k, int tile_m, int persistent, std::string* why) {
  if (bn_mma % 16 != 0 || bn_mma < 16 || bn_mma > 256) {
    if (why) *why = "UMMA N must be a multiple of 16 in [16, 256]";
    return false;
  }
  if (tile_m != 128 && tile_m != 256 && tile_m != 512) {
    if (why) *why = "M tile must be 128 (one CTA), 256 (a CTA pair) or 512 (four CTAs sharing B)";
    return false;
  }
  if (tile_m == 512 && (bn_mma % 32 != 0 || persistent)) {
    // each of the four CTAs loads BN / 4 rows of B: whole 8-row swizzle atoms
    if (why) *why = "a B-multicast cluster needs an N tile divisible by 32 and one tile per cluster";
    return false;
  }
  if (tile_m == 256 && bn_mma < 32) {
    if (why) *why = "a CTA pair splits the N tile: at least 32 columns";
    return false;
  }
  // (persistent CTA pairs with N tiles above 128 take all 512 TMEM columns of their SMs; the
  // launcher then asks for enough shared memory that no other CTA shares those SMs)
  if (tile_k != 64 && tile_k != 128) {
    if (why) *why = "K per stage must be 64 or 128";
    return false;
  }
  if (tc_smem_bytes(bn_mma, stages, tile_k, tile_m) > kSmemLimit) {
    if (why) *why = "operand ring exceeds 227 KB of shared memory";
    return false;
  }
  return true;
}

// MoE grouped GEMM with exchanged operand roles (Layout 2): one CTA computes 256 weight rows
// (two UMMAs of M = 128) x a token tile of tn rows into two TMEM accumulators of tn columns; a CTA
// pair (M tile 256) 512 weight rows with the token tile's rows split over its two CTAs.
bool moe_t_ok(const rc_op_desc& o, int stage, const rc_knobs& k, std::string* why) {
  auto no = [&](const char* m) {
    if (why) *why = m;
    return false;
  };
  const int tn = stage == 1 ? 2 * k.tile_n : k.tile_n;
  if (k.tile_m != 128 && k.tile_m != 256) return no("exchanged operand roles: M tile 128 or 256 (a CTA pair)");
  if (tn != 64 && tn != 128 && tn != 256) return no("exchanged operand roles: token tile of 64, 128 or 256 rows");
  if (stage == 1 && k.location != 0) return no("exchanged operand roles: token rows from the gathered copy");
  if (stage == 2 && k.fuse) return no("exchanged operand roles: the bf16 store epilogue (combine as a pass)");
  // (persistent CTAs with 256-row token tiles keep one accumulator of all 512 TMEM columns: the
  // producer runs ahead into the next tile while the epilogue drains, the tensor core waits)
  if (k.tile_k != 64 && k.tile_k != 128) return no("K per stage must be 64 or 128");
  if (o.hidden % 8 || o.inter % 8) return no("exchanged operand roles: 16-byte runs of output features");
  if (tc_t_smem_bytes(tn, k.stages, k.tile_k, k.tile_m == 256) > kSmemLimit)
    return no("operand ring exceeds 227 KB of shared memory");
  return true;
}

const char* kind_name(int k) {
  switch (k) {
    case RC_OP_GEMM_F32: return "gemm_f32";
    case RC_OP_LINEAR: return "linear";
    case RC_OP_SWIGLU: return "swiglu";
    case RC_OP_MLP: return "mlp";
    case RC_OP_ATTENTION: return "attention";
    case RC_OP_CONV2D: return "conv2d";
    case RC_OP_MOE_ROUTE: return "moe_route";
    case RC_OP_MOE: return "moe";
    case RC_OP_DECODER_LAYER: return "decoder_layer";
  }
  return "?";
}

int n_stages_of(int kind) {
  switch (kind) {
    case RC_OP_MLP: return 2;
    case RC_OP_MOE: return 3;
    case RC_OP_DECODER_LAYER: return 6;
    default: return 1;
  }
}

bool pow2(int64_t x) { return x > 0 && (x & (x - 1)) == 0; }
}  // namespace

rc_status rc_fail(rc_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return st;
}

void rc_clear_error() { g_err.clear(); }

extern "C" const char* rc_last_error(void) { return g_err.c_str(); }
extern "C" const char* rc_version(void) { return "rc 0.1 (sm_103a)"; }

// ------------------------------------------------------------ knob spaces --
// The transformation vocabulary of the paper's prompt (App. A: TileSize,
// Parallel, ComputeLocation, Unroll) extended with loop order, fusion,
// layout, vectorisation, pipeline stages and split-K. Every value listed
// selects a distinct compiled kernel variant or launch configuration.
std::vector<KnobSpec> rc_knob_space(const rc_op_s* op, int stage) {
  std::vector<KnobSpec> v;
  const int kind = op->d.kind;
  // bytes per access of the memory-bound pass a stage may run after its GEMM (SwiGLU, bias/SiLU,
  // split-K reduce, MoE gather and combine); normalised to the default where the stage runs none
  auto vectorize = [&]() { v.push_back({RC_T_VECTORIZE, 0, {4, 8, 16}, {}}); };
  auto gemm_common = [&](std::vector<int32_t> tn) {
    v.push_back({RC_T_TILE_SIZE, 1, tn, {}});
    v.push_back({RC_T_TILE_SIZE, 2, {64, 128}, {}});  // K per ring stage: one or two 64-wide sub-blocks
    v.push_back({RC_T_PIPELINE_STAGES, 0, {1, 2, 3, 4, 6}, {}});
    v.push_back({RC_T_LOOP_ORDER, 0, {0, 1}, {1, 8}});
    v.push_back({RC_T_PARALLEL, 0, {0, 1}, {}});  // one CTA per tile, or persistent CTAs
  };
  switch (kind) {
    case RC_OP_GEMM_F32:
      v.push_back({RC_T_TILE_SIZE, 0, {16, 32, 64}, {}});
      v.push_back({RC_T_TILE_SIZE, 1, {16, 32, 64}, {}});
      v.push_back({RC_T_TILE_SIZE, 2, {16, 32, 64}, {}});
      v.push_back({RC_T_UNROLL, 0, {1, 4}, {}});
      break;
    case RC_OP_LINEAR:
      gemm_common({64, 128, 224, 256});
      // one CTA, a CTA pair sharing each UMMA, or four CTAs sharing the B tile by TMA multicast
      v.push_back({RC_T_TILE_SIZE, 0, {128, 256, 512}, {}});
      v.push_back({RC_T_SPLIT_K, 0, {1, 2, 4}, {}});
      vectorize();
      break;
    case RC_OP_SWIGLU:
      gemm_common({32, 64, 128});
      v.push_back({RC_T_TILE_SIZE, 0, {128, 256}, {}});
      v.push_back({RC_T_FUSE, 0, {0, 1}, {}});
      vectorize();
      break;
    case RC_OP_MLP:
      if (stage == 0) {
        gemm_common({32, 64, 128});
        v.push_back({RC_T_FUSE, 0, {0, 1}, {}});
      } else {
        gemm_common({64, 128, 224, 256});
        v.push_back({RC_T_SPLIT_K, 0, {1, 2, 4}, {}});
      }
      // the down projection may also share its B tile across four CTAs
      v.push_back({RC_T_TILE_SIZE, 0, stage == 0 ? std::vector<int32_t>{128, 256} : std::vector<int32_t>{128, 256, 512},
                   {}});
      vectorize();
      break;
    case RC_OP_CONV2D:
      gemm_common({64, 80, 160});
      v.push_back({RC_T_TILE_SIZE, 0, {128, 256, 512}, {}});
      v.push_back({RC_T_SPLIT_K, 0, {1, 3, 5}, {}});
      v.push_back({RC_T_FUSE, 0, {0, 1}, {}});
      vectorize();
      // implicit zero padding (one 4-D box), or a padded copy read as one 4-D box or as row boxes
      v.push_back({RC_T_LAYOUT, 0, {0, 1, 2}, {}});
      break;
    case RC_OP_DECODER_LAYER:
      if (stage == 1) {  // RoPE and the split of q, k, v: tokens per CTA
        v.push_back({RC_T_TILE_SIZE, 0, {1, 2, 4, 8}, {}});
        break;
      }
      if (stage != 2) {
        // 0: QKV projection, 3: O projection, 4: gate/up + SwiGLU, 5: down projection
        gemm_common(stage == 4 ? std::vector<int32_t>{32, 64, 128} : std::vector<int32_t>{64, 128, 224, 256});
        v.push_back({RC_T_TILE_SIZE, 0, stage == 4 ? std::vector<int32_t>{128, 256} : std::vector<int32_t>{128, 256, 512},
                     {}});
        if (stage == 4) {
          v.push_back({RC_T_FUSE, 0, {0, 1}, {}});
          vectorize();  // the SwiGLU pass of the unfused gate/up GEMM
        }
        break;
      }
      [[fallthrough]];  // 2: the attention core
    case RC_OP_ATTENTION:
      v.push_back({RC_T_TILE_SIZE, 1, {64, 128}, {}});  // key block BN
      // query rows per CTA: one 128-row tile, or two tiles sharing each K and V block (128-key
      // blocks, one CTA per SM, the tensor core working on one tile while the other's softmax runs)
      v.push_back({RC_T_TILE_SIZE, 0, {128, 256}, {}});
      v.push_back({RC_T_PIPELINE_STAGES, 0, {1, 2, 3, 4, 5}, {}});
      v.push_back({RC_T_LOOP_ORDER, 0, {0, 1}, {1}});  // 0 = head-major tiles, 1 = longest causal rows first
      v.push_back({RC_T_LAYOUT, 0, {0, 1}, {}});        // V as [keys][d] or transposed to [d][keys]
      // P stored in shared (0) or tensor memory (1); 2: P in tensor memory and the row sums of P
      // formed by the tensor core (a block of ones appended to V)
      v.push_back({RC_T_COMPUTE_LOCATION, 0, {0, 1, 2}, {}});
      v.push_back({RC_T_UNROLL, 0, {1, 2}, {}});  // S buffers: key blocks in flight per query tile
      // 0: one UMMA-issuing warp; 1: the S and P V products issued by warps of their own;
      // 2: as 1 with two softmax threads per query row
      v.push_back({RC_T_PARALLEL, 0, {0, 1, 2}, {}});
      break;
    case RC_OP_MOE_ROUTE:
      v.push_back({RC_T_TILE_SIZE, 0, {4, 8, 16}, {}});
      break;
    case RC_OP_MOE:
      if (stage == 0) {
        v.push_back({RC_T_TILE_SIZE, 0, {4, 8, 16}, {}});
        vectorize();  // the row gather
      } else if (stage == 1) {
        gemm_common({32, 64, 128});
        v.push_back({RC_T_TILE_SIZE, 0, {128, 256}, {}});  // 256: a CTA pair within one expert's rows
        // where the token rows are gathered: 0 = a separate pass writes the grouped copy (stage 0),
        // 1 = the grouped GEMM's producer gathers them from X (M tile 128)
        v.push_back({RC_T_COMPUTE_LOCATION, 0, {0, 1}, {}});
        // how the grouped GEMM lays out a ragged expert segment: 0 = whole M tiles of tokens, 1 = CTA-pair
        // tiles and a last 128-row single-CTA tile where the remainder fits it (a second, one-CTA launch),
        // 2 = the operand roles exchanged: weight rows on UMMA M, the segment's tokens on N in tiles of
        // whole 16-row units (the tile transposed in TMEM; the N tile knob sets the token tile)
        v.push_back({RC_T_LAYOUT, 0, {0, 1, 2}, {}});
      } else {
        gemm_common({64, 128, 224, 256});
        v.push_back({RC_T_FUSE, 0, {0, 1}, {}});
        v.push_back({RC_T_TILE_SIZE, 0, {128, 256}, {}});
        v.push_back({RC_T_LAYOUT, 0, {0, 1, 2}, {}});  // as in stage 1
        vectorize();  // the combine (or the fp32 -> bf16 pass of the atomic combine)
      }
      break;
  }
  return v;
}

rc_knobs rc_default_knobs(const rc_op_s* op, int stage) {
  rc_knobs k;
  memset(&k, 0, sizeof k);
  k.tile_m = 128;
  k.tile_k = 64;
  k.unroll = 1;
  k.stages = 1;
  k.split_k = 1;
  k.raster = 0;
  k.group = 1;
  k.persistent = 0;
  k.fuse = 0;
  k.layout = 0;
  k.vec = 16;
  k.location = 0;
  switch (op->d.kind) {
    case RC_OP_GEMM_F32:
      k.tile_m = k.tile_n = k.tile_k = 16;
      k.vec = 4;
      k.fuse = 1;
      break;
    case RC_OP_LINEAR: k.tile_n = 64; break;
    case RC_OP_SWIGLU: k.tile_n = 32; break;
    case RC_OP_MLP: k.tile_n = stage == 0 ? 32 : 64; break;
    case RC_OP_CONV2D: k.tile_n = 64; break;
    case RC_OP_ATTENTION:
      k.tile_n = 64;
      k.stages = 2;
      k.layout = 1;
      break;
    case RC_OP_MOE_ROUTE: k.tile_m = 4; break;
    case RC_OP_MOE:
      if (stage == 0) k.tile_m = 4;
      else k.tile_n = stage == 1 ? 32 : 64;
      break;
    case RC_OP_DECODER_LAYER:
      if (stage == 1) {
        k.tile_m = 1;
      } else if (stage == 2) {
        k.tile_n = 64;
        k.stages = 2;
        k.layout = 1;
      } else {
        k.tile_n = stage == 4 ? 32 : 64;
      }
      break;
  }
  return k;
}

static bool in(const std::vector<int32_t>& v, int32_t x) {
  for (int32_t y : v)
    if (y == x) return true;
  return false;
}

static bool attention_knobs_ok(const rc_knobs& k, int64_t seq, std::string* why);

bool rc_knobs_legal(const rc_op_s* op, int stage, const rc_knobs& k, std::string* why) {
  // 1) every tunable knob holds one of its listed values; untunable knobs keep P0's value
  const rc_knobs d = rc_default_knobs(op, stage);
  const auto space = rc_knob_space(op, stage);
  auto spec_of = [&](int tk, int axis) -> const KnobSpec* {
    for (auto& s : space)
      if (s.tkind == tk && s.axis == axis) return &s;
    return nullptr;
  };
  struct F { int tk, axis; int32_t v, dv; } fields[] = {
      {RC_T_TILE_SIZE, 0, k.tile_m, d.tile_m},       {RC_T_TILE_SIZE, 1, k.tile_n, d.tile_n},
      {RC_T_TILE_SIZE, 2, k.tile_k, d.tile_k},       {RC_T_UNROLL, 0, k.unroll, d.unroll},
      {RC_T_PIPELINE_STAGES, 0, k.stages, d.stages}, {RC_T_SPLIT_K, 0, k.split_k, d.split_k},
      {RC_T_LOOP_ORDER, 0, k.raster, d.raster},      {RC_T_PARALLEL, 0, k.persistent, d.persistent},
      {RC_T_FUSE, 0, k.fuse, d.fuse},                {RC_T_LAYOUT, 0, k.layout, d.layout},
      {RC_T_VECTORIZE, 0, k.vec, d.vec},             {RC_T_COMPUTE_LOCATION, 0, k.location, d.location},
  };
  for (auto& f : fields) {
    const KnobSpec* s = spec_of(f.tk, f.axis);
    if (s ? !in(s->values, f.v) : f.v != f.dv) {
      if (why) *why = "knob value outside this op's transformation space";
      return false;
    }
  }
  const KnobSpec* lo = spec_of(RC_T_LOOP_ORDER, 0);
  if (lo ? !in(lo->values1, k.group) : k.group != d.group) {
    if (why) *why = "raster group outside this op's transformation space";
    return false;
  }
  // 2) resource and shape rules of the kernel the knobs select
  const rc_op_desc& o = op->d;
  switch (o.kind) {
    case RC_OP_LINEAR:
      return tc_gemm_ok(k.tile_n, k.stages, k.tile_k, k.tile_m, k.persistent, why);
    case RC_OP_SWIGLU:
      return tc_gemm_ok(2 * k.tile_n, k.stages, k.tile_k, k.tile_m, k.persistent, why);
    case RC_OP_MLP:
      return tc_gemm_ok(stage == 0 ? 2 * k.tile_n : k.tile_n, k.stages, k.tile_k, k.tile_m, k.persistent, why);
    case RC_OP_CONV2D:
      if (o.c_out % k.tile_n != 0) {
        if (why) *why = "conv N tile must divide Cout";
        return false;
      }
      if (k.tile_m >= 256 && k.layout == 2) {
        if (why) *why = "a CTA pair or a B-multicast cluster loads A as one 4-D box (layouts 0 and 1)";
        return false;
      }
      if (k.tile_m == 512 && (o.img_n * o.img_h * o.img_w) % 512 != 0) {
        if (why) *why = "a B-multicast cluster needs whole 512-row tiles of output pixels";
        return false;
      }
      return tc_gemm_ok(k.tile_n, k.stages, k.tile_k, k.tile_m, k.persistent, why);
    case RC_OP_MOE:
      if (stage == 0) return true;
      if (stage == 1 && k.location == 1 && k.tile_m != 128) {
        if (why) *why = "rows gathered in the GEMM producer need one CTA per tile (M tile 128)";
        return false;
      }
      if (k.layout == 2) return moe_t_ok(o, stage, k, why);
      return tc_gemm_ok(stage == 1 ? 2 * k.tile_n : k.tile_n, k.stages, k.tile_k, k.tile_m, k.persistent, why);
    case RC_OP_DECODER_LAYER:
      if (stage == 1) return true;
      if (stage == 2) return attention_knobs_ok(k, o.tokens, why);
      return tc_gemm_ok(stage == 4 ? 2 * k.tile_n : k.tile_n, k.stages, k.tile_k, k.tile_m, k.persistent, why);
    case RC_OP_ATTENTION:
      return attention_knobs_ok(k, o.seq, why);
    default:
      return true;
  }
}

// Resource and variant rules of the attention kernels (RC_OP_ATTENTION and the
// decoder layer's attention stage).
static bool attention_knobs_ok(const rc_knobs& k, int64_t seq, std::string* why) {
  auto no = [&](const char* m) {
    if (why) *why = m;
    return false;
  };
  // (rc_schedule_apply canonicalises location and unroll per kernel family before this check)
  if (k.tile_m == 256) {
    if (k.tile_n != 128 || k.persistent != 1 || k.location != 1 || k.unroll != 1)
      return no("two query tiles per CTA take 128-key blocks, P in tensor memory and one S buffer per tile");
    if (k.layout == 1 && seq % 8) return no("transposed V needs seq % 8 == 0 (16-byte TMA rows)");
    // two query tiles, the K ring, a two-slot V ring, barriers, TMEM address and abort flag, slack
    const int64_t smem2 = 2 * 128 * 128 * 2 + (k.stages + 2) * 128 * 128 * 2 + (14 + k.stages) * 8 + 8 + 1024;
    if (smem2 > kSmemLimit) return no("attention ring exceeds 227 KB of shared memory");
    return true;
  }
  if (k.tile_m != 128) return no("query tiles of 128 or 256 rows");
  if (k.persistent == 0) {
    if (k.location != 0 || k.unroll != 1) return no("one UMMA-issuing warp keeps P in shared memory and one S buffer");
  } else if (k.location == 0) {
    return no("split UMMA issue keeps P in tensor memory");
  }
  if (k.location == 2 && k.layout != 0) return no("row sums on the tensor core need V as given");
  if (k.layout == 1 && seq % 8) return no("transposed V needs seq % 8 == 0 (16-byte TMA rows)");
  int64_t smem;
  if (k.persistent == 0) {
    // Q tile, K/V ring, P tile, slack and barriers
    smem = 128 * 128 * 2 + (int64_t)k.stages * 2 * k.tile_n * 128 * 2 + 128 * (int64_t)k.tile_n * 2 + 1024 + 512;
  } else {
    // Q, the K ring and a V ring (two slots when two CTAs share an SM), the row-exchange area with two
    // softmax threads per row, barriers, and alignment slack when one CTA holds the SM
    const bool split = k.persistent == 2, sumc = k.location == 2;
    const bool two_ctas = k.tile_n == 64 && !(k.unroll == 2 && sumc);  // TMEM <= 256 columns
    const int64_t vst = two_ctas && k.stages > 2 ? 2 : k.stages;
    const int64_t vslot = k.tile_n * 128 * 2 + (sumc ? k.tile_n * 128 : 0);  // + the ones atom
    smem = 128 * 128 * 2 + k.stages * k.tile_n * 128 * 2 + vst * vslot + (split ? 2048 : 0) +
           (11 + 2 * k.stages + 2 * vst + (split ? 8 : 0)) * 8 + 8 + (two_ctas ? 0 : 1024);
  }
  if (smem > kSmemLimit) return no("attention ring exceeds 227 KB of shared memory");
  return true;
}

// -------------------------------------------------------------- op slots --
std::vector<SlotInfo> rc_slots(const rc_op_s* op) {
  const rc_op_desc& d = op->d;
  std::vector<SlotInfo> s;
  const size_t b2 = 2, b4 = 4;
  switch (d.kind) {
    case RC_OP_GEMM_F32:
      s = {{b4 * d.m * d.k, true, false, false},
           {b4 * d.k * d.n, true, false, false},
           {b4 * d.n, true, false, true},
           {b4 * d.m * d.n, false, true, false}};
      break;
    case RC_OP_LINEAR:
      s = {{b2 * d.m * d.k, true, false, false},
           {b2 * d.n * d.k, true, false, false},
           {b2 * d.m * d.n, false, true, false}};
      break;
    case RC_OP_SWIGLU:
      s = {{b2 * d.m * d.k, true, false, false},
           {b2 * 2 * d.n * d.k, true, false, false},
           {b2 * d.m * d.n, false, true, false}};
      break;
    case RC_OP_MLP:
      s = {{b2 * d.m * d.k, true, false, false},
           {b2 * 2 * d.n * d.k, true, false, false},
           {b2 * d.k * d.n, true, false, false, 1},  // W2: read by the down projection only
           {b2 * d.m * d.k, false, true, false}};
      break;
    case RC_OP_ATTENTION: {
      const size_t q = b2 * d.batch * d.seq * d.heads_q * d.head_dim;
      const size_t kv = b2 * d.batch * d.seq * d.heads_kv * d.head_dim;
      s = {{q, true, false, false},
           {kv, true, false, false},
           {kv, true, false, false},
           {q, false, true, false},
           {b4 * d.batch * d.heads_q * d.seq, false, true, true}};
      break;
    }
    case RC_OP_CONV2D:
      s = {{b2 * d.img_n * d.img_h * d.img_w * d.c_in, true, false, false},
           {b2 * d.c_out * d.kr * d.ks * d.c_in, true, false, false},
           {b2 * d.c_out, true, false, true},
           {b2 * d.img_n * d.img_h * d.img_w * d.c_out, false, true, false}};
      break;
    case RC_OP_MOE_ROUTE: {
      const size_t lg = (d.logits_fp32 ? b4 : b2) * d.tokens * d.experts;
      const size_t tk = (size_t)d.tokens * d.top_k;
      s = {{lg, true, false, false},
           {b4 * tk, false, true, false},
           {b4 * tk, false, true, false},
           {b4 * (d.experts + 1), false, true, false},
           {b4 * tk, false, true, false}};
      break;
    }
    case RC_OP_MOE: {
      const size_t lg = (d.logits_fp32 ? b4 : b2) * d.tokens * d.experts;
      const size_t tk = (size_t)d.tokens * d.top_k;
      s = {{lg, true, false, false},
           {b2 * d.tokens * d.hidden, true, false, false},
           {b2 * d.experts * 2 * d.inter * d.hidden, true, false, false, 1},  // W1: grouped gate/up
           {b2 * d.experts * d.hidden * d.inter, true, false, false, 2},      // W2: grouped down
           {b2 * d.tokens * d.hidden, false, true, false},
           {b4 * tk, false, true, true},
           {b4 * tk, false, true, true},
           {b4 * (d.experts + 1), false, true, true},
           {b4 * tk, false, true, true}};
      break;
    }
    case RC_OP_DECODER_LAYER: {
      const size_t T = d.tokens, H = d.hidden, D = d.head_dim;
      s = {{b2 * T * H, true, false, false},
           {b2 * H, true, false, false},
           {b2 * (d.heads_q + 2 * d.heads_kv) * D * H, true, false, false},
           {b2 * H * d.heads_q * D, true, false, false, 3},  // Wo: O projection
           {b2 * H, true, false, false, 3},                  // g2: the second RMSNorm
           {b2 * 2 * d.inter * H, true, false, false, 4},    // W1: gate/up
           {b2 * H * d.inter, true, false, false, 5},        // W2: down
           {b2 * T * H, false, true, false}};
      break;
    }
  }
  return s;
}

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t rc_workspace_bytes(const rc_op_s* op, const rc_schedule_s* s) {
  const rc_op_desc& d = op->d;
  const rc_knobs* k = s ? s->k : nullptr;
  switch (d.kind) {
    case RC_OP_LINEAR:
      return (k && k[0].split_k > 1) ? align256(4ull * k[0].split_k * d.m * d.n) : 0;
    case RC_OP_SWIGLU:
      return (k && !k[0].fuse) ? align256(2ull * d.m * 2 * d.n) : 0;
    case RC_OP_MLP: {
      size_t b = align256(2ull * d.m * d.n);                          // h
      if (k && !k[0].fuse) b += align256(2ull * d.m * 2 * d.n);       // gate|up before SwiGLU
      if (k && k[1].split_k > 1) b += align256(4ull * k[1].split_k * d.m * d.k);
      return b;
    }
    case RC_OP_CONV2D: {
      const size_t rows = (size_t)d.img_n * d.img_h * d.img_w;
      size_t b = 0;
      if (k && k[0].layout >= 1) b += align256(2ull * d.img_n * (d.img_h + 2 * d.pad) * (d.img_w + 2 * d.pad) * d.c_in);
      if (k && k[0].split_k > 1) b += align256(4ull * k[0].split_k * rows * d.c_out);
      if (k && (!k[0].fuse || k[0].split_k > 1)) b += align256(2ull * rows * d.c_out);
      return b;
    }
    case RC_OP_ATTENTION:
      return (k && k[0].layout == 1) ? align256(2ull * d.batch * d.heads_kv * d.head_dim * d.seq) : 0;
    case RC_OP_DECODER_LAYER: {
      const size_t T = d.tokens, H = d.hidden, D = d.head_dim, I = d.inter;
      const size_t hq = d.heads_q * D, hkv = d.heads_kv * D;
      size_t b = align256(2 * T * H);                               // a = RMSNorm(x) g1
      b += align256(2 * T * (hq + 2 * hkv));                        // qkv
      b += align256(2 * T * hq) + 2 * align256(2 * T * hkv);        // Q, K, V after RoPE
      b += align256(2 * T * hq);                                    // attention output o
      b += 2 * align256(2 * T * H);                                 // h1, b
      b += align256(2 * T * I);                                     // SwiGLU output
      if (k && !k[4].fuse) b += align256(2 * T * 2 * I);            // gate|up before SwiGLU
      if (k && k[2].layout == 1) b += align256(2 * hkv * T);        // V transposed for attention
      return b;
    }
    case RC_OP_MOE_ROUTE:
      return align256(4ull * d.experts);  // per-expert counts
    case RC_OP_MOE: {
      const size_t slots = (size_t)d.tokens * d.top_k;
      size_t b = 0;
      b += align256(4 * slots) * 4 + align256(4 * (d.experts + 1));  // ids, w, perm, inv_perm, offsets
      b += align256(4ull * d.experts);                                // per-expert counts
      b += align256(2 * slots * d.hidden);                            // gathered X
      b += align256(2 * slots * d.inter);                             // H
      b += align256(2 * slots * d.hidden);                            // Y (bf16) for gather-reduce
      b += align256(4ull * d.tokens * d.hidden);                      // fp32 out for atomic combine
      return b;
    }
    default:
      return 0;
  }
}

// -------------------------------------------------------------- describe --
extern "C" rc_status rc_op_describe(const rc_op_desc* desc, rc_op** out) {
  if (!desc || !out) return rc_fail(RC_ERR_INVALID_ARG, "rc_op_describe: NULL argument");
  *out = nullptr;
  rc_op_desc d = *desc;
  rc_op_info_t info;
  memset(&info, 0, sizeof info);
  auto bad = [&](const char* what) {
    return rc_fail(RC_ERR_INVALID_ARG, "rc_op_describe(%s): %s", kind_name(d.kind), what);
  };
  auto unsup = [&](const char* what) {
    return rc_fail(RC_ERR_UNSUPPORTED_OP, "rc_op_describe(%s): %s", kind_name(d.kind), what);
  };
  const double ridge = 283.0;  // bf16 tensor FLOP per HBM byte on GB300 (measured peaks ratio)
  switch (d.kind) {
    case RC_OP_GEMM_F32:
      if (d.m <= 0 || d.n <= 0 || d.k <= 0) return bad("m, n, k must be positive");
      info.flops = 2.0 * d.m * d.n * d.k;
      info.bytes = 4.0 * (d.m * d.k + d.k * d.n + d.n + d.m * d.n);
      info.bound = RC_BOUND_FP32_SIMT;
      info.n_tensors = 4;
      break;
    case RC_OP_LINEAR:
    case RC_OP_SWIGLU:
    case RC_OP_MLP: {
      if (d.m <= 0 || d.n <= 0 || d.k <= 0) return bad("m, n, k must be positive");
      if (d.k % 8 || d.n % 8) return unsup("k and n must be multiples of 8 (16-byte rows)");
      const double ncols = d.kind == RC_OP_SWIGLU ? 2.0 * d.n : (double)d.n;
      if (d.kind == RC_OP_MLP) {
        info.flops = 6.0 * d.m * d.n * d.k;
        info.bytes = 2.0 * (2.0 * d.m * d.k + 3.0 * d.n * d.k);
        info.n_tensors = 4;
      } else {
        info.flops = 2.0 * d.m * ncols * d.k;
        info.bytes = 2.0 * (d.m * d.k + ncols * d.k + (double)d.m * d.n);
        info.n_tensors = 3;
      }
      info.bound = info.flops / info.bytes >= ridge ? RC_BOUND_TENSOR : RC_BOUND_HBM;
      break;
    }
    case RC_OP_ATTENTION: {
      if (d.batch <= 0 || d.seq <= 0 || d.heads_q <= 0 || d.heads_kv <= 0 || d.head_dim <= 0)
        return bad("sizes must be positive");
      if (d.heads_q % d.heads_kv) return bad("heads_q must be a multiple of heads_kv");
      if (d.head_dim != 128) return unsup("head_dim must be 128");
      if (d.scale == 0.0) d.scale = 1.0 / std::sqrt((double)d.head_dim);
      const double pairs = d.causal ? 0.5 * (double)d.seq * (d.seq + 1) : (double)d.seq * d.seq;
      info.flops = 4.0 * d.head_dim * d.heads_q * d.batch * pairs;
      info.bytes = 2.0 * d.batch * d.seq * d.head_dim * (2.0 * d.heads_q + 2.0 * d.heads_kv) +
                   4.0 * d.batch * d.heads_q * d.seq;
      info.bound = RC_BOUND_TENSOR;
      info.n_tensors = 5;
      break;
    }
    case RC_OP_CONV2D: {
      if (d.img_n <= 0 || d.img_h <= 0 || d.img_w <= 0 || d.c_in <= 0 || d.c_out <= 0 || d.kr <= 0 ||
          d.ks <= 0)
        return bad("sizes must be positive");
      if (d.stride == 0) d.stride = 1;
      if (d.stride != 1 || d.kr != d.ks || d.kr % 2 == 0 || d.pad != (d.kr - 1) / 2)
        return unsup("only stride-1 'same' convolutions with an odd square kernel");
      if (d.c_in % 64) return unsup("c_in must be a multiple of 64");
      if (d.c_out % 16) return unsup("c_out must be a multiple of 16");
      if (!pow2(d.img_w) || d.img_w < 8 || d.img_w > 128 || d.img_h % (128 / d.img_w))
        return unsup("img_w must be a power of two in [8, 128] and img_h a multiple of 128/img_w");
      const double pix = (double)d.img_n * d.img_h * d.img_w;
      info.flops = 2.0 * pix * d.c_out * d.kr * d.ks * d.c_in;
      info.bytes = 2.0 * (pix * d.c_in + (double)d.c_out * d.kr * d.ks * d.c_in + d.c_out + pix * d.c_out);
      info.bound = info.flops / info.bytes >= ridge ? RC_BOUND_TENSOR : RC_BOUND_HBM;
      info.n_tensors = 4;
      break;
    }
    case RC_OP_MOE_ROUTE:
    case RC_OP_MOE: {
      if (d.tokens <= 0 || d.experts <= 0 || d.top_k <= 0) return bad("sizes must be positive");
      if (d.top_k > d.experts) return bad("top_k must not exceed experts");
      if (d.experts > 256 || d.top_k > 16) return unsup("experts <= 256 and top_k <= 16");
      const double slots = (double)d.tokens * d.top_k;
      const double lg = (d.logits_fp32 ? 4.0 : 2.0) * d.tokens * d.experts;
      if (d.kind == RC_OP_MOE_ROUTE) {
        info.flops = 0.0;
        info.bytes = lg + 12.0 * slots + 4.0 * (d.experts + 1);
        info.bound = RC_BOUND_HBM;
        info.n_tensors = 5;
      } else {
        if (d.hidden <= 0 || d.inter <= 0) return bad("hidden and inter must be positive");
        if (d.hidden % 64 || d.inter % 64) return unsup("hidden and inter must be multiples of 64");
        info.flops = 6.0 * slots * d.hidden * d.inter;
        info.bytes = lg + 2.0 * (2.0 * d.tokens * d.hidden + 3.0 * d.experts * d.hidden * d.inter);
        info.bound = info.flops / info.bytes >= ridge ? RC_BOUND_TENSOR : RC_BOUND_HBM;
        info.n_tensors = 9;
      }
      break;
    }
    case RC_OP_DECODER_LAYER: {
      if (d.tokens <= 0 || d.hidden <= 0 || d.inter <= 0 || d.heads_q <= 0 || d.heads_kv <= 0)
        return bad("tokens, hidden, inter, heads_q, heads_kv must be positive");
      if (d.head_dim == 0) d.head_dim = 128;
      if (d.head_dim != 128) return unsup("head_dim must be 128");
      if (d.heads_q % d.heads_kv) return bad("heads_q must be a multiple of heads_kv");
      if (d.hidden % 256 || d.hidden > 32768)
        return unsup("hidden must be a multiple of 256 and at most 32768 (one RMSNorm row per CTA in registers)");
      if (d.inter % 64) return unsup("inter must be a multiple of 64");
      if (d.tokens > 0x7fffffffLL) return unsup("tokens must fit in 31 bits");
      if (d.rope_theta == 0.0) d.rope_theta = 500000.0;
      if (d.norm_eps == 0.0) d.norm_eps = 1e-5;
      if (!(d.rope_theta > 1.0) || !(d.norm_eps > 0.0)) return bad("rope_theta must be > 1 and norm_eps > 0");
      d.batch = 1;
      d.seq = d.tokens;
      d.causal = 1;
      d.scale = 1.0 / std::sqrt(128.0);
      const double T = (double)d.tokens, H = (double)d.hidden, I = (double)d.inter, D = 128.0;
      const double hq = d.heads_q * D, hkv = d.heads_kv * D;
      const double pairs = 0.5 * T * (T + 1);
      info.flops = 2.0 * T * H * (hq + 2 * hkv)      // QKV projection
                   + 4.0 * D * d.heads_q * pairs      // causal attention (QK^T and PV)
                   + 2.0 * T * hq * H                 // O projection
                   + 6.0 * T * H * I;                 // gate/up and down projections
      info.bytes = 2.0 * (2.0 * T * H + 2.0 * H + H * (hq + 2 * hkv) + H * hq + 3.0 * H * I);
      info.bound = info.flops / info.bytes >= ridge ? RC_BOUND_TENSOR : RC_BOUND_HBM;
      info.n_tensors = 8;
      break;
    }
    default:
      return rc_fail(RC_ERR_UNSUPPORTED_OP, "rc_op_describe: unknown op kind %d", d.kind);
  }
  rc_op_s* op = new (std::nothrow) rc_op_s;
  if (!op) return rc_fail(RC_ERR_OOM, "rc_op_describe: out of host memory");
  op->d = d;
  op->n_stages = n_stages_of(d.kind);
  rc_schedule_s p0;
  p0.op_kind = d.kind;
  p0.n_stages = op->n_stages;
  for (int i = 0; i < op->n_stages; ++i) p0.k[i] = rc_default_knobs(op, i);
  info.workspace_bytes = (int64_t)rc_workspace_bytes(op, &p0);
  op->info = info;
  *out = op;
  return RC_OK;
}

extern "C" rc_status rc_op_info(const rc_op* op, rc_op_info_t* info) {
  if (!op || !info) return rc_fail(RC_ERR_INVALID_ARG, "rc_op_info: NULL argument");
  *info = op->info;
  return RC_OK;
}

// rc_op_destroy lives in run.cu (it frees device memory).

// -------------------------------------------------------------- schedules --
// Whether stage `g` of schedule s runs a memory-bound pass whose access width is the Vectorize knob.
static bool vectorize_used(const rc_op_s* op, const rc_schedule_s& s, int g) {
  const rc_knobs& k = s.k[g];
  switch (op->d.kind) {
    case RC_OP_LINEAR: return k.split_k > 1;
    case RC_OP_SWIGLU: return !k.fuse;
    case RC_OP_MLP: return g == 0 ? !k.fuse : k.split_k > 1;
    case RC_OP_CONV2D: return k.split_k > 1 || (!k.fuse && (op->d.flags & (RC_EPI_BIAS | RC_EPI_SILU)));
    case RC_OP_MOE: return g == 0 ? s.k[1].location == 0 : g == 2;
    case RC_OP_DECODER_LAYER: return g == 4 && !k.fuse;
    default: return false;
  }
}

static rc_status apply_one(const rc_op_s* op, rc_schedule_s* s, const rc_transform& t) {
  if (t.stage < 0 || t.stage >= s->n_stages)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "transform stage %d out of range", t.stage);
  if (t.reserved != 0) return rc_fail(RC_ERR_INVALID_ARG, "rc_transform.reserved must be 0");
  rc_knobs& k = s->k[t.stage];
  const int32_t v = (int32_t)t.value[0];
  if ((int64_t)v != t.value[0]) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "transform value out of range");
  switch (t.kind) {
    case RC_T_TILE_SIZE:
      if (t.axis == 0) k.tile_m = v;
      else if (t.axis == 1) k.tile_n = v;
      else if (t.axis == 2) k.tile_k = v;
      else return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "TileSize axis %d", t.axis);
      break;
    case RC_T_PARALLEL: k.persistent = v; break;
    case RC_T_COMPUTE_LOCATION: k.location = v; break;
    case RC_T_UNROLL: k.unroll = v; break;
    case RC_T_LOOP_ORDER:
      k.raster = v;
      k.group = t.value[1] > 0 ? (int32_t)t.value[1] : 1;
      break;
    case RC_T_FUSE: k.fuse = v; break;
    case RC_T_LAYOUT: k.layout = v; break;
    case RC_T_VECTORIZE: k.vec = v; break;
    case RC_T_PIPELINE_STAGES: k.stages = v; break;
    case RC_T_SPLIT_K: k.split_k = v; break;
    default: return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "unknown transform kind %d", t.kind);
  }
  (void)op;
  return RC_OK;
}

extern "C" rc_status rc_schedule_apply(const rc_op* op, const rc_schedule* base, const rc_transform* seq,
                                       size_t n, rc_schedule** out) {
  if (!op || !out || (n && !seq)) return rc_fail(RC_ERR_INVALID_ARG, "rc_schedule_apply: NULL argument");
  *out = nullptr;
  rc_schedule_s s;
  memset(&s, 0, sizeof s);
  if (base) {
    if (base->op_kind != op->d.kind || base->n_stages != op->n_stages)
      return rc_fail(RC_ERR_INVALID_ARG, "rc_schedule_apply: base schedule belongs to another op kind");
    s = *base;
  } else {
    s.op_kind = op->d.kind;
    s.n_stages = op->n_stages;
    for (int i = 0; i < op->n_stages; ++i) s.k[i] = rc_default_knobs(op, i);
  }
  for (size_t i = 0; i < n; ++i) RC_TRY(apply_one(op, &s, seq[i]));
  // Vectorize acts only on the memory-bound pass a stage runs; where the chosen knobs run none it
  // leaves the program unchanged, so the canonical form keeps the default
  for (int i = 0; i < s.n_stages; ++i)
    if (!vectorize_used(op, s, i)) s.k[i].vec = rc_default_knobs(op, i).vec;
  // MoE grouped GEMMs: splitting ragged segments (layout 1) applies to CTA-pair launches only
  if (op->d.kind == RC_OP_MOE)
    for (int i = 1; i < s.n_stages; ++i)
      if (s.k[i].layout == 1 && s.k[i].tile_m != 256) s.k[i].layout = 0;
  // attention: the one-issuing-warp kernel keeps P in shared memory and one S buffer, the
  // split-issue kernels keep P in tensor memory, and the two-query-tile kernel has a single form,
  // so each family's canonical form fixes the knobs it does not offer (a single Parallel or
  // TileSize transformation then moves between the families)
  for (int i = 0; i < s.n_stages; ++i) {
    if (!(op->d.kind == RC_OP_ATTENTION || (op->d.kind == RC_OP_DECODER_LAYER && i == 2))) continue;
    rc_knobs& k = s.k[i];
    if (k.tile_m == 256) {  // two query tiles per CTA: one kernel, whatever the other families' knobs
      k.tile_n = 128;
      k.persistent = 1;
      k.location = 1;
      k.unroll = 1;
    } else if (k.persistent == 0) {
      k.location = 0;
      k.unroll = 1;
    } else if (k.location == 0) {
      k.location = 1;
    }
  }
  for (int i = 0; i < s.n_stages; ++i) {
    std::string why;
    if (!rc_knobs_legal(op, i, s.k[i], &why))
      return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "stage %d: %s", i, why.c_str());
  }
  rc_schedule_s* r = new (std::nothrow) rc_schedule_s(s);
  if (!r) return rc_fail(RC_ERR_OOM, "rc_schedule_apply: out of host memory");
  *out = r;
  return RC_OK;
}

extern "C" rc_status rc_schedule_knobs(const rc_schedule* s, int32_t stage, rc_knobs* out) {
  if (!s || !out) return rc_fail(RC_ERR_INVALID_ARG, "rc_schedule_knobs: NULL argument");
  if (stage < 0 || stage >= s->n_stages) return rc_fail(RC_ERR_INVALID_ARG, "stage out of range");
  *out = s->k[stage];
  return RC_OK;
}

extern "C" int32_t rc_schedule_num_stages(const rc_schedule* s) { return s ? s->n_stages : 0; }

extern "C" uint64_t rc_schedule_hash(const rc_schedule* s) {
  if (!s) return 0;
  // FNV-1a over the op kind and the canonical knob vectors
  uint64_t h = 1469598103934665603ull;
  auto mixin = [&](int32_t v) {
    for (int b = 0; b < 4; ++b) {
      h ^= (uint64_t)((v >> (8 * b)) & 0xFF);
      h *= 1099511628211ull;
    }
  };
  mixin(s->op_kind);
  mixin(s->n_stages);
  for (int i = 0; i < s->n_stages; ++i) {
    const rc_knobs& k = s->k[i];
    for (int32_t v : {k.tile_m, k.tile_n, k.tile_k, k.unroll, k.stages, k.split_k, k.raster, k.group,
                      k.persistent, k.fuse, k.layout, k.vec, k.location})
      mixin(v);
  }
  return h;
}

extern "C" rc_status rc_schedule_to_string(const rc_schedule* s, char* buf, size_t cap, size_t* needed) {
  if (!s) return rc_fail(RC_ERR_INVALID_ARG, "rc_schedule_to_string: NULL schedule");
  std::string out = std::string("op=") + kind_name(s->op_kind);
  char tmp[256];
  for (int i = 0; i < s->n_stages; ++i) {
    const rc_knobs& k = s->k[i];
    snprintf(tmp, sizeof tmp,
             ";s%d:tile=%dx%dx%d,unroll=%d,stages=%d,split_k=%d,raster=%d/%d,persistent=%d,fuse=%d,"
             "layout=%d,vec=%d,loc=%d",
             i, k.tile_m, k.tile_n, k.tile_k, k.unroll, k.stages, k.split_k, k.raster, k.group,
             k.persistent, k.fuse, k.layout, k.vec, k.location);
    out += tmp;
  }
  if (needed) *needed = out.size() + 1;
  if (buf && cap) {
    size_t n = out.size() < cap - 1 ? out.size() : cap - 1;
    memcpy(buf, out.data(), n);
    buf[n] = 0;
  }
  return RC_OK;
}

extern "C" rc_status rc_schedule_clone(const rc_schedule* s, rc_schedule** out) {
  if (!s || !out) return rc_fail(RC_ERR_INVALID_ARG, "rc_schedule_clone: NULL argument");
  *out = new (std::nothrow) rc_schedule_s(*s);
  return *out ? RC_OK : rc_fail(RC_ERR_OOM, "rc_schedule_clone: out of host memory");
}

extern "C" void rc_schedule_destroy(rc_schedule* s) { delete s; }

extern "C" rc_status rc_transform_space(const rc_op* op, rc_transform* buf, size_t cap, size_t* n) {
  if (!op || !n) return rc_fail(RC_ERR_INVALID_ARG, "rc_transform_space: NULL argument");
  size_t cnt = 0;
  for (int st = 0; st < op->n_stages; ++st) {
    for (const KnobSpec& ks : rc_knob_space(op, st)) {
      const size_t n1 = ks.values1.empty() ? 1 : ks.values1.size();
      if (ks.values.size() * n1 < 2) continue;  // nothing to choose
      for (int32_t v : ks.values) {
        for (size_t j = 0; j < n1; ++j) {
          if (buf && cnt < cap) {
            rc_transform t;
            memset(&t, 0, sizeof t);
            t.kind = ks.tkind;
            t.axis = ks.axis;
            t.stage = st;
            t.value[0] = v;
            if (!ks.values1.empty()) t.value[1] = ks.values1[j];
            buf[cnt] = t;
          }
          ++cnt;
        }
      }
    }
  }
  *n = cnt;
  if (buf && cnt > cap) return rc_fail(RC_ERR_INVALID_ARG, "rc_transform_space: buffer too small");
  return RC_OK;
}
