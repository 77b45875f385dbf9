// Internal declarations shared by the host-side C++ and the CUDA translation
// units of librc. Not part of the public ABI (include/rc.h is).
#pragma once

#include <cstdarg>
#include <cstddef>
#include <cstdint>
#include <string>
#include <vector>

#include "rc.h"

// ------------------------------------------------------------------ errors --
rc_status rc_fail(rc_status st, const char* fmt, ...);
void rc_clear_error();

#define RC_TRY(expr)                      \
  do {                                    \
    rc_status _st = (expr);               \
    if (_st != RC_OK) return _st;         \
  } while (0)

// Device status words (written by kernels whose bounded waits gave up).
enum {
  RC_DEV_OK = 0,
  RC_DEV_TIMEOUT_FULL = 1,   // MMA issuer gave up waiting for a TMA stage
  RC_DEV_TIMEOUT_EMPTY = 2,  // producer gave up waiting for a free stage
  RC_DEV_TIMEOUT_ACCUM = 3,  // epilogue gave up waiting for the accumulator
  RC_DEV_TIMEOUT_DRAIN = 4,  // teardown gave up waiting for in-flight copies / MMAs
  RC_DEV_BAD_ARG = 5,        // a kernel-side argument check failed
  RC_DEV_MISALIGNED = 6      // dynamic shared memory not at the alignment a packed layout needs
};

// ------------------------------------------------------------------ ops --
struct rc_op_s {
  rc_op_desc d;
  rc_op_info_t info;
  int n_stages;
  // library-owned device memory, allocated on first use and freed by
  // rc_op_destroy: workspace for intermediates, staging for rc_run_host,
  // and one int status word written by kernels.
  mutable void* ws = nullptr;
  mutable size_t ws_bytes = 0;
  mutable void* stage_buf[RC_MAX_TENSORS] = {};
  mutable size_t stage_bytes[RC_MAX_TENSORS] = {};
  // rc_run_host: a copy stream for inputs of later stages, and per stage an
  // event recorded when that stage's inputs have landed
  mutable void* copy_stream = nullptr;
  mutable void* input_ready[RC_MAX_STAGES] = {};
  mutable void* first_inputs_done = nullptr;
  mutable int* d_status = nullptr;
  mutable int device = -1;
};

struct rc_schedule_s {
  int32_t op_kind;
  int32_t n_stages;
  rc_knobs k[RC_MAX_STAGES];
};

// One tunable knob of one stage: the transform that sets it and its legal values.
struct KnobSpec {
  int32_t tkind;                  // rc_transform_kind
  int32_t axis;                   // TILE_SIZE axis, else 0
  std::vector<int32_t> values;    // legal values of value[0]
  std::vector<int32_t> values1;   // LOOP_ORDER: legal groups (value[1])
};

std::vector<KnobSpec> rc_knob_space(const rc_op_s* op, int stage);
rc_knobs rc_default_knobs(const rc_op_s* op, int stage);
// Checks resource and shape legality of one stage's knob vector.
bool rc_knobs_legal(const rc_op_s* op, int stage, const rc_knobs& k, std::string* why);

// Tensor slot descriptions: bytes of each slot and whether it is an input,
// an output or optional. Used for validation and rc_run_host staging.
struct SlotInfo {
  size_t bytes;
  bool input;
  bool output;
  bool optional;
  int first_stage = 0;  // inputs: the first stage of the op that reads the slot
};
std::vector<SlotInfo> rc_slots(const rc_op_s* op);

// Device workspace bytes a schedule needs (intermediates, split-K partials).
size_t rc_workspace_bytes(const rc_op_s* op, const rc_schedule_s* s);

// ----------------------------------------------------------- launchers --
// Every launcher validates what it needs and returns a status; none
// synchronises. `status` is the op's device status word.
struct LaunchCtx {
  void* stream;
  int* status;
  int num_sms;
  // optional stage markers (rc_run_profiled): event i is recorded after stage i
  void** stage_events = nullptr;
  int n_stage_events = 0;
  mutable int next_event = 0;
  // optional (rc_run_host): before stage i > 0 runs, the stream waits on
  // stage_inputs[i] (NULL = nothing to wait for)
  void* const* stage_inputs = nullptr;
  mutable int stages_done = 0;
};
// End of a stage: record the next stage marker, if markers were requested, and
// make the stream wait for the next stage's inputs, if given.
rc_status rc_mark_stage(const LaunchCtx& c);

rc_status rc_launch_gemm_f32(const rc_knobs& k, int64_t M, int64_t N, int64_t K, const float* A,
                             const float* B, const float* bias, float* C, bool relu,
                             const LaunchCtx& c);

// Dense bf16 tensor-core GEMM family (tcgen05 + TMA): D = A B^T with A[M][K],
// B[N][K] K-major, fp32 accumulate in tensor memory.
enum TcEpilogue {
  TC_EPI_STORE_BF16 = 0,   // D -> bf16
  TC_EPI_SWIGLU = 1,       // D holds [gate | up] column halves -> silu(g)*u bf16
  TC_EPI_PARTIAL_F32 = 2,  // D -> fp32 partial (split-K), slice z at z*M*ldc
  TC_EPI_BIAS_SILU = 3,    // D + bias[n] -> silu -> bf16
  TC_EPI_SCALE_ATOMIC = 4  // row_scale[row] * D atomically added to fp32 out[row_map[row]]
};
// Which rows of each grouped segment a launch covers (see seg_rows in tc_gemm.cuh).
enum TcSegMode {
  TC_SEG_ALL = 0,    // every row, in tiles of the launch's M tile
  TC_SEG_PAIRS = 1,  // a CTA-pair launch: the segment minus a last remainder of 1 .. 128 rows
  TC_SEG_REST = 2    // a one-CTA launch: that remainder alone (one 128-row tile per segment at most)
};
enum TcAMode {
  TC_A_2D = 0,         // A is a row-major [M][K] matrix
  TC_A_CONV = 1,       // A rows are output pixels of an NHWC 'same' conv; K = (r, s, c); one 4-D box
  TC_A_CONV_ROWS = 2,  // as TC_A_CONV over an explicitly padded input, one 2-D box per image row
  TC_A_GATHER = 3      // grouped only: A row i is row row_map[i] / row_div of a [a_rows][K] matrix
};
struct TcGemmArgs {
  int64_t M, N, K;         // N = UMMA columns of the whole problem (2I for SwiGLU)
  const void* A;           // bf16
  const void* B;           // bf16 [N][K] (SwiGLU: [2I][K], gate rows then up rows)
  void* D;                 // output
  int64_t ldd;             // output row stride in elements
  int epilogue;            // TcEpilogue
  int a_mode;              // TcAMode
  const void* bias;        // TC_EPI_BIAS_SILU: bf16[N] (NULL = no bias)
  int silu;                // TC_EPI_BIAS_SILU: 1 = apply SiLU after the bias
  // conv geometry (TC_A_CONV); padded = 1: A is an explicitly padded copy
  // [N][H+2pad][W+2pad][C] read without out-of-range coordinates
  int64_t img_n, img_h, img_w, c_in, kr, ks, pad;
  int padded;
  // grouped (MoE) mode: groups > 0 means rows of A are partitioned into
  // `groups` segments by offsets[g] (device int32[groups+1]); segment g uses
  // B rows [g*b_group_rows, (g+1)*b_group_rows).
  int groups;
  const int* offsets;
  int64_t b_group_rows;
  int64_t max_tiles_m;     // upper bound on m-tiles over all groups
  int seg_mode;            // TcSegMode
  const float* row_scale;  // TC_EPI_SCALE_ATOMIC
  const int* row_map;      // TC_EPI_SCALE_ATOMIC: A row -> slot; output row = slot / row_div
  int row_div;             // (TC_A_GATHER: A row i is source row row_map[i] / row_div)
  int64_t a_rows;          // TC_A_GATHER: rows of the source matrix A
  const void* resid;       // TC_EPI_STORE_BF16: bf16 [M][ldd] added to D before the one rounding (NULL = none)
};
rc_status rc_launch_tc_gemm(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);
// Shared memory of one CTA of the tensor-core GEMM (the schedule legality check's figure).
int64_t tc_smem_bytes(int bn_mma, int stages, int tile_k, int tile_m);
// The same for the grouped GEMM with exchanged operand roles (Layout 2: weights on UMMA M, a token
// tile of tn rows on N, split over the two CTAs of a pair).
int64_t tc_t_smem_bytes(int tn, int stages, int tile_k, bool pair);
// Split-K reduction: out_bf16[M][N] = sum_z part[z][M][N].
rc_status rc_launch_splitk_reduce(const float* part, int splits, int64_t M, int64_t N, void* out,
                                  int vec, const LaunchCtx& c);
// Separate epilogue passes (unfused schedules).
rc_status rc_launch_swiglu_pass(const void* gu, int64_t M, int64_t I, void* h, int vec,
                                const LaunchCtx& c);
rc_status rc_launch_bias_silu_pass(const void* y, const void* bias, int64_t rows, int64_t C,
                                   bool silu, void* out, int vec, const LaunchCtx& c);

// L2 flush: writes `bytes` of the scratch buffer.
rc_status rc_launch_l2_flush(void* buf, size_t bytes, void* stream);

// Attention and MoE launchers.
// Attention: workspace holds the transposed V when k.layout == 1.
rc_status rc_launch_attention(const rc_knobs& k, const rc_op_desc& d, const void* Q, const void* K,
                              const void* V, void* O, float* lse, void* workspace, const LaunchCtx& c);
// Routing: counts is device scratch of E ints; inv_perm may be NULL.
rc_status rc_launch_moe_route(const rc_knobs& k, const rc_op_desc& d, const void* logits, int* ids,
                              float* w, int* offsets, int* perm, int* inv_perm, int* counts,
                              const LaunchCtx& c);
rc_status rc_launch_moe_gather(const void* X, const int* perm, int64_t rows, int64_t H, int topk,
                               void* Xp, int vec, const LaunchCtx& c);
rc_status rc_launch_moe_combine(const void* Y, const float* w, const int* inv_perm, int64_t T,
                                int64_t H, int topk, void* out, int vec, const LaunchCtx& c);
rc_status rc_launch_f32_to_bf16(const float* in, int64_t n, void* out, int vec, const LaunchCtx& c);
// Explicitly zero-padded copy of an NHWC tensor ([N][H+2p][W+2p][C]).
rc_status rc_launch_pad_nhwc(const void* x, int64_t N, int64_t H, int64_t W, int64_t C, int64_t pad, void* xp,
                             const LaunchCtx& c);
// Decoder-layer passes (bf16 storage, fp32 arithmetic). RMSNorm of rows[H]:
// y = x / sqrt(mean(x^2) + eps) * g, H % 256 == 0 and H <= 32768.
rc_status rc_launch_rmsnorm(const void* x, const void* g, int64_t rows, int64_t H, double eps, void* y,
                            const LaunchCtx& c);
// qkv[T][(Hq + 2 Hkv) D] -> Q[T][Hq][D], K[T][Hkv][D] (rotate-half RoPE at
// positions 0 .. T-1) and V[T][Hkv][D]; k.tile_m tokens per CTA.
rc_status rc_launch_rope_split(const rc_knobs& k, const void* qkv, int64_t T, int64_t Hq, int64_t Hkv, int64_t D,
                               double theta, void* Q, void* K, void* V, const LaunchCtx& c);
