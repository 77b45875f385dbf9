/*
 * rc.h - C ABI of the schedule-parameterised tensor-program library.
 *
 * The paper (arXiv 2506.01374) states the problem (Sec. 2, Eq. 1) as finding
 * a sequence of at most T semantics-preserving transformations
 * tau_1 .. tau_n that maximises a measured objective f of the transformed
 * program (tau_n o ... o tau_1)(P0). It casts the search as an MDP whose
 * states are programs, whose actions are transformations, whose transition
 * is deterministic and whose reward is s * f (Sec. 2), and solves it with
 * Monte Carlo tree search (Sec. 3.2). This header maps those objects to C:
 *
 *   program P0          -> rc_op        (rc_op_describe)
 *   transformation tau  -> rc_transform (vocabulary of Sec. 3.1 / App. A:
 *                          TileSize, Parallel, ComputeLocation, Unroll, plus
 *                          loop order, fusion, layout, vectorisation,
 *                          pipeline stages and split-K)
 *   transformed program -> rc_schedule  (rc_schedule_apply)
 *   objective f         -> rc_candidate_measure (device-timed throughput)
 *   MCTS                -> rc_search_*  (Sec. 3.2: UCT selection, expansion,
 *                          rollout, backpropagation; measurements only)
 *
 * Conventions for every call:
 *   - Every function returns an rc_status and never aborts the process. On
 *     failure a message is stored in thread-local storage (rc_last_error).
 *   - Handles (rc_op, rc_schedule, rc_search) are owned by the library and
 *     freed by the matching rc_*_destroy; destroying NULL is a no-op.
 *   - Tensors are caller-owned CUDA device pointers (except rc_run_host),
 *     row-major and contiguous, 16-byte aligned; a NULL or misaligned
 *     required pointer gives RC_ERR_INVALID_ARG.
 *   - bf16 tensors hold IEEE bfloat16 bit patterns; all fp32 -> bf16
 *     conversions round to nearest even.
 *   - Kernels run on the caller's CUDA stream (cudaStream_t passed as
 *     void*; NULL = legacy default stream) and return without synchronising
 *     unless stated otherwise.
 *   - Device waits inside kernels are bounded; a wait that gives up sets a
 *     device status word and the call that observes it returns
 *     RC_ERR_DEVICE_TIMEOUT (the CUDA context stays usable).
 */
#ifndef RC_H
#define RC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RC_OK = 0,
  RC_ERR_INVALID_ARG = 1,      /* bad pointer, size, alignment or handle */
  RC_ERR_UNSUPPORTED_OP = 2,   /* op kind or shape this library cannot run */
  RC_ERR_ILLEGAL_SCHEDULE = 3, /* transformation not legal for this op */
  RC_ERR_DUPLICATE = 4,        /* program already in the search tree (Sec. 3.2 acyclicity) */
  RC_ERR_CUDA = 5,             /* a CUDA runtime/driver call failed (message has the code) */
  RC_ERR_DEVICE_TIMEOUT = 6,   /* a bounded device wait gave up */
  RC_ERR_TIMEOUT = 7,          /* host wall-clock budget of a measurement exceeded */
  RC_ERR_PARITY = 8,           /* optional correctness check of a candidate failed */
  RC_ERR_OOM = 9,              /* device or host allocation failed */
  RC_ERR_EXHAUSTED = 10        /* search has no unexplored legal program left */
} rc_status;

/* ------------------------------------------------------------ operators -- */

typedef enum {
  /* C[M,N] = epi(A[M,K] B[K,N] + bias[N]), fp32 in/out, fp32 FFMA (no TF32).
   * epi = ReLU when flags & RC_EPI_RELU. App. A loop nest plus bias/ReLU.
   * tensors: 0 A f32[M][K], 1 B f32[K][N], 2 bias f32[N] (NULL = none), 3 C f32[M][N] */
  RC_OP_GEMM_F32 = 0,
  /* Y[M,N] = X[M,K] W[N,K]^T, bf16 in/out, fp32 accumulate.
   * tensors: 0 X bf16[M][K], 1 W bf16[N][K], 2 Y bf16[M][N] */
  RC_OP_LINEAR = 1,
  /* h[M,I] = silu(X W1[0:I]^T) * (X W1[I:2I]^T), silu(x) = x / (1 + e^-x).
   * n = I. tensors: 0 X bf16[M][K], 1 W1 bf16[2I][K], 2 h bf16[M][I] */
  RC_OP_SWIGLU = 2,
  /* SwiGLU MLP block Y = swiglu(X, W1) W2^T; m = tokens T, k = hidden H, n = I.
   * tensors: 0 X bf16[T][H], 1 W1 bf16[2I][H], 2 W2 bf16[H][I], 3 Y bf16[T][H].
   * The bf16 intermediate h[T][I] lives in library workspace. */
  RC_OP_MLP = 3,
  /* Attention core O = softmax(scale Q K^T + causal mask) V with GQA: query
   * head h reads KV head h / (heads_q / heads_kv). Layout BSHD.
   * tensors: 0 Q bf16[B][S][Hq][D], 1 K bf16[B][S][Hkv][D], 2 V (as K),
   *          3 O bf16[B][S][Hq][D], 4 LSE f32[B][Hq][S] (NULL = not written) */
  RC_OP_ATTENTION = 4,
  /* y = act(conv2d(x, w) + bias), NHWC input/output, KRSC weights, zero pad.
   * act = SiLU when flags & RC_EPI_SILU.
   * tensors: 0 x bf16[N][H][W][Cin], 1 w bf16[Cout][R][S][Cin],
   *          2 bias bf16[Cout] (NULL = none), 3 y bf16[N][P][Q][Cout] */
  RC_OP_CONV2D = 5,
  /* Top-k softmax routing: softmax over E logits, top-k by (logit desc, id
   * asc), weights renormalised over the k when renorm != 0; per-expert counts,
   * exclusive-scan offsets, and the slot permutation ordered by
   * (expert, token, k). Bit-exact ids/offsets/perm.
   * tensors: 0 logits bf16 or f32 [T][E], 1 ids i32[T][k], 2 weights f32[T][k],
   *          3 offsets i32[E+1], 4 perm i32[T*k] (slot s = t*k + j) */
  RC_OP_MOE_ROUTE = 6,
  /* MoE layer: routing as RC_OP_MOE_ROUTE, gather of routed rows, grouped
   * SwiGLU gate/up GEMM, grouped down GEMM, weighted combine
   * out[t] = sum_j w[t,j] Y_{ids[t,j]}(x_t) (fp32 sum in j order).
   * tensors: 0 logits, 1 X bf16[T][H], 2 W1 bf16[E][2I][H], 3 W2 bf16[E][H][I],
   *          4 out bf16[T][H]; optional outputs (NULL = library workspace):
   *          5 ids, 6 weights, 7 offsets, 8 perm (as RC_OP_MOE_ROUTE) */
  RC_OP_MOE = 7,
  /* Pre-norm decoder layer of the Llama family (the paper's end-to-end model,
   * Sec. 4), batch 1, T = tokens positions 0 .. T-1:
   *   a = RMSNorm(x) g1; [q k v] = a Wqkv^T; q, k = RoPE(q, k);
   *   o = causal GQA attention(q, k, v); h1 = x + o Wo^T;
   *   y = h1 + W2 (silu(b Wg^T) * (b Wu^T)), b = RMSNorm(h1) g2,
   * RMSNorm(v) = v / sqrt(mean(v^2) + norm_eps); RoPE turns the pair
   * (j, j + D/2) of each head by p * rope_theta^(-2j/D). head_dim = 128.
   * tokens = T, hidden = H, inter = I, heads_q, heads_kv.
   * tensors: 0 x bf16[T][H], 1 g1 bf16[H], 2 Wqkv bf16[(Hq + 2 Hkv) D][H]
   *          (query rows, then key rows, then value rows), 3 Wo bf16[H][Hq D],
   *          4 g2 bf16[H], 5 W1 bf16[2I][H] (gate rows, then up rows),
   *          6 W2 bf16[H][I], 7 y bf16[T][H].
   * Stages: 0 RMSNorm + QKV GEMM, 1 RoPE (and the split into Q, K, V),
   * 2 attention, 3 O GEMM + residual + RMSNorm, 4 gate/up GEMM + SwiGLU,
   * 5 down GEMM + residual. Intermediates live in library workspace. */
  RC_OP_DECODER_LAYER = 8
} rc_op_kind;

enum { RC_EPI_BIAS = 1, RC_EPI_RELU = 2, RC_EPI_SILU = 4 };

#define RC_MAX_TENSORS 10

typedef struct {
  int32_t kind;   /* rc_op_kind */
  int32_t flags;  /* RC_EPI_* where the op has an epilogue */
  /* GEMM_F32 / LINEAR / SWIGLU / MLP: m rows, n output columns (I for
   * SWIGLU and MLP), k reduction (hidden size H for MLP) */
  int64_t m, n, k;
  /* ATTENTION */
  int64_t batch, seq, heads_q, heads_kv, head_dim;
  int32_t causal;
  double scale;   /* 0 = 1/sqrt(head_dim) */
  /* CONV2D */
  int64_t img_n, img_h, img_w, c_in, c_out, kr, ks, stride, pad;
  /* MOE_ROUTE / MOE: tokens = T, hidden = H, experts = E, inter = I */
  int64_t tokens, hidden, experts, inter, top_k;
  int32_t logits_fp32; /* 0 = bf16 logits, 1 = f32 logits */
  int32_t renorm;      /* 1 = renormalise the k weights (default reading) */
  /* DECODER_LAYER */
  double rope_theta;   /* 0 = 500000 (Llama 3) */
  double norm_eps;     /* 0 = 1e-5 */
} rc_op_desc;

typedef enum { RC_BOUND_TENSOR = 0, RC_BOUND_HBM = 1, RC_BOUND_FP32_SIMT = 2 } rc_bound;

typedef struct {
  double flops;            /* algorithmic flops (2 per multiply-add; causal half for attention) */
  double bytes;            /* algorithmic HBM bytes: each input read once, each output written once */
  int32_t bound;           /* rc_bound at this shape */
  int32_t n_tensors;       /* tensor slots the op uses */
  int64_t workspace_bytes; /* device workspace of the default schedule (library-owned) */
} rc_op_info_t;

typedef struct rc_op_s rc_op;
typedef struct rc_schedule_s rc_schedule;
typedef struct rc_search_s rc_search;

/* Validate desc and create the op P0. Error: RC_ERR_INVALID_ARG (bad sizes),
 * RC_ERR_UNSUPPORTED_OP (shape outside what the kernels handle). */
rc_status rc_op_describe(const rc_op_desc* desc, rc_op** out);
rc_status rc_op_info(const rc_op* op, rc_op_info_t* info);
void rc_op_destroy(rc_op* op);

/* ------------------------------------------------------------ schedules -- */

typedef enum {
  RC_T_TILE_SIZE = 0,        /* axis 0/1/2 = M/N/K tile; value[0] = extent */
  RC_T_PARALLEL = 1,         /* value[0]: GEMM-shaped ops: 0 = one CTA per output tile, 1 = persistent
                              * CTAs; ATTENTION: 0 = one UMMA-issuing warp per CTA, 1 = UMMA issue
                              * split over warps (P in TMEM only): one issuer per query tile for two
                              * tiles, separate S and P V issuers for one tile */
  RC_T_COMPUTE_LOCATION = 2, /* value[0]: where producer work runs (op specific, see knobs);
                              * ATTENTION: 1 = P kept in TMEM, 0 = P in shared memory */
  RC_T_UNROLL = 3,           /* value[0]: unroll factor of the innermost reduction loop;
                              * ATTENTION: key blocks in flight per query tile (1 or 2 S buffers);
                              * one tile with split issue and one S buffer at key blocks of 64
                              * runs two CTAs per SM */
  RC_T_LOOP_ORDER = 4,       /* value[0]: tile raster 0 = M fastest, 1 = N fastest; value[1] = group */
  RC_T_FUSE = 5,             /* value[0]: 1 = epilogue fused into the producing kernel, 0 = separate pass */
  RC_T_LAYOUT = 6,           /* value[0]: op-specific data layout choice; CONV2D: 0 = implicit zero
                              * padding, 1 and 2 = a padded copy read as one box or as row boxes;
                              * ATTENTION: 1 = V transposed to [d][keys]; MOE stages 1 and 2 (the
                              * grouped GEMMs): 0 = each expert's tokens in M tiles, 1 = CTA-pair
                              * tiles with a segment's short remainder in a second one-CTA launch,
                              * 2 = operand roles exchanged (expert weight rows on UMMA M, the
                              * segment's tokens on N in tiles of whole 16-row units, 32 on a CTA
                              * pair; the N tile knob sets the token tile) */
  RC_T_VECTORIZE = 7,        /* value[0]: bytes per global access in the vectorised passes */
  RC_T_PIPELINE_STAGES = 8,  /* value[0]: depth of the shared-memory operand ring */
  RC_T_SPLIT_K = 9,          /* value[0]: number of reduction splits */
  RC_T_COUNT = 10
} rc_transform_kind;

typedef struct {
  int32_t kind;     /* rc_transform_kind */
  int32_t axis;     /* TILE_SIZE only: 0 = M, 1 = N, 2 = K */
  int32_t stage;    /* which kernel of a composite op the transform targets
                     * (TVM's "block"): MLP 0 = gate/up, 1 = down;
                     * MOE 0 = routing/gather, 1 = grouped gate/up, 2 = grouped down
                     * and combine; every other op has the single stage 0 */
  int32_t reserved; /* must be 0 */
  int64_t value[4]; /* value[0] = new knob value (LOOP_ORDER: value[1] = group) */
} rc_transform;

/* The canonical form of a schedule: one knob vector per stage. Applying a
 * transformation sets one knob of one stage; a sequence therefore
 * canonicalises to the knob vectors of its last writers. */
typedef struct {
  int32_t tile_m, tile_n, tile_k;
  int32_t unroll;
  int32_t stages;
  int32_t split_k;
  int32_t raster, group;
  int32_t persistent;
  int32_t fuse;
  int32_t layout;
  int32_t vec;
  int32_t location;
} rc_knobs;

/* (tau_n o ... o tau_1)(base), base = NULL means P0 (the op's default
 * schedule). The result is checked for legality (tile divisibility or
 * supported ragged tails, shared memory <= 227 KB per CTA, TMEM <= 512
 * columns, alignment) and canonicalised. RC_ERR_ILLEGAL_SCHEDULE when any
 * step or the result is illegal; *out is then NULL. */
rc_status rc_schedule_apply(const rc_op* op, const rc_schedule* base, const rc_transform* seq,
                            size_t n, rc_schedule** out);
#define RC_MAX_STAGES 6
/* Number of stages of the op the schedule belongs to, and one stage's knobs. */
rc_status rc_schedule_knobs(const rc_schedule* s, int32_t stage, rc_knobs* out);
int32_t rc_schedule_num_stages(const rc_schedule* s);
uint64_t rc_schedule_hash(const rc_schedule* s); /* hash of the canonical knob vector */
/* Canonical text "op=...;tile=MxNxK;stages=...". Writes at most cap bytes
 * (NUL included) and reports the needed size. */
rc_status rc_schedule_to_string(const rc_schedule* s, char* buf, size_t cap, size_t* needed);
rc_status rc_schedule_clone(const rc_schedule* s, rc_schedule** out);
void rc_schedule_destroy(rc_schedule* s);

/* Every single transformation this op's space offers (whether it is legal
 * from a given schedule is decided by rc_schedule_apply). */
rc_status rc_transform_space(const rc_op* op, rc_transform* buf, size_t cap, size_t* n);

/* --------------------------------------------------------- execution -- */

typedef struct {
  void* p[RC_MAX_TENSORS]; /* slots as documented per rc_op_kind */
} rc_tensors;

/* Run the op once under schedule s on the stream. Library workspace is
 * allocated on first use and cached in the op (not thread safe per op). */
rc_status rc_run(const rc_op* op, const rc_schedule* s, const rc_tensors* io, void* stream);

/* rc_run with CUDA events recorded between the op's stages (MLP: gate/up,
 * down; MOE: routing+gather, grouped gate/up, grouped down+combine; other
 * ops: one stage). Synchronises the stream; stage_ms[i] = device time of
 * stage i in milliseconds; *n_stages = stages written (<= cap). */
rc_status rc_run_profiled(const rc_op* op, const rc_schedule* s, const rc_tensors* io, void* stream,
                          double* stage_ms, size_t cap, size_t* n_stages);

/* End-to-end form of rc_run: io holds HOST pointers. Inputs are copied to
 * device staging buffers owned by the op, the op runs, outputs are copied
 * back, and the stream is synchronised before returning. Host buffers
 * should be pinned for full copy bandwidth. */
rc_status rc_run_host(const rc_op* op, const rc_schedule* s, const rc_tensors* host_io,
                      void* stream);

/* Synchronise the stream and report device-side failures of earlier runs of
 * this op (RC_ERR_DEVICE_TIMEOUT when a bounded wait gave up; the status
 * word is cleared). */
rc_status rc_op_check(const rc_op* op, void* stream);

/* Self-test of the bounded device waits (no paper counterpart): one CTA
 * waits on an mbarrier phase that nothing completes, with a wait limit of
 * wait_ms (0 < wait_ms <= 2000). The wait gives up, records a timeout in a
 * device status word and the call returns RC_ERR_DEVICE_TIMEOUT after
 * synchronising `stream`; RC_OK would mean the wait did not give up. The
 * CUDA context stays usable. Allocates and frees a 4-byte status word. */
rc_status rc_selftest_bounded_wait(double wait_ms, void* stream);

/* ---------------------------------------------------------- measurement -- */

typedef struct {
  int32_t warmup;     /* untimed runs per candidate (default 5) */
  int32_t repeats;    /* timed runs per candidate (default 20, as in the paper's 20 repetitions) */
  int32_t flush_l2;   /* 1 = write a buffer of 2x L2 before every timed run (default 1) */
  double budget_s;    /* host wall-clock budget for the whole batch, 0 = none */
} rc_measure_opts;

typedef struct {
  int32_t status;     /* rc_status of this candidate (illegal/failed -> non-zero) */
  double ms_median, ms_min, ms_mean;
  double tflops;      /* algorithmic flops / median time */
  double gbps;        /* algorithmic bytes / median time */
  uint64_t sched_hash;
  int32_t n_stages;                 /* stages timed separately (0 = none) */
  double stage_ms[RC_MAX_STAGES];   /* median device time of each stage (ms) */
} rc_measurement;

/* Device-timed measurement of n candidates on the caller's stream: per
 * candidate W warm-ups, then R x {L2 flush, event, run with an event after
 * each stage}; medians of the whole run and of each stage.
 * out[] is caller-allocated. The call synchronises the stream. The batch
 * status is RC_OK if every candidate could be attempted; per-candidate
 * failures are reported in out[i].status. */
rc_status rc_candidate_measure(const rc_op* op, const rc_schedule* const* cands, size_t n,
                               const rc_tensors* io, void* stream, const rc_measure_opts* opts,
                               rc_measurement* out);

/* --------------------------------------------------------------- search -- */

typedef struct {
  uint64_t seed;      /* seeds the counter-based expansion/rollout generator */
  double c;           /* UCT exploration constant (paper: sqrt(2)) */
  int32_t branching;  /* children per expansion B (paper: 2) */
  int32_t horizon;    /* maximum transformation-sequence length T (default 8) */
  int32_t rollout;    /* random transformations per rollout q (default 2) */
  int32_t max_tries;  /* sampling attempts per expansion (default 64) */
  int32_t surrogate;  /* 0 (default): rollout programs are measured; 1: once >= 24 programs are
                       * measured, rollout programs are scored by a surrogate f-hat learned from the
                       * measurements (Sec. 3.2: reward = t(P0) / f-hat(P_sim)) and only expanded
                       * nodes are measured. f-hat: ridge regression of log device time on one-hot
                       * knob values and knob-pair values, one model per op stage when the
                       * measurements carry per-stage times. */
  int32_t screen;     /* surrogate = 1 only: an expansion draws up to screen * B distinct legal
                       * proposals and keeps the B with the lowest predicted time (the cost model
                       * pruning low-value proposals before they join the tree); <= 1 = off */
  uint32_t stage_mask; /* 0 (default): every stage of the op may be transformed and the objective
                        * is the op's device time. Else only transformations of the stages whose
                        * bit is set are proposed, and the objective is the sum of those stages'
                        * medians (rc_measurement.stage_ms; the whole time where a measurement has
                        * no per-stage times): one task of a composite op tuned on its own, as a
                        * compiler tunes the subgraphs of a network one by one */
  const rc_schedule* root; /* NULL (default): the search starts from P0. Else from this program of
                            * the same op (copied; the caller keeps ownership), and rewards are
                            * speedups over it: a later task's search starts from the best program
                            * of the earlier ones. A schedule of another op is RC_ERR_INVALID_ARG */
} rc_search_opts;

/* Create an LLM-free MCTS search over op's schedule space (Sec. 3.2 with the
 * random-valid expansion policy the paper falls back to, App. G). opts NULL
 * = defaults. The first rc_search_step call returns the root (P0, or opts->root)
 * to measure. */
rc_status rc_search_create(const rc_op* op, const rc_search_opts* opts, rc_search** out);

/* One search iteration. results[0..n_results) are the measurements of the
 * schedules returned by the previous call, in the same order (a reward of
 * median-time(P0) / median-time(candidate); a failed candidate gets 0).
 * The call backpropagates them, then selects by UCT, expands, draws
 * rollouts and returns up to cap schedules to measure next in next[]
 * (owned by the search, valid until it is destroyed). *n_next = 0 with
 * RC_ERR_EXHAUSTED when nothing unmeasured remains. */
rc_status rc_search_step(rc_search* s, const rc_measurement* results, size_t n_results,
                         const rc_schedule** next, size_t cap, size_t* n_next);

/* Best measured schedule so far (owned by the search) and its measurement. */
rc_status rc_search_best(const rc_search* s, const rc_schedule** best, rc_measurement* m);

/* Introspection for tests and logs. */
typedef struct {
  int64_t nodes;        /* nodes in the tree */
  int64_t samples;      /* distinct schedules measured */
  int64_t iterations;   /* rc_search_step calls that expanded */
  double best_reward;
  int64_t model_samples;   /* measurements the current surrogate fit used (0 = not fitted) */
  int64_t model_features;  /* columns of the current fit, intercept included */
  int64_t predicted;       /* rollout rewards taken from the surrogate */
} rc_search_stats;
rc_status rc_search_get_stats(const rc_search* s, rc_search_stats* st);
/* The surrogate's predicted device time (ms) of a schedule of the search's
 * op: the sum over stages of exp(w . x_stage) (per-stage models; with a
 * stage_mask, over the selected stages only: the search's objective) or
 * exp(w . x) (one model). RC_ERR_INVALID_ARG when the surrogate is off or not
 * fitted yet. Deterministic given the measurement sequence. */
rc_status rc_search_predict(rc_search* s, const rc_schedule* sched, double* ms);
/* Node i (0 = root): parent index (-1 for root), Q (cumulative reward), N (visits). */
rc_status rc_search_node(const rc_search* s, int64_t i, int64_t* parent, double* q, int64_t* n,
                         uint64_t* sched_hash);
void rc_search_destroy(rc_search* s);

/* ------------------------------------------------- no-allocation routing -- */

/* The paper has no counterpart to this entry point; it exists for callers
 * that cannot allocate device memory. Examples: a process whose GPU memory
 * has been reserved by another allocator (a framework's caching pool), or a
 * latency-critical path where cudaMalloc is off limits because it can
 * synchronise the device and has no time bound.
 *
 * It computes exactly what rc_run does for an RC_OP_MOE_ROUTE op with
 * renorm/logits_fp32 as given (same kernels, same bit-exact ids, offsets and
 * permutation), but allocates nothing: the per-expert counts it needs live
 * in a fixed device array of RC_NOALLOC_MAX_EXPERTS ints inside the library,
 * which every GPU that loads the library keeps until the process exits.
 *
 *   logits  : device bf16 (logits_fp32 = 0) or f32 [tokens][experts]
 *   ids     : device i32 [tokens][top_k]      (output)
 *   weights : device f32 [tokens][top_k]      (output)
 *   offsets : device i32 [experts + 1]        (output)
 *   perm    : device i32 [tokens * top_k]     (output, slot s = t*top_k + j)
 * All tensors are caller-owned and 16-byte aligned. experts above
 * RC_NOALLOC_MAX_EXPERTS gives RC_ERR_INVALID_ARG; top_k above 16 gives
 * RC_ERR_UNSUPPORTED_OP. Kernels are queued on `stream` (no synchronisation).
 *
 * The first call on each device looks up the array's device address with
 * that device current (cudaGetSymbolAddress); make that first call before
 * any stream capture. Every call on a device shares the one array, so calls
 * whose kernels overlap on the GPU (different streams, no ordering) race;
 * order them on one stream or with events. The array keeps the last call's
 * counts; each call first zeroes the entries it uses (cudaMemsetAsync on
 * `stream`), then the count kernel adds to them with atomicAdd, so the
 * caller never clears it. The cached address is looked up again when the
 * device's context changes (after cudaDeviceReset). A NaN logit ranks below
 * every number, as in rc_run. */
#define RC_NOALLOC_MAX_EXPERTS 256
rc_status rc_moe_route_noalloc(const void* logits, int32_t logits_fp32, int64_t tokens, int64_t experts,
                               int64_t top_k, int32_t renorm, int32_t* ids, float* weights, int32_t* offsets,
                               int32_t* perm, void* stream);

/* Thread-local message of the last failing call on this thread. */
const char* rc_last_error(void);
/* Library version string. */
const char* rc_version(void);

#ifdef __cplusplus
}
#endif
#endif /* RC_H */
