// Execution and measurement: rc_run dispatches a schedule's knob vectors to
// the kernel variants they select; rc_candidate_measure is the objective f of
// Eq. 1 measured on the device (the paper repeats each experiment 20 times,
// Sec. 4.1; here each candidate gets W warm-ups and R timed runs, each
// preceded by an L2 flush, and the median is reported).
#include <cuda_runtime.h>

#include <algorithm>
#include <chrono>
#include <cstring>
#include <mutex>
#include <vector>

#include "rc_internal.h"

namespace {

struct DevInfo {
  int num_sms = 0;
  size_t l2_bytes = 0;
  void* flush = nullptr;
  size_t flush_bytes = 0;
};
std::mutex g_dev_mu;
DevInfo g_dev[64];

rc_status cuda_err(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return RC_OK;
  if (e == cudaErrorMemoryAllocation) return rc_fail(RC_ERR_OOM, "%s: %s", what, cudaGetErrorString(e));
  return rc_fail(RC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

rc_status dev_info(DevInfo** out, int* device) {
  int d = 0;
  RC_TRY(cuda_err(cudaGetDevice(&d), "cudaGetDevice"));
  if (d < 0 || d >= 64) return rc_fail(RC_ERR_CUDA, "device index %d out of range", d);
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DevInfo& di = g_dev[d];
  if (!di.num_sms) {
    int sms = 0, l2 = 0;
    RC_TRY(cuda_err(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, d), "SM count"));
    RC_TRY(cuda_err(cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, d), "L2 size"));
    di.num_sms = sms;
    di.l2_bytes = (size_t)l2;
  }
  *out = &di;
  *device = d;
  return RC_OK;
}

rc_status ensure_status_word(const rc_op_s* op, int device) {
  if (op->d_status && op->device == device) return RC_OK;
  if (op->d_status) return rc_fail(RC_ERR_INVALID_ARG, "op was first used on device %d, now on %d", op->device, device);
  RC_TRY(cuda_err(cudaMalloc((void**)&op->d_status, 256), "cudaMalloc(status)"));
  RC_TRY(cuda_err(cudaMemset(op->d_status, 0, 256), "cudaMemset(status)"));
  op->device = device;
  return RC_OK;
}

rc_status ensure_ws(const rc_op_s* op, size_t bytes) {
  if (bytes <= op->ws_bytes) return RC_OK;
  if (op->ws) cudaFree(op->ws);
  op->ws = nullptr;
  op->ws_bytes = 0;
  RC_TRY(cuda_err(cudaMalloc(&op->ws, bytes), "cudaMalloc(workspace)"));
  op->ws_bytes = bytes;
  return RC_OK;
}

rc_status check_io(const rc_op_s* op, const rc_tensors* io) {
  if (!io) return rc_fail(RC_ERR_INVALID_ARG, "tensors: NULL");
  const auto slots = rc_slots(op);
  for (size_t i = 0; i < slots.size(); ++i) {
    void* p = io->p[i];
    if (!p) {
      if (slots[i].optional) continue;
      return rc_fail(RC_ERR_INVALID_ARG, "tensor slot %zu is NULL", i);
    }
    if ((uintptr_t)p % 16) return rc_fail(RC_ERR_INVALID_ARG, "tensor slot %zu is not 16-byte aligned", i);
  }
  return RC_OK;
}

size_t a256(size_t x) { return (x + 255) & ~(size_t)255; }

// Split a workspace into consecutive 256-byte aligned pieces.
struct Carve {
  char* p;
  void* take(size_t bytes) {
    void* r = p;
    p += a256(bytes);
    return r;
  }
};

TcGemmArgs gemm_args(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* D, int64_t ldd, int epi) {
  TcGemmArgs a;
  memset(&a, 0, sizeof a);
  a.M = M;
  a.N = N;
  a.K = K;
  a.A = A;
  a.B = B;
  a.D = D;
  a.ldd = ldd;
  a.epilogue = epi;
  a.a_mode = TC_A_2D;
  return a;
}

// A grouped (MoE) GEMM. Layout 1 with CTA pairs splits every expert segment
// whose last pair tile would hold at most 128 rows: one launch of CTA pairs
// over the rest of the segments, then one launch of single CTAs over those
// remainders (one 128-row tile each), so a ragged segment pads at most 127
// rows instead of 255. The remainder launch keeps the knobs but the M tile,
// with as many of the ring stages as fit one CTA's shared memory.
rc_status launch_grouped(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  if (k.layout != 1 || k.tile_m != 256) return rc_launch_tc_gemm(k, a, c);
  TcGemmArgs head = a;
  head.seg_mode = TC_SEG_PAIRS;
  RC_TRY(rc_launch_tc_gemm(k, head, c));
  rc_knobs kr = k;
  kr.tile_m = 128;
  kr.layout = 0;
  const int bn_mma = a.epilogue == TC_EPI_SWIGLU ? 2 * k.tile_n : k.tile_n;
  while (kr.stages > 1 && tc_smem_bytes(bn_mma, kr.stages, kr.tile_k, 128) > 232448) --kr.stages;
  TcGemmArgs rest = a;
  rest.seg_mode = TC_SEG_REST;
  return rc_launch_tc_gemm(kr, rest, c);
}

// Y[M,N] = X W^T with optional split-K through an fp32 partial buffer.
rc_status run_linear(const rc_knobs& k, int64_t M, int64_t N, int64_t K, const void* X, const void* W, void* Y,
                     void* part, const LaunchCtx& c) {
  if (k.split_k > 1) {
    TcGemmArgs a = gemm_args(M, N, K, X, W, part, N, TC_EPI_PARTIAL_F32);
    RC_TRY(rc_launch_tc_gemm(k, a, c));
    return rc_launch_splitk_reduce((const float*)part, k.split_k, M, N, Y, k.vec, c);
  }
  return rc_launch_tc_gemm(k, gemm_args(M, N, K, X, W, Y, N, TC_EPI_STORE_BF16), c);
}

// h[M,I] = silu(X W1[:I]^T) * (X W1[I:]^T); unfused: gu = X W1^T, then a pass.
rc_status run_swiglu(const rc_knobs& k, int64_t M, int64_t I, int64_t K, const void* X, const void* W1, void* h,
                     void* gu, const LaunchCtx& c) {
  if (k.fuse) return rc_launch_tc_gemm(k, gemm_args(M, 2 * I, K, X, W1, h, I, TC_EPI_SWIGLU), c);
  // unfused: the same UMMA shape (N = 2 x the output tile) writes gate|up, then a pass
  rc_knobs kg = k;
  kg.tile_n = 2 * k.tile_n;
  RC_TRY(rc_launch_tc_gemm(kg, gemm_args(M, 2 * I, K, X, W1, gu, 2 * I, TC_EPI_STORE_BF16), c));
  return rc_launch_swiglu_pass(gu, M, I, h, k.vec, c);
}

rc_status run_impl(const rc_op_s* op, const rc_schedule_s* s, const rc_tensors* io, const LaunchCtx& c) {
  const rc_op_desc& d = op->d;
  void* const* p = io->p;
  Carve ws{(char*)op->ws};
  switch (d.kind) {
    case RC_OP_GEMM_F32:
      return rc_launch_gemm_f32(s->k[0], d.m, d.n, d.k, (const float*)p[0], (const float*)p[1],
                                (const float*)p[2], (float*)p[3], (d.flags & RC_EPI_RELU) != 0, c);
    case RC_OP_LINEAR:
      return run_linear(s->k[0], d.m, d.n, d.k, p[0], p[1], p[2], op->ws, c);
    case RC_OP_SWIGLU:
      return run_swiglu(s->k[0], d.m, d.n, d.k, p[0], p[1], p[2], op->ws, c);
    case RC_OP_MLP: {
      void* h = ws.take(2ull * d.m * d.n);
      void* gu = s->k[0].fuse ? nullptr : ws.take(2ull * d.m * 2 * d.n);
      void* part = s->k[1].split_k > 1 ? ws.take(4ull * s->k[1].split_k * d.m * d.k) : nullptr;
      RC_TRY(run_swiglu(s->k[0], d.m, d.n, d.k, p[0], p[1], h, gu, c));
      RC_TRY(rc_mark_stage(c));
      RC_TRY(run_linear(s->k[1], d.m, d.k, d.n, h, p[2], p[3], part, c));
      return rc_mark_stage(c);
    }
    case RC_OP_CONV2D: {
      const rc_knobs& k = s->k[0];
      const int64_t rows = d.img_n * d.img_h * d.img_w;
      const int64_t K = d.kr * d.ks * d.c_in;
      TcGemmArgs a = gemm_args(rows, d.c_out, K, p[0], p[1], p[3], d.c_out, TC_EPI_STORE_BF16);
      a.a_mode = TC_A_CONV;
      a.img_n = d.img_n;
      a.img_h = d.img_h;
      a.img_w = d.img_w;
      a.c_in = d.c_in;
      a.kr = d.kr;
      a.ks = d.ks;
      a.pad = d.pad;
      a.bias = p[2];
      if (k.layout >= 1) {
        // layouts 1 and 2: explicitly zero-padded copy of x, read without out-of-range
        // TMA coordinates, as one 4-D box (1) or one 2-D box per image row (2)
        void* xp = ws.take(2ull * d.img_n * (d.img_h + 2 * d.pad) * (d.img_w + 2 * d.pad) * d.c_in);
        RC_TRY(rc_launch_pad_nhwc(p[0], d.img_n, d.img_h, d.img_w, d.c_in, d.pad, xp, c));
        a.A = xp;
        a.padded = 1;
        if (k.layout == 2) a.a_mode = TC_A_CONV_ROWS;
      }
      const bool silu = (d.flags & RC_EPI_SILU) != 0;
      if (k.split_k > 1) {
        void* part = ws.take(4ull * k.split_k * rows * d.c_out);
        void* y = ws.take(2ull * rows * d.c_out);
        a.D = part;
        a.epilogue = TC_EPI_PARTIAL_F32;
        RC_TRY(rc_launch_tc_gemm(k, a, c));
        RC_TRY(rc_launch_splitk_reduce((const float*)part, k.split_k, rows, d.c_out, y, k.vec, c));
        return rc_launch_bias_silu_pass(y, p[2], rows, d.c_out, silu, p[3], k.vec, c);
      }
      if (k.fuse && (silu || p[2])) {
        a.epilogue = TC_EPI_BIAS_SILU;
        a.silu = silu ? 1 : 0;
        return rc_launch_tc_gemm(k, a, c);
      }
      if (!silu && !p[2]) return rc_launch_tc_gemm(k, a, c);
      void* y = ws.take(2ull * rows * d.c_out);
      a.D = y;
      RC_TRY(rc_launch_tc_gemm(k, a, c));
      return rc_launch_bias_silu_pass(y, p[2], rows, d.c_out, silu, p[3], k.vec, c);
    }
    case RC_OP_ATTENTION:
      return rc_launch_attention(s->k[0], d, p[0], p[1], p[2], p[3], (float*)p[4], op->ws, c);
    case RC_OP_DECODER_LAYER: {
      const int64_t T = d.tokens, H = d.hidden, I = d.inter, D = d.head_dim;
      const int64_t hq = d.heads_q * D, hkv = d.heads_kv * D, nqkv = hq + 2 * hkv;
      void* a = ws.take(2ull * T * H);
      void* qkv = ws.take(2ull * T * nqkv);
      void* Q = ws.take(2ull * T * hq);
      void* K = ws.take(2ull * T * hkv);
      void* V = ws.take(2ull * T * hkv);
      void* O = ws.take(2ull * T * hq);
      void* h1 = ws.take(2ull * T * H);
      void* b = ws.take(2ull * T * H);
      void* hb = ws.take(2ull * T * I);
      void* gu = s->k[4].fuse ? nullptr : ws.take(2ull * T * 2 * I);
      void* vt = s->k[2].layout == 1 ? ws.take(2ull * hkv * T) : nullptr;
      // 0: a = RMSNorm(x) g1, qkv = a Wqkv^T
      RC_TRY(rc_launch_rmsnorm(p[0], p[1], T, H, d.norm_eps, a, c));
      RC_TRY(run_linear(s->k[0], T, nqkv, H, a, p[2], qkv, nullptr, c));
      RC_TRY(rc_mark_stage(c));
      // 1: RoPE on q and k, split into contiguous heads
      RC_TRY(rc_launch_rope_split(s->k[1], qkv, T, d.heads_q, d.heads_kv, D, d.rope_theta, Q, K, V, c));
      RC_TRY(rc_mark_stage(c));
      // 2: causal GQA attention over the T positions
      RC_TRY(rc_launch_attention(s->k[2], d, Q, K, V, O, nullptr, vt, c));
      RC_TRY(rc_mark_stage(c));
      // 3: h1 = x + o Wo^T (residual added in the GEMM epilogue); b = RMSNorm(h1) g2
      TcGemmArgs go = gemm_args(T, H, hq, O, p[3], h1, H, TC_EPI_STORE_BF16);
      go.resid = p[0];
      RC_TRY(rc_launch_tc_gemm(s->k[3], go, c));
      RC_TRY(rc_launch_rmsnorm(h1, p[4], T, H, d.norm_eps, b, c));
      RC_TRY(rc_mark_stage(c));
      // 4: SwiGLU of the gate/up projection
      RC_TRY(run_swiglu(s->k[4], T, I, H, b, p[5], hb, gu, c));
      RC_TRY(rc_mark_stage(c));
      // 5: y = h1 + hb W2^T (residual added in the GEMM epilogue)
      TcGemmArgs gd = gemm_args(T, H, I, hb, p[6], p[7], H, TC_EPI_STORE_BF16);
      gd.resid = h1;
      RC_TRY(rc_launch_tc_gemm(s->k[5], gd, c));
      return rc_mark_stage(c);
    }
    case RC_OP_MOE_ROUTE: {
      int* counts = (int*)ws.take(4 * d.experts);
      return rc_launch_moe_route(s->k[0], d, p[0], (int*)p[1], (float*)p[2], (int*)p[3], (int*)p[4], nullptr,
                                 counts, c);
    }
    case RC_OP_MOE: {
      const int64_t slots = d.tokens * d.top_k;
      int* ids = p[5] ? (int*)p[5] : (int*)ws.take(4 * slots);
      float* w = p[6] ? (float*)p[6] : (float*)ws.take(4 * slots);
      int* offsets = p[7] ? (int*)p[7] : (int*)ws.take(4 * (d.experts + 1));
      int* perm = p[8] ? (int*)p[8] : (int*)ws.take(4 * slots);
      int* inv = (int*)ws.take(4 * slots);
      int* counts = (int*)ws.take(4 * d.experts);
      void* Xp = ws.take(2ull * slots * d.hidden);
      void* Hb = ws.take(2ull * slots * d.inter);
      void* Yb = ws.take(2ull * slots * d.hidden);
      float* acc = (float*)ws.take(4ull * d.tokens * d.hidden);
      // gate/up compute location 1: the GEMM's producer gathers X's rows itself (no gathered copy)
      const bool gather_in_gemm = s->k[1].location == 1;
      RC_TRY(rc_launch_moe_route(s->k[0], d, p[0], ids, w, offsets, perm, inv, counts, c));
      if (!gather_in_gemm)
        RC_TRY(rc_launch_moe_gather(p[1], perm, slots, d.hidden, (int)d.top_k, Xp, s->k[0].vec, c));
      RC_TRY(rc_mark_stage(c));
      const int64_t max_tiles = slots / 128 + d.experts;
      TcGemmArgs g1 =
          gemm_args(slots, 2 * d.inter, d.hidden, gather_in_gemm ? p[1] : Xp, p[2], Hb, d.inter, TC_EPI_SWIGLU);
      g1.groups = (int)d.experts;
      g1.offsets = offsets;
      g1.b_group_rows = 2 * d.inter;
      g1.max_tiles_m = max_tiles;
      if (gather_in_gemm) {
        g1.a_mode = TC_A_GATHER;
        g1.row_map = perm;
        g1.row_div = (int)d.top_k;
        g1.a_rows = d.tokens;
      }
      RC_TRY(launch_grouped(s->k[1], g1, c));
      RC_TRY(rc_mark_stage(c));
      TcGemmArgs g2 = gemm_args(slots, d.hidden, d.inter, Hb, p[3], Yb, d.hidden, TC_EPI_STORE_BF16);
      g2.groups = (int)d.experts;
      g2.offsets = offsets;
      g2.b_group_rows = d.hidden;
      g2.max_tiles_m = max_tiles;
      if (s->k[2].fuse) {
        // weighted combine fused into the down GEMM epilogue: fp32 atomics
        RC_TRY(cuda_err(cudaMemsetAsync(acc, 0, 4ull * d.tokens * d.hidden, (cudaStream_t)c.stream), "memset"));
        g2.D = acc;
        g2.epilogue = TC_EPI_SCALE_ATOMIC;
        g2.row_scale = w;
        g2.row_map = perm;
        g2.row_div = (int)d.top_k;
        g2.ldd = d.hidden;
        RC_TRY(launch_grouped(s->k[2], g2, c));
        RC_TRY(rc_launch_f32_to_bf16(acc, d.tokens * d.hidden, p[4], s->k[2].vec, c));
        return rc_mark_stage(c);
      }
      RC_TRY(launch_grouped(s->k[2], g2, c));
      RC_TRY(rc_launch_moe_combine(Yb, w, inv, d.tokens, d.hidden, (int)d.top_k, p[4], s->k[2].vec, c));
      return rc_mark_stage(c);
    }
  }
  return rc_fail(RC_ERR_UNSUPPORTED_OP, "rc_run: op kind %d", d.kind);
}

rc_status prepare(const rc_op_s* op, const rc_schedule_s* s, LaunchCtx* c, void* stream) {
  if (!op || !s) return rc_fail(RC_ERR_INVALID_ARG, "NULL op or schedule");
  if (s->op_kind != op->d.kind || s->n_stages != op->n_stages)
    return rc_fail(RC_ERR_INVALID_ARG, "schedule belongs to another op kind");
  for (int i = 0; i < s->n_stages; ++i) {
    std::string why;
    if (!rc_knobs_legal(op, i, s->k[i], &why)) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "stage %d: %s", i, why.c_str());
  }
  DevInfo* di = nullptr;
  int device = 0;
  RC_TRY(dev_info(&di, &device));
  RC_TRY(ensure_status_word(op, device));
  RC_TRY(ensure_ws(op, rc_workspace_bytes(op, s)));
  c->stream = stream;
  c->status = op->d_status;
  c->num_sms = di->num_sms;
  return RC_OK;
}

rc_status read_status(const rc_op_s* op) {
  int st = 0;
  RC_TRY(cuda_err(cudaMemcpy(&st, op->d_status, sizeof st, cudaMemcpyDeviceToHost), "read status"));
  if (st != RC_DEV_OK) {
    cudaMemset(op->d_status, 0, sizeof st);
    if (st == RC_DEV_BAD_ARG) return rc_fail(RC_ERR_INVALID_ARG, "a kernel rejected its arguments");
    if (st == RC_DEV_MISALIGNED)
      return rc_fail(RC_ERR_CUDA, "dynamic shared memory was not 1024-byte aligned for a packed kernel layout");
    return rc_fail(RC_ERR_DEVICE_TIMEOUT, "a bounded device wait gave up (code %d)", st);
  }
  return RC_OK;
}

}  // namespace

extern "C" void rc_op_destroy(rc_op* op) {
  if (!op) return;
  if (op->ws) cudaFree(op->ws);
  for (int i = 0; i < RC_MAX_TENSORS; ++i)
    if (op->stage_buf[i]) cudaFree(op->stage_buf[i]);
  if (op->d_status) cudaFree(op->d_status);
  for (int i = 0; i < RC_MAX_STAGES; ++i)
    if (op->input_ready[i]) cudaEventDestroy((cudaEvent_t)op->input_ready[i]);
  if (op->first_inputs_done) cudaEventDestroy((cudaEvent_t)op->first_inputs_done);
  if (op->copy_stream) cudaStreamDestroy((cudaStream_t)op->copy_stream);
  delete op;
}

extern "C" rc_status rc_run(const rc_op* op, const rc_schedule* s, const rc_tensors* io, void* stream) {
  if (!op || !s) return rc_fail(RC_ERR_INVALID_ARG, "rc_run: NULL op or schedule");
  RC_TRY(check_io(op, io));  // host-side argument checks come before any CUDA call
  LaunchCtx c;
  RC_TRY(prepare(op, s, &c, stream));
  return run_impl(op, s, io, c);
}

rc_status rc_mark_stage(const LaunchCtx& c) {
  const int done = ++c.stages_done;
  if (c.stage_events && c.next_event < c.n_stage_events)
    RC_TRY(cuda_err(cudaEventRecord((cudaEvent_t)c.stage_events[c.next_event++], (cudaStream_t)c.stream),
                    "cudaEventRecord(stage)"));
  if (c.stage_inputs && done < RC_MAX_STAGES && c.stage_inputs[done])
    RC_TRY(cuda_err(cudaStreamWaitEvent((cudaStream_t)c.stream, (cudaEvent_t)c.stage_inputs[done], 0),
                    "cudaStreamWaitEvent(stage inputs)"));
  return RC_OK;
}

extern "C" rc_status rc_run_profiled(const rc_op* op, const rc_schedule* s, const rc_tensors* io, void* stream,
                                     double* stage_ms, size_t cap, size_t* n_stages) {
  if (!stage_ms || !n_stages) return rc_fail(RC_ERR_INVALID_ARG, "rc_run_profiled: NULL output");
  if (!op || !s) return rc_fail(RC_ERR_INVALID_ARG, "rc_run_profiled: NULL op or schedule");
  RC_TRY(check_io(op, io));
  LaunchCtx c;
  RC_TRY(prepare(op, s, &c, stream));
  void* ev[RC_MAX_STAGES + 1] = {};
  for (int i = 0; i <= RC_MAX_STAGES; ++i) {
    rc_status st = cuda_err(cudaEventCreate((cudaEvent_t*)&ev[i]), "cudaEventCreate");
    if (st != RC_OK) {
      for (int j = 0; j < i; ++j) cudaEventDestroy((cudaEvent_t)ev[j]);
      return st;
    }
  }
  c.stage_events = ev + 1;
  c.n_stage_events = RC_MAX_STAGES;
  rc_status st = cuda_err(cudaEventRecord((cudaEvent_t)ev[0], (cudaStream_t)stream), "cudaEventRecord");
  if (st == RC_OK) st = run_impl(op, s, io, c);
  if (st == RC_OK && c.next_event == 0) st = rc_mark_stage(c);  // single-stage ops: mark the end
  if (st == RC_OK) st = cuda_err(cudaStreamSynchronize((cudaStream_t)stream), "cudaStreamSynchronize");
  if (st == RC_OK) st = read_status(op);
  size_t n = 0;
  if (st == RC_OK) {
    for (int i = 0; i < c.next_event && n < cap; ++i, ++n) {
      float ms = 0.f;
      cudaEventElapsedTime(&ms, (cudaEvent_t)ev[i], (cudaEvent_t)ev[i + 1]);
      stage_ms[n] = ms;
    }
  }
  *n_stages = n;
  for (int i = 0; i <= RC_MAX_STAGES; ++i) cudaEventDestroy((cudaEvent_t)ev[i]);
  return st;
}

// Synchronise the stream and report device-side failures of earlier runs.
extern "C" rc_status rc_op_check(const rc_op* op, void* stream) {
  if (!op) return rc_fail(RC_ERR_INVALID_ARG, "rc_op_check: NULL op");
  RC_TRY(cuda_err(cudaStreamSynchronize((cudaStream_t)stream), "cudaStreamSynchronize"));
  if (!op->d_status) return RC_OK;
  return read_status(op);
}

extern "C" rc_status rc_run_host(const rc_op* op, const rc_schedule* s, const rc_tensors* host_io, void* stream) {
  LaunchCtx c;
  RC_TRY(prepare(op, s, &c, stream));
  if (!host_io) return rc_fail(RC_ERR_INVALID_ARG, "rc_run_host: NULL tensors");
  const auto slots = rc_slots(op);
  rc_tensors dev;
  memset(&dev, 0, sizeof dev);
  cudaStream_t st = (cudaStream_t)stream;
  // Inputs first read by a later stage are copied on a second stream after
  // the first stage's inputs, so that their copy overlaps the earlier stages
  // (the copy engines are shared: issuing them in parallel would only delay
  // the first stage). Stage i waits for its inputs at the end of stage i - 1.
  bool later = false;
  for (size_t i = 0; i < slots.size(); ++i) later = later || (slots[i].input && slots[i].first_stage > 0);
  if (later && !op->copy_stream) {
    cudaStream_t cs = nullptr;
    RC_TRY(cuda_err(cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking), "cudaStreamCreate(copies)"));
    op->copy_stream = cs;
    for (int i = 0; i < RC_MAX_STAGES; ++i)
      RC_TRY(cuda_err(cudaEventCreateWithFlags((cudaEvent_t*)&op->input_ready[i], cudaEventDisableTiming),
                      "cudaEventCreate(inputs)"));
    RC_TRY(cuda_err(cudaEventCreateWithFlags((cudaEvent_t*)&op->first_inputs_done, cudaEventDisableTiming),
                    "cudaEventCreate(inputs)"));
  }
  for (size_t i = 0; i < slots.size(); ++i) {
    if (!host_io->p[i]) {
      if (slots[i].optional) continue;
      return rc_fail(RC_ERR_INVALID_ARG, "rc_run_host: slot %zu is NULL", i);
    }
    if (op->stage_bytes[i] < slots[i].bytes) {
      if (op->stage_buf[i]) cudaFree(op->stage_buf[i]);
      op->stage_buf[i] = nullptr;
      op->stage_bytes[i] = 0;
      RC_TRY(cuda_err(cudaMalloc(&op->stage_buf[i], slots[i].bytes > 0 ? slots[i].bytes : 16), "cudaMalloc(staging)"));
      op->stage_bytes[i] = slots[i].bytes;
    }
    dev.p[i] = op->stage_buf[i];
    if (slots[i].input && slots[i].bytes && slots[i].first_stage == 0)
      RC_TRY(cuda_err(cudaMemcpyAsync(dev.p[i], host_io->p[i], slots[i].bytes, cudaMemcpyHostToDevice, st), "H2D"));
  }
  void* waits[RC_MAX_STAGES] = {};
  if (later) {
    cudaStream_t cs = (cudaStream_t)op->copy_stream;
    RC_TRY(cuda_err(cudaEventRecord((cudaEvent_t)op->first_inputs_done, st), "cudaEventRecord(inputs)"));
    RC_TRY(cuda_err(cudaStreamWaitEvent(cs, (cudaEvent_t)op->first_inputs_done, 0), "cudaStreamWaitEvent(inputs)"));
    for (int g = 1; g < RC_MAX_STAGES; ++g) {
      bool any = false;
      for (size_t i = 0; i < slots.size(); ++i) {
        if (!(slots[i].input && slots[i].first_stage == g && dev.p[i] && slots[i].bytes)) continue;
        RC_TRY(cuda_err(cudaMemcpyAsync(dev.p[i], host_io->p[i], slots[i].bytes, cudaMemcpyHostToDevice, cs), "H2D"));
        any = true;
      }
      if (any) {
        RC_TRY(cuda_err(cudaEventRecord((cudaEvent_t)op->input_ready[g], cs), "cudaEventRecord(inputs)"));
        waits[g] = op->input_ready[g];
      }
    }
  }
  c.stage_inputs = waits;
  rc_status rs = run_impl(op, s, &dev, c);
  // a stage whose inputs were never waited for (an error before it) must not outlive the call
  if (rs != RC_OK) {  // no copy into the caller's buffers may outlive the call
    if (op->copy_stream) cudaStreamSynchronize((cudaStream_t)op->copy_stream);
    cudaStreamSynchronize(st);
    return rs;
  }
  for (size_t i = 0; i < slots.size(); ++i)
    if (slots[i].output && dev.p[i] && slots[i].bytes)
      RC_TRY(cuda_err(cudaMemcpyAsync(host_io->p[i], dev.p[i], slots[i].bytes, cudaMemcpyDeviceToHost, st), "D2H"));
  RC_TRY(cuda_err(cudaStreamSynchronize(st), "cudaStreamSynchronize"));
  return read_status(op);
}

extern "C" rc_status rc_candidate_measure(const rc_op* op, const rc_schedule* const* cands, size_t n,
                                          const rc_tensors* io, void* stream, const rc_measure_opts* opts,
                                          rc_measurement* out) {
  if (!op || (n && (!cands || !out))) return rc_fail(RC_ERR_INVALID_ARG, "rc_candidate_measure: NULL argument");
  RC_TRY(check_io(op, io));
  rc_measure_opts o{5, 20, 1, 0.0};
  if (opts) {
    o = *opts;
    if (o.warmup < 0) o.warmup = 0;
    if (o.repeats < 1) o.repeats = 1;
  }
  DevInfo* di = nullptr;
  int device = 0;
  RC_TRY(dev_info(&di, &device));
  if (o.flush_l2) {
    std::lock_guard<std::mutex> lk(g_dev_mu);
    const size_t want = 2 * di->l2_bytes;
    if (di->flush_bytes < want) {
      if (di->flush) cudaFree(di->flush);
      di->flush = nullptr;
      di->flush_bytes = 0;
      RC_TRY(cuda_err(cudaMalloc(&di->flush, want), "cudaMalloc(L2 flush)"));
      di->flush_bytes = want;
    }
  }
  cudaStream_t st = (cudaStream_t)stream;
  // per repeat: a start event and one event after each stage (the last one ends the run)
  constexpr int EV = RC_MAX_STAGES + 1;
  std::vector<cudaEvent_t> ev((size_t)EV * o.repeats, nullptr);
  for (auto& e : ev) {
    rc_status cs = cuda_err(cudaEventCreate(&e), "cudaEventCreate");
    if (cs != RC_OK) {
      for (auto& x : ev)
        if (x) cudaEventDestroy(x);
      return cs;
    }
  }
  auto destroy = [&]() {
    for (auto& e : ev) cudaEventDestroy(e);
  };
  const auto t_start = std::chrono::steady_clock::now();
  rc_status batch = RC_OK;
  for (size_t i = 0; i < n; ++i) {
    rc_measurement& m = out[i];
    memset(&m, 0, sizeof m);
    m.sched_hash = rc_schedule_hash(cands[i]);
    if (o.budget_s > 0) {
      const double el = std::chrono::duration<double>(std::chrono::steady_clock::now() - t_start).count();
      if (el > o.budget_s) {
        for (size_t j = i; j < n; ++j) {
          memset(&out[j], 0, sizeof out[j]);
          out[j].status = RC_ERR_TIMEOUT;
          out[j].sched_hash = rc_schedule_hash(cands[j]);
        }
        batch = rc_fail(RC_ERR_TIMEOUT, "measurement budget of %.1f s exceeded", o.budget_s);
        break;
      }
    }
    LaunchCtx c;
    rc_status s = prepare(op, cands[i], &c, stream);
    for (int w = 0; s == RC_OK && w < o.warmup; ++w) s = run_impl(op, cands[i], io, c);
    int n_marks = 0;  // stage-end events of a run (the same for every repeat)
    for (int r = 0; s == RC_OK && r < o.repeats; ++r) {
      cudaEvent_t* er = ev.data() + (size_t)EV * r;
      if (o.flush_l2) s = rc_launch_l2_flush(di->flush, di->flush_bytes, stream);
      if (s == RC_OK) s = cuda_err(cudaEventRecord(er[0], st), "cudaEventRecord");
      c.stage_events = (void**)(er + 1);
      c.n_stage_events = RC_MAX_STAGES;
      c.next_event = 0;
      if (s == RC_OK) s = run_impl(op, cands[i], io, c);
      if (s == RC_OK && c.next_event == 0) s = rc_mark_stage(c);  // single-stage ops: mark the end
      n_marks = c.next_event;
    }
    c.stage_events = nullptr;
    if (s == RC_OK) s = cuda_err(cudaStreamSynchronize(st), "cudaStreamSynchronize");
    if (s == RC_OK) s = read_status(op);
    if (s == RC_ERR_CUDA) {
      // a sticky CUDA error poisons the context: stop the batch
      m.status = s;
      batch = s;
      for (size_t j = i + 1; j < n; ++j) {
        memset(&out[j], 0, sizeof out[j]);
        out[j].status = RC_ERR_CUDA;
      }
      break;
    }
    if (s != RC_OK) {
      m.status = s;
      continue;
    }
    auto median = [](std::vector<double> v) {
      std::sort(v.begin(), v.end());
      const size_t R = v.size();
      return R % 2 ? v[R / 2] : 0.5 * (v[R / 2 - 1] + v[R / 2]);
    };
    std::vector<double> t(o.repeats);
    for (int r = 0; r < o.repeats; ++r) {
      float ms = 0.f;
      cudaEventElapsedTime(&ms, ev[(size_t)EV * r], ev[(size_t)EV * r + n_marks]);
      t[r] = ms;
    }
    m.n_stages = n_marks;
    for (int g = 0; g < n_marks; ++g) {
      std::vector<double> ts(o.repeats);
      for (int r = 0; r < o.repeats; ++r) {
        float ms = 0.f;
        cudaEventElapsedTime(&ms, ev[(size_t)EV * r + g], ev[(size_t)EV * r + g + 1]);
        ts[r] = ms;
      }
      m.stage_ms[g] = median(ts);
    }
    std::vector<double> srt = t;
    std::sort(srt.begin(), srt.end());
    const size_t R = srt.size();
    m.ms_median = median(t);
    m.ms_min = srt[0];
    double sum = 0;
    for (double x : t) sum += x;
    m.ms_mean = sum / R;
    m.tflops = op->info.flops / (m.ms_median * 1e-3) / 1e12;
    m.gbps = op->info.bytes / (m.ms_median * 1e-3) / 1e9;
    m.status = RC_OK;
  }
  destroy();
  return batch;
}
