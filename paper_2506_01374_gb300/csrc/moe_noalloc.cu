// Top-k routing for callers that cannot allocate device memory.
//
// The regular routing path (rc_run on an RC_OP_MOE_ROUTE op) keeps the
// per-expert token counts in library workspace that it allocates on first
// use. rc_moe_route_noalloc runs the same three routing kernels but keeps
// those counts in the fixed array below, so the call itself never allocates.
#include <cuda_runtime.h>

#include <cstring>
#include <mutex>

#include "rc_internal.h"

// Per-expert counts of the no-allocation routing path. Every GPU that loads
// the library holds this array (1 KB) until the process exits.
static __device__ __align__(256) int g_noalloc_route_counts[RC_NOALLOC_MAX_EXPERTS];

namespace {
std::mutex g_mu;
// Device address of g_noalloc_route_counts per device ordinal, with the
// context it was looked up in: a new primary context (after cudaDeviceReset)
// loads the module again, so a changed context means a fresh lookup.
struct CountsAddr {
  void* ctx = nullptr;
  int* ptr = nullptr;
};
CountsAddr g_counts_dev[64];

typedef int (*CtxGetCurrentFn)(void**);
CtxGetCurrentFn g_ctx_get_current = nullptr;

// The current driver context, or nullptr when the driver entry point is unavailable.
void* current_context() {
  if (!g_ctx_get_current) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_ctx_get_current = (CtxGetCurrentFn)p;
    if (!g_ctx_get_current) return nullptr;
  }
  void* ctx = nullptr;
  return g_ctx_get_current(&ctx) == 0 ? ctx : nullptr;
}
}  // namespace

extern "C" rc_status rc_moe_route_noalloc(const void* logits, int32_t logits_fp32, int64_t tokens, int64_t experts,
                                          int64_t top_k, int32_t renorm, int32_t* ids, float* weights,
                                          int32_t* offsets, int32_t* perm, void* stream) {
  if (!logits || !ids || !weights || !offsets || !perm)
    return rc_fail(RC_ERR_INVALID_ARG, "rc_moe_route_noalloc: NULL tensor");
  for (const void* p : {logits, (const void*)ids, (const void*)weights, (const void*)offsets, (const void*)perm})
    if ((uintptr_t)p % 16) return rc_fail(RC_ERR_INVALID_ARG, "rc_moe_route_noalloc: tensor not 16-byte aligned");
  if (tokens <= 0 || experts <= 0 || top_k <= 0 || top_k > experts)
    return rc_fail(RC_ERR_INVALID_ARG, "rc_moe_route_noalloc: need tokens > 0 and 0 < top_k <= experts");
  if (experts > RC_NOALLOC_MAX_EXPERTS)
    return rc_fail(RC_ERR_INVALID_ARG, "rc_moe_route_noalloc: experts = %lld exceeds the fixed scratch of %d experts",
                   (long long)experts, RC_NOALLOC_MAX_EXPERTS);
  if (top_k > 16) return rc_fail(RC_ERR_UNSUPPORTED_OP, "rc_moe_route_noalloc: top_k must be <= 16");
  // tokens * top_k is limited further by rc_launch_moe_route (the routing kernels' slot range).

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "rc_moe_route_noalloc: cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= 64) return rc_fail(RC_ERR_CUDA, "rc_moe_route_noalloc: device ordinal %d", dev);
  int* counts = nullptr;
  {
    // One-time set-up per device (and per context of that device), with that
    // device current: translate the array's host-side name into its device
    // address.
    std::lock_guard<std::mutex> lk(g_mu);
    void* ctx = current_context();
    CountsAddr& a = g_counts_dev[dev];
    if (!a.ptr || ctx != a.ctx) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_route_counts);
      if (e != cudaSuccess)
        return rc_fail(RC_ERR_CUDA, "rc_moe_route_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
      a.ptr = (int*)p;
      a.ctx = current_context();  // the lookup may have created the primary context
    }
    counts = a.ptr;
  }

  rc_knobs k;
  memset(&k, 0, sizeof k);
  k.tile_m = 4;  // tokens (warps) per CTA of the top-k kernel
  rc_op_desc d;
  memset(&d, 0, sizeof d);
  d.kind = RC_OP_MOE_ROUTE;
  d.tokens = tokens;
  d.experts = experts;
  d.top_k = top_k;
  d.logits_fp32 = logits_fp32 ? 1 : 0;
  d.renorm = renorm ? 1 : 0;
  LaunchCtx c;
  c.stream = stream;
  c.status = nullptr;
  c.num_sms = 0;
  // rc_launch_moe_route zeroes counts[0, experts) with cudaMemsetAsync on
  // `stream` before the count kernel adds to them with atomicAdd, so the
  // previous call's counts left in the array do not matter.
  return rc_launch_moe_route(k, d, logits, ids, weights, offsets, perm, nullptr, counts, c);
}
