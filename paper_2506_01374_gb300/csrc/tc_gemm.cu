// Host side of the tensor-core GEMM family: TMA descriptor encoding and the
// routing of (A mode, grouped, epilogue) to the instantiation units.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "tc_gemm.cuh"

rc_status tc_dispatch_dense(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);
rc_status tc_dispatch_dense_pair(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);
rc_status tc_dispatch_conv_pair(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);
rc_status tc_dispatch_grouped_pair(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);
rc_status tc_dispatch_conv(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);
rc_status tc_dispatch_grouped(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);
rc_status tc_dispatch_mc(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);
rc_status tc_dispatch_grouped_t(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c);

namespace tcg {
namespace {
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn g_encode = nullptr;
std::once_flag g_once;

rc_status get_encode(EncodeTiledFn* fn) {
  std::call_once(g_once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = (EncodeTiledFn)p;
  });
  if (!g_encode) return rc_fail(RC_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
  *fn = g_encode;
  return RC_OK;
}
}  // namespace

// [rows][inner] bf16 row-major matrix, box = 64 x box_rows, 128-byte swizzle,
// out-of-range elements read as zero.
rc_status encode_2d(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows) {
  EncodeTiledFn fn;
  RC_TRY(get_encode(&fn));
  if ((uintptr_t)base % 16 || (inner * 2) % 16) return rc_fail(RC_ERR_INVALID_ARG, "TMA: 16-byte alignment");
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return rc_fail(RC_ERR_CUDA, "cuTensorMapEncodeTiled(2d) failed: %d", (int)r);
  return RC_OK;
}

// NHWC activation x[n][h][w][c] seen as a 4-D tensor {c, w, h, n}; one box is
// 64 channels x box_w columns x box_h rows of one image = the 128 output
// pixels of an M tile, shifted by the filter tap (r, s). For an explicitly
// padded input the tensor is (w + 2 pad) wide and (h + 2 pad) high.
rc_status encode_conv(CUtensorMap* m, const void* x, uint64_t c, uint64_t w, uint64_t h, uint64_t n,
                      uint64_t box_w, uint64_t box_h) {
  EncodeTiledFn fn;
  RC_TRY(get_encode(&fn));
  if ((uintptr_t)x % 16 || (c * 2) % 16) return rc_fail(RC_ERR_INVALID_ARG, "TMA: 16-byte alignment");
  cuuint64_t dims[4] = {c, w, h, n};
  cuuint64_t strides[3] = {c * 2, w * c * 2, h * w * c * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)box_w, (cuuint32_t)box_h, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return rc_fail(RC_ERR_CUDA, "cuTensorMapEncodeTiled(conv) failed: %d", (int)r);
  return RC_OK;
}
}  // namespace tcg

rc_status rc_launch_tc_gemm(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  if (a.M <= 0 || a.N <= 0 || a.K <= 0) return rc_fail(RC_ERR_INVALID_ARG, "tc_gemm: empty problem");
  if (a.M > 0x7fffffff || a.N > 0x7fffffff || a.K > 0x7fffffff)
    return rc_fail(RC_ERR_UNSUPPORTED_OP, "tc_gemm: dimension exceeds 2^31");
  if (k.stages < 1) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm: stages < 1");
  if (k.tile_m != 128 && k.tile_m != 256 && k.tile_m != 512)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm: M tile %d", k.tile_m);
  if (k.tile_m == 512) return tc_dispatch_mc(k, a, c);  // four CTAs sharing the B tile by multicast
  const bool pair = k.tile_m == 256;  // a CTA pair per 256-row tile
  if (a.a_mode == TC_A_CONV || a.a_mode == TC_A_CONV_ROWS)
    return pair ? tc_dispatch_conv_pair(k, a, c) : tc_dispatch_conv(k, a, c);
  if (a.a_mode == TC_A_GATHER && (pair || a.groups <= 0))
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm: gathered A rows need a grouped GEMM on one CTA (M tile 128)");
  if (a.groups > 0) {
    // Layout 2: weights on UMMA M, each segment's tokens on N (the tile transposed in TMEM)
    if (k.layout == 2) return tc_dispatch_grouped_t(k, a, c);
    return pair ? tc_dispatch_grouped_pair(k, a, c) : tc_dispatch_grouped(k, a, c);
  }
  return pair ? tc_dispatch_dense_pair(k, a, c) : tc_dispatch_dense(k, a, c);
}
