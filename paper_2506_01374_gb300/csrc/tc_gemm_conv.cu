// Implicit-GEMM convolution instantiations of the tensor-core GEMM: N tile
// {64, 80, 160} x epilogue {bf16 store, bias+SiLU, fp32 split-K} x A operand
// {one 4-D box with zero-filled borders, 2-D row boxes of a padded copy}.
#include "tc_gemm.cuh"

rc_status tc_dispatch_conv(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  using namespace tcg;
#define RC_CASE(BN)                                                                                       \
  case BN:                                                                                                \
    if (a.a_mode == TC_A_CONV_ROWS) {                                                                     \
      switch (a.epilogue) {                                                                               \
        case TC_EPI_STORE_BF16: return launch<BN, TC_EPI_STORE_BF16, TC_A_CONV_ROWS, false>(k, a, c);   \
        case TC_EPI_BIAS_SILU: return launch<BN, TC_EPI_BIAS_SILU, TC_A_CONV_ROWS, false>(k, a, c);     \
        case TC_EPI_PARTIAL_F32: return launch<BN, TC_EPI_PARTIAL_F32, TC_A_CONV_ROWS, false>(k, a, c); \
      }                                                                                                   \
      break;                                                                                              \
    }                                                                                                     \
    switch (a.epilogue) {                                                                                 \
      case TC_EPI_STORE_BF16: return launch<BN, TC_EPI_STORE_BF16, TC_A_CONV, false>(k, a, c);          \
      case TC_EPI_BIAS_SILU: return launch<BN, TC_EPI_BIAS_SILU, TC_A_CONV, false>(k, a, c);            \
      case TC_EPI_PARTIAL_F32: return launch<BN, TC_EPI_PARTIAL_F32, TC_A_CONV, false>(k, a, c);        \
    }                                                                                                     \
    break;
  switch (k.tile_n) {
    RC_CASE(64)
    RC_CASE(80)
    RC_CASE(160)
  }
#undef RC_CASE
  return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm conv: no variant for N tile %d epilogue %d", k.tile_n,
                 a.epilogue);
}
