// Implicit-GEMM convolution instantiations of the tensor-core GEMM on CTA
// pairs (TileSize M = 256, cta_group::2 UMMAs): N tile {64, 80, 160} x
// epilogue {bf16 store, bias+SiLU, fp32 split-K}, A as one 4-D box per CTA.
#include "tc_gemm.cuh"

rc_status tc_dispatch_conv_pair(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  using namespace tcg;
  if (a.a_mode != TC_A_CONV)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm conv pair: only the 4-D box A layout");
#define RC_CASE(BN)                                                                                       \
  case BN:                                                                                                \
    switch (a.epilogue) {                                                                                 \
      case TC_EPI_STORE_BF16: return launch<BN, TC_EPI_STORE_BF16, TC_A_CONV, false, true>(k, a, c);    \
      case TC_EPI_BIAS_SILU: return launch<BN, TC_EPI_BIAS_SILU, TC_A_CONV, false, true>(k, a, c);      \
      case TC_EPI_PARTIAL_F32: return launch<BN, TC_EPI_PARTIAL_F32, TC_A_CONV, false, true>(k, a, c);  \
    }                                                                                                     \
    break;
  switch (k.tile_n) {
    RC_CASE(64)
    RC_CASE(80)
    RC_CASE(160)
  }
#undef RC_CASE
  return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm conv pair: no variant for N tile %d epilogue %d", k.tile_n,
                 a.epilogue);
}
