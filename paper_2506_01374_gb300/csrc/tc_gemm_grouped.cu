// Grouped (MoE) instantiations of the tensor-core GEMM: N tile {64, 128, 224, 256}
// (SwiGLU: 2 x {32, 64, 128}) x epilogue {SwiGLU, bf16 store, scaled fp32
// atomic combine}, plus SwiGLU with A rows gathered in the producer.
#include "tc_gemm.cuh"

rc_status tc_dispatch_grouped(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  using namespace tcg;
  const int bn = a.epilogue == TC_EPI_SWIGLU ? 2 * k.tile_n : k.tile_n;
#define RC_CASE(BN)                                                                                       \
  case BN:                                                                                                \
    switch (a.epilogue) {                                                                                 \
      case TC_EPI_STORE_BF16: return launch<BN, TC_EPI_STORE_BF16, TC_A_2D, true>(k, a, c);             \
      case TC_EPI_SWIGLU: return launch<BN, TC_EPI_SWIGLU, TC_A_2D, true>(k, a, c);                     \
      case TC_EPI_SCALE_ATOMIC: return launch<BN, TC_EPI_SCALE_ATOMIC, TC_A_2D, true>(k, a, c);         \
    }                                                                                                     \
    break;
  if (a.a_mode == TC_A_GATHER) {  // A rows gathered by the producer (grouped SwiGLU only)
    if (a.epilogue != TC_EPI_SWIGLU) return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm: gathered A needs SwiGLU");
    switch (bn) {
      case 64: return launch<64, TC_EPI_SWIGLU, TC_A_GATHER, true>(k, a, c);
      case 128: return launch<128, TC_EPI_SWIGLU, TC_A_GATHER, true>(k, a, c);
      case 256: return launch<256, TC_EPI_SWIGLU, TC_A_GATHER, true>(k, a, c);
    }
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm: gathered A: N tile %d", bn);
  }
  switch (bn) {
    RC_CASE(64)
    RC_CASE(128)
    RC_CASE(256)
    case 224:
      if (a.epilogue == TC_EPI_STORE_BF16) return launch<224, TC_EPI_STORE_BF16, TC_A_2D, true>(k, a, c);
      if (a.epilogue == TC_EPI_SCALE_ATOMIC) return launch<224, TC_EPI_SCALE_ATOMIC, TC_A_2D, true>(k, a, c);
      break;
  }
#undef RC_CASE
  return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm grouped: no variant for N tile %d epilogue %d", bn, a.epilogue);
}
