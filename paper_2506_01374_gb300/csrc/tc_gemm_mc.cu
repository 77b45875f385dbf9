// Instantiations of the tensor-core GEMM whose B tile is shared by a cluster
// of four CTAs along M through TMA multicast (TileSize M = 512, cta_group::1
// UMMAs): dense 2-D GEMMs with N tile {64, 128, 256} x epilogue {bf16 store,
// fp32 split-K}, and convolutions with N tile {64, 160} x epilogue {bf16
// store, bias+SiLU, fp32 split-K} x A as one 4-D box. Every B slice is
// BN / 4 rows, a whole number of 8-row swizzle atoms.
#include "tc_gemm.cuh"

rc_status tc_dispatch_mc(const rc_knobs& k, const TcGemmArgs& a, const LaunchCtx& c) {
  using namespace tcg;
  constexpr int MC = 4;
  if (a.groups > 0 || a.a_mode == TC_A_GATHER || a.epilogue == TC_EPI_SWIGLU)
    return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm: a B-multicast cluster takes dense or convolution GEMMs");
  if (a.a_mode == TC_A_CONV) {
#define RC_CONV(BN)                                                                                         \
  case BN:                                                                                                  \
    switch (a.epilogue) {                                                                                   \
      case TC_EPI_STORE_BF16: return launch<BN, TC_EPI_STORE_BF16, TC_A_CONV, false, false, MC>(k, a, c);  \
      case TC_EPI_BIAS_SILU: return launch<BN, TC_EPI_BIAS_SILU, TC_A_CONV, false, false, MC>(k, a, c);    \
      case TC_EPI_PARTIAL_F32: return launch<BN, TC_EPI_PARTIAL_F32, TC_A_CONV, false, false, MC>(k, a, c); \
    }                                                                                                       \
    break;
    switch (k.tile_n) {
      RC_CONV(64)
      RC_CONV(160)
    }
#undef RC_CONV
  } else if (a.a_mode == TC_A_2D) {
#define RC_DENSE(BN)                                                                                        \
  case BN:                                                                                                  \
    switch (a.epilogue) {                                                                                   \
      case TC_EPI_STORE_BF16: return launch<BN, TC_EPI_STORE_BF16, TC_A_2D, false, false, MC>(k, a, c);    \
      case TC_EPI_PARTIAL_F32: return launch<BN, TC_EPI_PARTIAL_F32, TC_A_2D, false, false, MC>(k, a, c);  \
    }                                                                                                       \
    break;
    switch (k.tile_n) {
      RC_DENSE(64)
      RC_DENSE(128)
      RC_DENSE(256)
    }
#undef RC_DENSE
  }
  return rc_fail(RC_ERR_ILLEGAL_SCHEDULE, "tc_gemm B multicast: no variant for N tile %d, A mode %d, epilogue %d",
                 k.tile_n, a.a_mode, a.epilogue);
}
