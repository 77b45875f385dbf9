// Launchers of kernels that this build does not provide yet: they report
// RC_ERR_UNSUPPORTED_OP so callers see a clear error instead of a fallback.
#include "rc_internal.h"

rc_status rc_launch_attention(const rc_knobs&, const rc_op_desc&, const void*, const void*, const void*, void*,
                              float*, const LaunchCtx&) {
  return rc_fail(RC_ERR_UNSUPPORTED_OP, "attention not built");
}
