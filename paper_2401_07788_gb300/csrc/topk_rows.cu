// topk_rows.cu -- dispatch of the on-chip row TopK path to the fused variant.
#include "kernels.h"

namespace mpc {

cudaError_t launch_topk_rows(int mode, const TopkRowArgs& a, int num_sms, cudaStream_t s) {
  if (a.rows <= 0) return cudaSuccess;
  switch (mode) {
    case kPlain: return launch_topk_rows_plain(a, num_sms, s);
    case kEF: return launch_topk_rows_ef(a, num_sms, s);
    case kDelta: return launch_topk_rows_delta(a, num_sms, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace mpc
