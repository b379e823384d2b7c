// topk_rows_delta.cu -- instantiates the row TopK kernels of topk_rows.cuh
// for one fused variant (kDelta), so that the variants compile in parallel.
#include "topk_rows.cuh"

namespace mpc {

cudaError_t launch_topk_rows_delta(const TopkRowArgs& a, int num_sms, cudaStream_t s) {
  return rows::run_mode<kDelta>(a, num_sms, s);
}

}  // namespace mpc
