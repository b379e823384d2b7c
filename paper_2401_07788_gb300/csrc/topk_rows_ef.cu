// topk_rows_ef.cu -- instantiates the row TopK kernels of topk_rows.cuh
// for one fused variant (kEF), so that the variants compile in parallel.
#include "topk_rows.cuh"

namespace mpc {

cudaError_t launch_topk_rows_ef(const TopkRowArgs& a, int num_sms, cudaStream_t s) {
  return rows::run_mode<kEF>(a, num_sms, s);
}

}  // namespace mpc
