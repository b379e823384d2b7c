// topk_rows_plain.cu -- instantiates the row TopK kernels of topk_rows.cuh
// for one fused variant (kPlain), so that the variants compile in parallel.
#include "topk_rows.cuh"

namespace mpc {

cudaError_t launch_topk_rows_plain(const TopkRowArgs& a, int num_sms, cudaStream_t s) {
  return rows::run_mode<kPlain>(a, num_sms, s);
}

}  // namespace mpc
