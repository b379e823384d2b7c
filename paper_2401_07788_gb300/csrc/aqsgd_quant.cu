// aqsgd_quant.cu -- AQ-SGD with quantisation (§2.5: the change of the
// activations of each training sample is sent, here compressed by the min-max
// quantiser of §2.2 as in the cited work):
//   d = x - buf[id, r];  message = Quant(d);  buf[id, r] += Dequant(message).
// For 2/4/8-bit codes on rows of up to 4096 entries the sender runs in one pass
// (aqsgd_quant_fused_kernel, quant.cu).  Otherwise the abi runs:
// aqsgd_delta_kernel (d into a workspace, one row per logical row
// i * rows_per_sample + r), the quantiser on d, aqsgd_dequant_add_kernel.  The
// receiver's update of its copy of the buffer is aqsgd_dequant_add_kernel.
// All HBM-bound.
#include <cstdint>

#include "common.cuh"
#include "kernels.h"
#include "launch_util.h"

namespace mpc {
namespace {

constexpr int kT = 256;
constexpr int kPerT = 4;  // entries per thread per block

// Blocks of kT * kPerT consecutive entries of one logical row (bpr per row).
__global__ void __launch_bounds__(kT)
    aqsgd_delta_kernel(const float* __restrict__ x, const float* __restrict__ buf,
                       const int64_t* __restrict__ ids, int64_t rps, int64_t L, int bpr,
                       int64_t num_samples, float* __restrict__ d, unsigned* status) {
  pdl_begin();
  const int64_t lr = blockIdx.x / bpr;
  const int64_t j0 = static_cast<int64_t>(blockIdx.x % bpr) * (kT * kPerT);
  const int64_t sid = ids[lr / rps];
  const bool ok = sid >= 0 && sid < num_samples;
  if (!ok && threadIdx.x == 0 && j0 == 0) set_status(status, STATUS_BAD_SAMPLE);
  const float* xr = x + lr * L;
  const float* br = ok ? buf + (sid * rps + lr % rps) * L : nullptr;
  float* dr = d + lr * L;
#pragma unroll
  for (int u = 0; u < kPerT; ++u) {
    const int64_t j = j0 + u * kT + threadIdx.x;
    if (j < L) dr[j] = ok ? fsub(xr[j], br[j]) : 0.0f;
  }
}

// buf[id, r][j] += minv + q * scale (bits 1..16), or += the raw fp32 bits of
// the code word (bits = 32, the passthrough).
__global__ void __launch_bounds__(kT)
    aqsgd_dequant_add_kernel(const uint32_t* __restrict__ codes, const float* __restrict__ scale,
                             const float* __restrict__ minv, float* __restrict__ buf,
                             const int64_t* __restrict__ ids, int64_t rps, int64_t L, int64_t W,
                             int bits, int bpr, int64_t num_samples, unsigned* status) {
  pdl_begin();
  const int64_t lr = blockIdx.x / bpr;
  const int64_t j0 = static_cast<int64_t>(blockIdx.x % bpr) * (kT * kPerT);
  const int64_t sid = ids[lr / rps];
  if (sid < 0 || sid >= num_samples) {
    if (threadIdx.x == 0 && j0 == 0) set_status(status, STATUS_BAD_SAMPLE);
    return;
  }
  const uint32_t* cr = codes + lr * W;
  float* br = buf + (sid * rps + lr % rps) * L;
  const float sc = scale[lr], m = minv[lr];
  const uint32_t mask = bits >= 32 ? 0xffffffffu : (1u << bits) - 1u;
#pragma unroll
  for (int u = 0; u < kPerT; ++u) {
    const int64_t j = j0 + u * kT + threadIdx.x;
    if (j >= L) break;
    float dh;
    if (bits == 32) {
      dh = __uint_as_float(cr[j]);
    } else {
      const int64_t p = j * bits;
      const int64_t w = p >> 5;
      const int sh = static_cast<int>(p & 31);
      uint64_t v = cr[w];
      if (sh + bits > 32) v |= static_cast<uint64_t>(cr[w + 1]) << 32;
      const uint32_t q = static_cast<uint32_t>(v >> sh) & mask;
      dh = fadd(m, fmul(static_cast<float>(q), sc));
    }
    br[j] = fadd(br[j], dh);
  }
}

int blocks_per_row(int64_t L) { return static_cast<int>((L + kT * kPerT - 1) / (kT * kPerT)); }

}  // namespace

cudaError_t launch_aqsgd_delta(const float* x, const float* buf, const int64_t* ids, int64_t n_ids,
                               int64_t rps, int64_t L, int64_t num_samples, float* d,
                               unsigned* status, cudaStream_t s) {
  const int64_t rows = n_ids * rps;
  if (rows <= 0) return cudaSuccess;
  const int bpr = blocks_per_row(L);
  if (rows * bpr > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_kernel(aqsgd_delta_kernel, dim3(static_cast<unsigned>(rows * bpr)), dim3(kT), 0, s,
                       0u, x, buf, ids, rps, L, bpr, num_samples, d, status);
}

cudaError_t launch_aqsgd_dequant_add(const uint32_t* codes, const float* scale, const float* minv,
                                     float* buf, const int64_t* ids, int64_t n_ids, int64_t rps,
                                     int64_t L, int64_t W, int bits, int64_t num_samples,
                                     unsigned* status, cudaStream_t s) {
  const int64_t rows = n_ids * rps;
  if (rows <= 0) return cudaSuccess;
  const int bpr = blocks_per_row(L);
  if (rows * bpr > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_kernel(aqsgd_dequant_add_kernel, dim3(static_cast<unsigned>(rows * bpr)), dim3(kT),
                       0, s, 0u, codes, scale, minv, buf, ids, rps, L, W, bits, bpr, num_samples,
                       status);
}

}  // namespace mpc
