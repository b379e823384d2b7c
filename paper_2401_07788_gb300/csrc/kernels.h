// kernels.h -- host-side launch interface between the C ABI (abi.cu) and the
// kernel translation units.  Internal to libmpcomp.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace mpc {

// Which fused variant of the TopK selection a launch runs.
enum TopkMode : int {
  kPlain = 0,  // select on x
  kEF = 1,     // select on s = x + err; err <- kept ? +0 : s         (§2.4, Seide)
  kDelta = 2,  // select on d = x - state; state[kept] += d[kept]   (§2.4 EF21, §2.5 AQ-SGD)
};

struct TopkRowArgs {
  const float* x;         // [rows][L] logical rows
  float* aux;             // kEF: err [rows][L]; kDelta: state rows (see ids)
  const int64_t* ids;     // kDelta: per-sample ids [rows / rps] (nullptr = identity map)
  int64_t rows;           // logical rows
  int64_t L;              // row length
  int64_t k;              // kept per row
  int64_t rps;            // kDelta with ids: rows per sample
  int64_t num_samples;    // kDelta with ids: buffer samples
  float* vals;            // [rows][k]
  int32_t* idx;           // [rows][k]
  int64_t slice;          // CTA kernel: elements per CTA slice (multiple of 4)
  int aligned;            // 1: every row start is 16-byte aligned (bulk copies allowed)
  uint32_t spin_limit;    // polls before a wait gives up
  unsigned* status;       // device status word
  int wide_cta;           // 1: rows of 8193..32768 entries may take one wide CTA each
  int band;               // 1: rows of 1025..8192 entries take the band kernel
};

// Largest row the on-chip row path handles (cluster of 8 CTAs x 8192).
constexpr int64_t kRowPathMaxLen = 65536;

// Launch the on-chip row TopK path.  Returns a CUDA error code.
cudaError_t launch_topk_rows(int mode, const TopkRowArgs& a, int num_sms, cudaStream_t s);
cudaError_t launch_topk_rows_plain(const TopkRowArgs& a, int num_sms, cudaStream_t s);
cudaError_t launch_topk_rows_ef(const TopkRowArgs& a, int num_sms, cudaStream_t s);
cudaError_t launch_topk_rows_delta(const TopkRowArgs& a, int num_sms, cudaStream_t s);

struct TopkGridArgs {
  const float* x;
  float* aux;
  int64_t rows, L, k;
  float* vals;
  int32_t* idx;
  void* ws;
  size_t ws_bytes;
  uint32_t spin_limit;
  unsigned* status;
};
size_t topk_grid_workspace_bytes(int64_t rows, int64_t L, int64_t k);
cudaError_t launch_topk_grid(int mode, const TopkGridArgs& a, int num_sms, cudaStream_t s);

cudaError_t launch_topk_decompress(const float* vals, const int32_t* idx, int64_t rows,
                                   int64_t L, int64_t k, float* y, int aligned, int num_sms,
                                   cudaStream_t s);
// AQ-SGD with quantisation (§2.5), aqsgd_quant.cu: d = x - buf[id, r], and
// buf[id, r] += Dequant(codes).
cudaError_t launch_aqsgd_delta(const float* x, const float* buf, const int64_t* ids, int64_t n_ids,
                               int64_t rps, int64_t L, int64_t num_samples, float* d,
                               unsigned* status, cudaStream_t s);
cudaError_t launch_aqsgd_dequant_add(const uint32_t* codes, const float* scale, const float* minv,
                                     float* buf, const int64_t* ids, int64_t n_ids, int64_t rps,
                                     int64_t L, int64_t W, int bits, int64_t num_samples,
                                     unsigned* status, cudaStream_t s);

// EF-mixed (§2.4): the steps between its two TopK calls (topk_efmix.cu).
cudaError_t launch_efmix_mark(float* err, const int32_t* idx, int64_t rows, int64_t L, int64_t k,
                              float* saved, int restore, cudaStream_t s);
cudaError_t launch_efmix_add(const float* x, float* err, int64_t n, int num_sms, cudaStream_t s);
cudaError_t launch_efmix_send(float* err, const int32_t* idx, int64_t rows, int64_t L, int64_t k,
                              float* vals, cudaStream_t s);
cudaError_t launch_topk_gather(const float* g, const int32_t* idx, int64_t rows, int64_t L,
                              int64_t k, float* vals, unsigned* status, cudaStream_t s);
cudaError_t launch_aqsgd_decompress(const float* vals, const int32_t* idx, float* buf,
                                    int64_t num_samples, const int64_t* ids, int64_t n_ids,
                                    int64_t rps, int64_t L, int64_t k, unsigned* status,
                                    int num_sms, cudaStream_t s);

struct QuantArgs {
  const float* x;
  int64_t rows, L;
  int bits;
  int stochastic;
  uint64_t seed;
  uint32_t* codes;
  float* scale;
  float* minv;
  int64_t W;        // words per code row
  int64_t slice;    // elements per CTA slice (multiple of 128)
  int aligned;      // rows of x 16-byte aligned
  void* ws;         // multi-pass path: [rows] x {min key, max key}
  uint32_t spin_limit;
  unsigned* status;
  // quantised AQ-SGD in one pass (aq_buf != nullptr): the rows quantised are
  // d = x - aq_buf[id, r] (id = aq_ids[row / aq_rps], r = row % aq_rps), and
  // aq_buf[id, r] += dequant(codes) is written in the same pass
  float* aq_buf = nullptr;
  const int64_t* aq_ids = nullptr;
  int64_t aq_rps = 1;
  int64_t aq_num_samples = 0;
};
constexpr int64_t kQuantRowPathMaxLen = 65536;
// Quantised AQ-SGD in one pass where the shape allows (2/4/8-bit codes, rows of
// up to 4096 entries); cudaErrorNotSupported otherwise (nothing launched).
cudaError_t launch_aqsgd_quant_fused(const QuantArgs& a, int num_sms, cudaStream_t s);
size_t quant_workspace_bytes(int64_t rows, int64_t L, int bits);
cudaError_t launch_quant_compress(const QuantArgs& a, int num_sms, cudaStream_t s);
// Allocation-free variant: the min/max scratch is a static device array.
int64_t quant_noalloc_max_rows();
cudaError_t launch_quant_compress_noalloc(const QuantArgs& a, int num_sms, cudaStream_t s);
cudaError_t launch_quant_decompress(const uint32_t* codes, const float* scale,
                                    const float* minv, int64_t rows, int64_t L, int bits,
                                    int64_t W, float* y, int aligned, int num_sms,
                                    cudaStream_t s);

}  // namespace mpc
