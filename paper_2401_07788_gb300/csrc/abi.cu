// abi.cu -- the extern "C" entry points of libmpcomp (declared in
// include/mpcomp.h): argument validation, path selection and the device
// status word.  No entry point allocates device memory.
#include <algorithm>
#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "kernels.h"
#include "mpcomp.h"

namespace {

// The library's device status word; kernels get its address.
__device__ unsigned g_status_word = 0;

thread_local char g_last_error[512];
std::atomic<uint32_t> g_spin_limit{1u << 20};
std::atomic<int> g_pdl{1};
std::atomic<int> g_topk_path{0};

constexpr int kMaxDevices = 64;
std::mutex g_dev_mutex;
unsigned* g_status_ptr[kMaxDevices];
int g_num_sms[kMaxDevices];

mpc_status set_error(mpc_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
  va_end(ap);
  return s;
}

mpc_status ok() {
  g_last_error[0] = '\0';
  return MPC_OK;
}

mpc_status cuda_error(cudaError_t e, const char* what) {
  return set_error(MPC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Per-device state, looked up once per device with that device current.
struct Device {
  unsigned* status;
  int num_sms;
};

mpc_status current_device(Device* d) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return set_error(MPC_ERR_UNSUPPORTED, "device %d", dev);
  std::lock_guard<std::mutex> lock(g_dev_mutex);
  if (g_status_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_status_word);
    if (e != cudaSuccess) return cuda_error(e, "cudaGetSymbolAddress(status)");
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_error(e, "cudaDeviceGetAttribute");
    g_num_sms[dev] = sms;
    g_status_ptr[dev] = static_cast<unsigned*>(p);
  }
  d->status = g_status_ptr[dev];
  d->num_sms = g_num_sms[dev];
  return MPC_OK;
}

bool aligned_to(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Code widths: 1..16 bits (§2.2 evaluates 2, 4, 6 and 8), or 32 (raw fp32 passthrough).
bool valid_bits(int bits) { return (bits >= 1 && bits <= 16) || bits == 32; }

mpc_status check_ptr(const void* p, uintptr_t align, const char* name) {
  if (p == nullptr) return set_error(MPC_ERR_INVALID_ARG, "%s is NULL", name);
  if (!aligned_to(p, align))
    return set_error(MPC_ERR_INVALID_ARG, "%s is not %d-byte aligned", name, static_cast<int>(align));
  return MPC_OK;
}

#define MPC_TRY(expr)                  \
  do {                                 \
    mpc_status s_ = (expr);            \
    if (s_ != MPC_OK) return s_;       \
  } while (0)

mpc_status check_shape(int64_t rows, int64_t row_len, int64_t k) {
  if (rows < 0) return set_error(MPC_ERR_INVALID_ARG, "rows=%lld < 0", (long long)rows);
  if (row_len < 1 || row_len > 0x7fffffffLL)
    return set_error(MPC_ERR_INVALID_ARG, "row_len=%lld outside [1, 2^31-1]", (long long)row_len);
  if (k < 1 || k > row_len)
    return set_error(MPC_ERR_INVALID_ARG, "k=%lld outside [1, row_len=%lld]", (long long)k,
                     (long long)row_len);
  if (rows > 0 && row_len > INT64_MAX / rows)
    return set_error(MPC_ERR_INVALID_ARG, "rows*row_len overflows");
  return MPC_OK;
}

bool use_row_path(int64_t row_len) {
  const int forced = g_topk_path.load();
  if (forced == 2) return false;
  return row_len <= mpc::kRowPathMaxLen;
}

// Shared body of the TopK compress entry points.
mpc_status topk_compress_common(int mode, const float* x, float* aux, int64_t rows,
                                int64_t row_len, int64_t k, float* vals, int32_t* idx,
                                void* ws, size_t ws_bytes, cudaStream_t stream) {
  MPC_TRY(check_shape(rows, row_len, k));
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(x, 4, "x"));
  if (mode != mpc::kPlain) MPC_TRY(check_ptr(aux, 4, mode == mpc::kEF ? "err" : "g"));
  MPC_TRY(check_ptr(vals, 4, "vals"));
  MPC_TRY(check_ptr(idx, 4, "idx"));
  Device d;
  MPC_TRY(current_device(&d));
  cudaError_t e;
  if (use_row_path(row_len)) {
    mpc::TopkRowArgs a = {};
    a.wide_cta = g_topk_path.load() != 3;
    a.band = g_topk_path.load() != 4;
    a.x = x;
    a.aux = aux;
    a.rows = rows;
    a.L = row_len;
    a.k = k;
    a.vals = vals;
    a.idx = idx;
    a.aligned = (row_len % 4 == 0) && aligned_to(x, 16) && (aux == nullptr || aligned_to(aux, 16));
    a.spin_limit = g_spin_limit.load();
    a.status = d.status;
    e = mpc::launch_topk_rows(mode, a, d.num_sms, stream);
  } else {
    const size_t need = mpc::topk_grid_workspace_bytes(rows, row_len, k);
    if (need > 0 && (ws == nullptr || ws_bytes < need))
      return set_error(MPC_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                       ws == nullptr ? (size_t)0 : ws_bytes);
    if (ws != nullptr && !aligned_to(ws, 256))
      return set_error(MPC_ERR_INVALID_ARG, "ws is not 256-byte aligned");
    mpc::TopkGridArgs a = {};
    a.x = x;
    a.aux = aux;
    a.rows = rows;
    a.L = row_len;
    a.k = k;
    a.vals = vals;
    a.idx = idx;
    a.ws = ws;
    a.ws_bytes = ws_bytes;
    a.spin_limit = g_spin_limit.load();
    a.status = d.status;
    e = mpc::launch_topk_grid(mode, a, d.num_sms, stream);
    if (e == cudaErrorNotSupported)
      return set_error(MPC_ERR_UNSUPPORTED, "row_len=%lld needs the multi-pass path",
                       (long long)row_len);
  }
  if (e != cudaSuccess) return cuda_error(e, "topk launch");
  return ok();
}

}  // namespace

namespace mpc {
bool pdl_enabled() { return g_pdl.load(std::memory_order_relaxed) != 0; }
}  // namespace mpc

extern "C" {

int mpc_version(void) { return 100; }

size_t mpc_topk_workspace_bytes(int64_t rows, int64_t row_len, int64_t k) {
  if (rows <= 0 || row_len < 1 || k < 1 || k > row_len) return 0;
  if (use_row_path(row_len)) return 0;
  return mpc::topk_grid_workspace_bytes(rows, row_len, k);
}

mpc_status mpc_topk_compress(const float* x, int64_t rows, int64_t row_len, int64_t k,
                             float* vals, int32_t* idx, void* ws, size_t ws_bytes,
                             mpc_stream_t stream) {
  return topk_compress_common(mpc::kPlain, x, nullptr, rows, row_len, k, vals, idx, ws, ws_bytes,
                              reinterpret_cast<cudaStream_t>(stream));
}

mpc_status mpc_ef_topk_compress(const float* x, float* err, int64_t rows, int64_t row_len,
                                int64_t k, float* vals, int32_t* idx, void* ws, size_t ws_bytes,
                                mpc_stream_t stream) {
  return topk_compress_common(mpc::kEF, x, err, rows, row_len, k, vals, idx, ws, ws_bytes,
                              reinterpret_cast<cudaStream_t>(stream));
}

mpc_status mpc_ef21_topk_compress(const float* x, float* g, int64_t rows, int64_t row_len,
                                  int64_t k, float* vals, int32_t* idx, void* ws,
                                  size_t ws_bytes, mpc_stream_t stream) {
  return topk_compress_common(mpc::kDelta, x, g, rows, row_len, k, vals, idx, ws, ws_bytes,
                              reinterpret_cast<cudaStream_t>(stream));
}

mpc_status mpc_topk_decompress(const float* vals, const int32_t* idx, int64_t rows,
                               int64_t row_len, int64_t k, float* y, mpc_stream_t stream) {
  MPC_TRY(check_shape(rows, row_len, k));
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(vals, 4, "vals"));
  MPC_TRY(check_ptr(idx, 4, "idx"));
  MPC_TRY(check_ptr(y, 4, "y"));
  Device d;
  MPC_TRY(current_device(&d));
  const int aligned = (row_len % 4 == 0) && aligned_to(y, 16);
  cudaError_t e = mpc::launch_topk_decompress(vals, idx, rows, row_len, k, y, aligned, d.num_sms,
                                              reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_error(e, "topk_decompress launch");
  return ok();
}

size_t mpc_efmix_workspace_bytes(int64_t rows, int64_t row_len, int64_t k) {
  if (rows <= 0 || row_len <= 0 || k < 1 || k > row_len || rows > INT64_MAX / row_len) return 0;
  const int64_t k1 = k - k / 2;
  const size_t share = (static_cast<size_t>(rows * k1) * 4u + 255u) / 256u * 256u;
  size_t grid = 0;
  if (!use_row_path(row_len))
    grid = std::max(mpc::topk_grid_workspace_bytes(rows, row_len, k1),
                    mpc::topk_grid_workspace_bytes(rows, row_len, k));
  return 2 * share + grid;
}

mpc_status mpc_efmix_topk_compress(const float* x, float* err, int64_t rows, int64_t row_len,
                                   int64_t k, float* vals, int32_t* idx, void* ws,
                                   size_t ws_bytes, mpc_stream_t stream) {
  MPC_TRY(check_shape(rows, row_len, k));
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(x, 4, "x"));
  MPC_TRY(check_ptr(err, 4, "err"));
  MPC_TRY(check_ptr(vals, 4, "vals"));
  MPC_TRY(check_ptr(idx, 4, "idx"));
  const size_t need = mpc_efmix_workspace_bytes(rows, row_len, k);
  if (ws == nullptr || ws_bytes < need)
    return set_error(MPC_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                     ws == nullptr ? (size_t)0 : ws_bytes);
  if (!aligned_to(ws, 256)) return set_error(MPC_ERR_INVALID_ARG, "ws is not 256-byte aligned");
  Device d;
  MPC_TRY(current_device(&d));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int64_t k1 = k - k / 2;
  const size_t share = (static_cast<size_t>(rows * k1) * 4u + 255u) / 256u * 256u;
  int32_t* idx1 = static_cast<int32_t*>(ws);
  float* saved = reinterpret_cast<float*>(static_cast<char*>(ws) + share);
  void* gws = static_cast<char*>(ws) + 2 * share;
  const size_t gws_bytes = ws_bytes - 2 * share;
  // the input's share (its values land in `saved`, which the marking then reuses)
  MPC_TRY(topk_compress_common(mpc::kPlain, x, nullptr, rows, row_len, k1, saved, idx1,
                               gws_bytes ? gws : nullptr, gws_bytes, s));
  cudaError_t e = mpc::launch_efmix_mark(err, idx1, rows, row_len, k1, saved, 0, s);
  if (e != cudaSuccess) return cuda_error(e, "efmix mark launch");
  // the k largest |err| with the input's share at +inf: that share and the
  // buffer's, in ascending index
  MPC_TRY(topk_compress_common(mpc::kPlain, err, nullptr, rows, row_len, k, vals, idx,
                               gws_bytes ? gws : nullptr, gws_bytes, s));
  e = mpc::launch_efmix_mark(err, idx1, rows, row_len, k1, saved, 1, s);
  if (e == cudaSuccess) e = mpc::launch_efmix_add(x, err, rows * row_len, d.num_sms, s);
  if (e == cudaSuccess) e = mpc::launch_efmix_send(err, idx, rows, row_len, k, vals, s);
  if (e != cudaSuccess) return cuda_error(e, "efmix launch");
  return ok();
}

mpc_status mpc_topk_gather(const float* g, int64_t rows, int64_t row_len, const int32_t* idx,
                           int64_t k, float* vals, mpc_stream_t stream) {
  MPC_TRY(check_shape(rows, row_len, k));
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(g, 4, "g"));
  MPC_TRY(check_ptr(idx, 4, "idx"));
  MPC_TRY(check_ptr(vals, 4, "vals"));
  Device d;
  MPC_TRY(current_device(&d));
  cudaError_t e = mpc::launch_topk_gather(g, idx, rows, row_len, k, vals, d.status,
                                          reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_error(e, "topk_gather launch");
  return ok();
}

mpc_status mpc_aqsgd_compress(const float* x, float* buf, int64_t num_samples,
                              const int64_t* sample_ids, int64_t n_ids, int64_t rows_per_sample,
                              int64_t row_len, int64_t k, float* vals, int32_t* idx, void* ws,
                              size_t ws_bytes, mpc_stream_t stream) {
  (void)ws;
  (void)ws_bytes;
  if (n_ids < 0) return set_error(MPC_ERR_INVALID_ARG, "n_ids < 0");
  if (rows_per_sample < 1) return set_error(MPC_ERR_INVALID_ARG, "rows_per_sample < 1");
  if (num_samples < 1) return set_error(MPC_ERR_INVALID_ARG, "num_samples < 1");
  if (n_ids > INT64_MAX / rows_per_sample) return set_error(MPC_ERR_INVALID_ARG, "rows overflow");
  const int64_t rows = n_ids * rows_per_sample;
  MPC_TRY(check_shape(rows, row_len, k));
  if (num_samples > INT64_MAX / rows_per_sample / row_len)
    return set_error(MPC_ERR_INVALID_ARG, "buffer size overflows");
  if (rows == 0) return ok();
  if (row_len > mpc::kRowPathMaxLen)
    return set_error(MPC_ERR_UNSUPPORTED, "AQ-SGD rows longer than %lld",
                     (long long)mpc::kRowPathMaxLen);
  MPC_TRY(check_ptr(x, 4, "x"));
  MPC_TRY(check_ptr(buf, 4, "buf"));
  MPC_TRY(check_ptr(sample_ids, 8, "sample_ids"));
  MPC_TRY(check_ptr(vals, 4, "vals"));
  MPC_TRY(check_ptr(idx, 4, "idx"));
  Device d;
  MPC_TRY(current_device(&d));
  mpc::TopkRowArgs a = {};
  a.wide_cta = g_topk_path.load() != 3;
  a.band = g_topk_path.load() != 4;
  a.x = x;
  a.aux = buf;
  a.ids = sample_ids;
  a.rows = rows;
  a.L = row_len;
  a.k = k;
  a.rps = rows_per_sample;
  a.num_samples = num_samples;
  a.vals = vals;
  a.idx = idx;
  a.aligned = (row_len % 4 == 0) && aligned_to(x, 16) && aligned_to(buf, 16);
  a.spin_limit = g_spin_limit.load();
  a.status = d.status;
  cudaError_t e = mpc::launch_topk_rows(mpc::kDelta, a, d.num_sms,
                                        reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_error(e, "aqsgd launch");
  return ok();
}

mpc_status mpc_aqsgd_decompress(const float* vals, const int32_t* idx, float* buf_recv,
                                int64_t num_samples, const int64_t* sample_ids, int64_t n_ids,
                                int64_t rows_per_sample, int64_t row_len, int64_t k,
                                mpc_stream_t stream) {
  if (n_ids < 0) return set_error(MPC_ERR_INVALID_ARG, "n_ids < 0");
  if (rows_per_sample < 1) return set_error(MPC_ERR_INVALID_ARG, "rows_per_sample < 1");
  if (num_samples < 1) return set_error(MPC_ERR_INVALID_ARG, "num_samples < 1");
  if (n_ids > INT64_MAX / rows_per_sample) return set_error(MPC_ERR_INVALID_ARG, "rows overflow");
  const int64_t rows = n_ids * rows_per_sample;
  MPC_TRY(check_shape(rows, row_len, k));
  if (num_samples > INT64_MAX / rows_per_sample / row_len)
    return set_error(MPC_ERR_INVALID_ARG, "buffer size overflows");
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(vals, 4, "vals"));
  MPC_TRY(check_ptr(idx, 4, "idx"));
  MPC_TRY(check_ptr(buf_recv, 4, "buf_recv"));
  MPC_TRY(check_ptr(sample_ids, 8, "sample_ids"));
  Device d;
  MPC_TRY(current_device(&d));
  cudaError_t e = mpc::launch_aqsgd_decompress(vals, idx, buf_recv, num_samples, sample_ids,
                                               n_ids, rows_per_sample, row_len, k, d.status,
                                               d.num_sms, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_error(e, "aqsgd_decompress launch");
  return ok();
}

size_t mpc_quant_codes_words(int64_t rows, int64_t row_len, int bits) {
  if (rows < 0 || row_len < 1) return 0;
  if (!valid_bits(bits)) return 0;
  const int64_t words = (row_len * bits + 31) / 32;
  return static_cast<size_t>(rows) * static_cast<size_t>((words + 3) / 4 * 4);
}

size_t mpc_quant_workspace_bytes(int64_t rows, int64_t row_len, int bits) {
  if (rows <= 0 || row_len < 1) return 0;
  return mpc::quant_workspace_bytes(rows, row_len, bits);
}

mpc_status mpc_quant_compress(const float* x, int64_t rows, int64_t row_len, int bits,
                              mpc_rounding mode, uint64_t seed, uint32_t* codes, float* scale,
                              float* minv, void* ws, size_t ws_bytes, mpc_stream_t stream) {
  MPC_TRY(check_shape(rows, row_len, 1));
  if (!valid_bits(bits))
    return set_error(MPC_ERR_INVALID_ARG, "bits=%d not in 1..16 or 32", bits);
  if (mode != MPC_ROUND_NEAREST && mode != MPC_ROUND_STOCHASTIC)
    return set_error(MPC_ERR_INVALID_ARG, "rounding mode %d", static_cast<int>(mode));
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(x, 4, "x"));
  MPC_TRY(check_ptr(codes, 4, "codes"));
  MPC_TRY(check_ptr(scale, 4, "scale"));
  MPC_TRY(check_ptr(minv, 4, "minv"));
  const size_t need = mpc::quant_workspace_bytes(rows, row_len, bits);
  if (need > 0 && (ws == nullptr || ws_bytes < need))
    return set_error(MPC_ERR_WORKSPACE, "workspace of %zu bytes needed", need);
  if (need > 0) MPC_TRY(check_ptr(ws, 8, "ws"));
  Device d;
  MPC_TRY(current_device(&d));
  mpc::QuantArgs a = {};
  a.x = x;
  a.rows = rows;
  a.L = row_len;
  a.bits = bits;
  a.stochastic = (mode == MPC_ROUND_STOCHASTIC);
  a.seed = seed;
  a.codes = codes;
  a.scale = scale;
  a.minv = minv;
  a.W = static_cast<int64_t>(mpc_quant_codes_words(1, row_len, bits));
  a.aligned = (row_len % 4 == 0) && aligned_to(x, 16);
  a.ws = need > 0 ? ws : nullptr;
  a.spin_limit = g_spin_limit.load();
  a.status = d.status;
  cudaError_t e = mpc::launch_quant_compress(a, d.num_sms, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_error(e, "quant_compress launch");
  return ok();
}

mpc_status mpc_quant_compress_noalloc(const float* x, int64_t rows, int64_t row_len, int bits,
                                      mpc_rounding mode, uint64_t seed, uint32_t* codes,
                                      float* scale, float* minv, mpc_stream_t stream) {
  MPC_TRY(check_shape(rows, row_len, 1));
  if (!valid_bits(bits))
    return set_error(MPC_ERR_INVALID_ARG, "bits=%d not in 1..16 or 32", bits);
  if (mode != MPC_ROUND_NEAREST && mode != MPC_ROUND_STOCHASTIC)
    return set_error(MPC_ERR_INVALID_ARG, "rounding mode %d", static_cast<int>(mode));
  if (rows > mpc::quant_noalloc_max_rows())
    return set_error(MPC_ERR_INVALID_ARG,
                     "rows=%lld exceeds the %lld rows of the static scratch of "
                     "mpc_quant_compress_noalloc",
                     (long long)rows, (long long)mpc::quant_noalloc_max_rows());
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(x, 4, "x"));
  MPC_TRY(check_ptr(codes, 4, "codes"));
  MPC_TRY(check_ptr(scale, 4, "scale"));
  MPC_TRY(check_ptr(minv, 4, "minv"));
  Device d;
  MPC_TRY(current_device(&d));
  mpc::QuantArgs a = {};
  a.x = x;
  a.rows = rows;
  a.L = row_len;
  a.bits = bits;
  a.stochastic = (mode == MPC_ROUND_STOCHASTIC);
  a.seed = seed;
  a.codes = codes;
  a.scale = scale;
  a.minv = minv;
  a.W = static_cast<int64_t>(mpc_quant_codes_words(1, row_len, bits));
  a.aligned = (row_len % 4 == 0) && aligned_to(x, 16);
  a.spin_limit = g_spin_limit.load();
  a.status = d.status;
  cudaError_t e = mpc::launch_quant_compress_noalloc(a, d.num_sms,
                                                     reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_error(e, "quant_compress_noalloc launch");
  return ok();
}

mpc_status mpc_quant_decompress(const uint32_t* codes, const float* scale, const float* minv,
                                int64_t rows, int64_t row_len, int bits, float* y,
                                mpc_stream_t stream) {
  MPC_TRY(check_shape(rows, row_len, 1));
  if (!valid_bits(bits))
    return set_error(MPC_ERR_INVALID_ARG, "bits=%d not in 1..16 or 32", bits);
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(codes, 4, "codes"));
  MPC_TRY(check_ptr(scale, 4, "scale"));
  MPC_TRY(check_ptr(minv, 4, "minv"));
  MPC_TRY(check_ptr(y, 4, "y"));
  Device d;
  MPC_TRY(current_device(&d));
  const int64_t W = static_cast<int64_t>(mpc_quant_codes_words(1, row_len, bits));
  const int aligned = (row_len % 4 == 0) && aligned_to(y, 16);
  cudaError_t e = mpc::launch_quant_decompress(codes, scale, minv, rows, row_len, bits, W, y,
                                               aligned, d.num_sms,
                                               reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_error(e, "quant_decompress launch");
  return ok();
}

namespace {

// Shared argument checks of the two quantised AQ-SGD calls.
mpc_status check_aqsgd_quant(int64_t num_samples, int64_t n_ids, int64_t rps, int64_t L,
                             int bits, int64_t* rows) {
  if (n_ids < 0) return set_error(MPC_ERR_INVALID_ARG, "n_ids < 0");
  if (rps < 1) return set_error(MPC_ERR_INVALID_ARG, "rows_per_sample < 1");
  if (num_samples < 1) return set_error(MPC_ERR_INVALID_ARG, "num_samples < 1");
  if (n_ids > INT64_MAX / rps) return set_error(MPC_ERR_INVALID_ARG, "rows overflow");
  *rows = n_ids * rps;
  MPC_TRY(check_shape(*rows, L, 1));
  if (!valid_bits(bits))
    return set_error(MPC_ERR_INVALID_ARG, "bits=%d not in 1..16 or 32", bits);
  if (num_samples > INT64_MAX / rps / L)
    return set_error(MPC_ERR_INVALID_ARG, "buffer size overflows");
  return ok();
}

size_t aqsgd_delta_bytes(int64_t rows, int64_t L) {
  return (static_cast<size_t>(rows) * static_cast<size_t>(L) * 4 + 255) / 256 * 256;
}

}  // namespace

size_t mpc_aqsgd_quant_workspace_bytes(int64_t n_ids, int64_t rows_per_sample, int64_t row_len,
                                       int bits) {
  if (n_ids <= 0 || rows_per_sample < 1 || row_len < 1 || !valid_bits(bits)) return 0;
  if (n_ids > INT64_MAX / rows_per_sample) return 0;
  const int64_t rows = n_ids * rows_per_sample;
  if (rows > INT64_MAX / 4 / row_len) return 0;
  return aqsgd_delta_bytes(rows, row_len) + mpc::quant_workspace_bytes(rows, row_len, bits);
}

mpc_status mpc_aqsgd_quant_compress(const float* x, float* buf, int64_t num_samples,
                                    const int64_t* sample_ids, int64_t n_ids,
                                    int64_t rows_per_sample, int64_t row_len, int bits,
                                    mpc_rounding mode, uint64_t seed, uint32_t* codes,
                                    float* scale, float* minv, void* ws, size_t ws_bytes,
                                    mpc_stream_t stream) {
  int64_t rows = 0;
  MPC_TRY(check_aqsgd_quant(num_samples, n_ids, rows_per_sample, row_len, bits, &rows));
  if (mode != MPC_ROUND_NEAREST && mode != MPC_ROUND_STOCHASTIC)
    return set_error(MPC_ERR_INVALID_ARG, "rounding mode %d", static_cast<int>(mode));
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(x, 4, "x"));
  MPC_TRY(check_ptr(buf, 4, "buf"));
  MPC_TRY(check_ptr(sample_ids, 8, "sample_ids"));
  MPC_TRY(check_ptr(codes, 4, "codes"));
  MPC_TRY(check_ptr(scale, 4, "scale"));
  MPC_TRY(check_ptr(minv, 4, "minv"));
  const size_t need = mpc_aqsgd_quant_workspace_bytes(n_ids, rows_per_sample, row_len, bits);
  if (ws == nullptr || ws_bytes < need)
    return set_error(MPC_ERR_WORKSPACE, "workspace of %zu bytes needed", need);
  MPC_TRY(check_ptr(ws, 8, "ws"));
  Device d;
  MPC_TRY(current_device(&d));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // one pass where the shape allows it (2/4/8-bit codes, rows of up to 4096)
  if (mpc::quant_workspace_bytes(rows, row_len, bits) == 0) {
    mpc::QuantArgs a = {};
    a.x = x;
    a.rows = rows;
    a.L = row_len;
    a.bits = bits;
    a.stochastic = (mode == MPC_ROUND_STOCHASTIC);
    a.seed = seed;
    a.codes = codes;
    a.scale = scale;
    a.minv = minv;
    a.W = static_cast<int64_t>(mpc_quant_codes_words(1, row_len, bits));
    a.aligned = (row_len % 4 == 0) && aligned_to(x, 16) && aligned_to(buf, 16);
    a.spin_limit = g_spin_limit.load();
    a.status = d.status;
    a.aq_buf = buf;
    a.aq_ids = sample_ids;
    a.aq_rps = rows_per_sample;
    a.aq_num_samples = num_samples;
    const cudaError_t f = mpc::launch_aqsgd_quant_fused(a, d.num_sms, s);
    if (f == cudaSuccess) return ok();
    if (f != cudaErrorNotSupported) return cuda_error(f, "aqsgd_quant launch");
  }
  // else: d into the workspace, the quantiser on it, then the buffer update
  float* delta = static_cast<float*>(ws);
  const size_t dbytes = aqsgd_delta_bytes(rows, row_len);
  cudaError_t e = mpc::launch_aqsgd_delta(x, buf, sample_ids, n_ids, rows_per_sample, row_len,
                                          num_samples, delta, d.status, s);
  if (e != cudaSuccess) return cuda_error(e, "aqsgd_delta launch");
  MPC_TRY(mpc_quant_compress(delta, rows, row_len, bits, mode, seed, codes, scale, minv,
                             static_cast<char*>(ws) + dbytes, ws_bytes - dbytes, stream));
  const int64_t W = static_cast<int64_t>(mpc_quant_codes_words(1, row_len, bits));
  e = mpc::launch_aqsgd_dequant_add(codes, scale, minv, buf, sample_ids, n_ids, rows_per_sample,
                                    row_len, W, bits, num_samples, d.status, s);
  if (e != cudaSuccess) return cuda_error(e, "aqsgd_dequant_add launch");
  return ok();
}

mpc_status mpc_aqsgd_quant_decompress(const uint32_t* codes, const float* scale,
                                      const float* minv, float* buf_recv, int64_t num_samples,
                                      const int64_t* sample_ids, int64_t n_ids,
                                      int64_t rows_per_sample, int64_t row_len, int bits,
                                      mpc_stream_t stream) {
  int64_t rows = 0;
  MPC_TRY(check_aqsgd_quant(num_samples, n_ids, rows_per_sample, row_len, bits, &rows));
  if (rows == 0) return ok();
  MPC_TRY(check_ptr(codes, 4, "codes"));
  MPC_TRY(check_ptr(scale, 4, "scale"));
  MPC_TRY(check_ptr(minv, 4, "minv"));
  MPC_TRY(check_ptr(buf_recv, 4, "buf_recv"));
  MPC_TRY(check_ptr(sample_ids, 8, "sample_ids"));
  Device d;
  MPC_TRY(current_device(&d));
  const int64_t W = static_cast<int64_t>(mpc_quant_codes_words(1, row_len, bits));
  cudaError_t e = mpc::launch_aqsgd_dequant_add(codes, scale, minv, buf_recv, sample_ids, n_ids,
                                                rows_per_sample, row_len, W, bits, num_samples,
                                                d.status, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_error(e, "aqsgd_dequant_add launch");
  return ok();
}

mpc_status mpc_get_status(mpc_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_error(e, "cudaStreamSynchronize");
  Device d;
  MPC_TRY(current_device(&d));
  unsigned word = 0;
  e = cudaMemcpyFromSymbol(&word, g_status_word, sizeof(word));
  if (e != cudaSuccess) return cuda_error(e, "read status word");
  if (word != 0) {
    const unsigned zero = 0;
    e = cudaMemcpyToSymbol(g_status_word, &zero, sizeof(zero));
    if (e != cudaSuccess) return cuda_error(e, "clear status word");
  }
  if (word & 1u) return set_error(MPC_ERR_TIMEOUT, "a device-side wait gave up (status 0x%x)", word);
  if (word != 0) return set_error(MPC_ERR_DEVICE, "device-side check failed (status 0x%x)", word);
  return ok();
}

const char* mpc_last_error(void) { return g_last_error; }

mpc_status mpc_set_knob(mpc_knob knob, int64_t value) {
  switch (knob) {
    case MPC_KNOB_PDL:
      if (value != 0 && value != 1) return set_error(MPC_ERR_INVALID_ARG, "pdl knob is 0 or 1");
      g_pdl.store(static_cast<int>(value));
      return ok();
    case MPC_KNOB_SPIN_LIMIT:
      if (value < 0 || value > 0xffffffffLL) return set_error(MPC_ERR_INVALID_ARG, "spin limit");
      g_spin_limit.store(static_cast<uint32_t>(value));
      return ok();
    case MPC_KNOB_TOPK_PATH:
      if (value < 0 || value > 4) return set_error(MPC_ERR_INVALID_ARG, "topk path");
      g_topk_path.store(static_cast<int>(value));
      return ok();
    default:
      return set_error(MPC_ERR_INVALID_ARG, "unknown knob %d", static_cast<int>(knob));
  }
}

}  // extern "C"
