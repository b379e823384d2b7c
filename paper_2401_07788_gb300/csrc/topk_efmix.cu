// topk_efmix.cu -- EF-mixed TopK (§2.4): the k sent entries are split between
// the input and the error buffer, half each, and x + err is sent on them; the
// buffer keeps x + err everywhere else.  The input's share is its ceil(k/2)
// largest |x|; the buffer's share its floor(k/2) largest |err| among the other
// entries, so that exactly k entries are sent.
//
// The abi runs it as: TopK of x (ceil(k/2)) -> mark those entries of err with
// +inf, saving their values -> TopK of err (k): the marked entries and the
// floor(k/2) largest of the rest, in ascending index -> restore err ->
// err = x + err -> gather the sent values from err and zero them there.  The
// kernels below are the four small steps between the two TopK calls; each is
// bound by HBM.
#include <cstdint>

#include "common.cuh"
#include "kernels.h"

namespace mpc {
namespace {

constexpr int kT = 256;
constexpr int kPer = 4;  // payload entries per thread per block pass

// Blocks of kT * kPer payload entries of one row (bpr blocks per row).
__device__ __forceinline__ void payload_block(int bpr, int64_t k, int64_t* row, int64_t* i0) {
  *row = blockIdx.x / bpr;
  *i0 = static_cast<int64_t>(blockIdx.x % bpr) * (kT * kPer);
}

// restore == 0: saved[r][i] = err[r][idx[r][i]] and err there = +inf.
// restore == 1: err[r][idx[r][i]] = saved[r][i].
__global__ void __launch_bounds__(kT)
    efmix_mark_kernel(float* __restrict__ err, const int32_t* __restrict__ idx, int64_t L,
                      int64_t k, int bpr, float* __restrict__ saved, int restore) {
  pdl_begin();
  int64_t row, i0;
  payload_block(bpr, k, &row, &i0);
  float* er = err + row * L;
#pragma unroll
  for (int u = 0; u < kPer; ++u) {
    const int64_t i = i0 + u * kT + threadIdx.x;
    if (i >= k) break;
    const int64_t c = idx[row * k + i];
    if (c < 0 || c >= L) continue;
    if (restore) {
      er[c] = saved[row * k + i];
    } else {
      saved[row * k + i] = er[c];
      er[c] = __int_as_float(0x7f800000);
    }
  }
}

// err = x + err (one fp32 round-to-nearest add per entry), 16-byte accesses
// when both are aligned and the count is a multiple of 4.
__global__ void __launch_bounds__(kT)
    efmix_add_kernel(const float* __restrict__ x, float* __restrict__ err, int64_t n, int vec) {
  pdl_begin();
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kT;
  if (vec) {
    const int64_t n4 = n / 4;
    for (int64_t q = blockIdx.x * static_cast<int64_t>(kT) + threadIdx.x; q < n4; q += stride) {
      const float4 a = reinterpret_cast<const float4*>(x)[q];
      float4 b = reinterpret_cast<float4*>(err)[q];
      b.x = fadd(a.x, b.x);
      b.y = fadd(a.y, b.y);
      b.z = fadd(a.z, b.z);
      b.w = fadd(a.w, b.w);
      reinterpret_cast<float4*>(err)[q] = b;
    }
  } else {
    for (int64_t i = blockIdx.x * static_cast<int64_t>(kT) + threadIdx.x; i < n; i += stride)
      err[i] = fadd(x[i], err[i]);
  }
}

// vals[r][i] = err[r][idx[r][i]] (which holds x + err), then +0 there.
__global__ void __launch_bounds__(kT)
    efmix_send_kernel(float* __restrict__ err, const int32_t* __restrict__ idx, int64_t L,
                      int64_t k, int bpr, float* __restrict__ vals) {
  pdl_begin();
  int64_t row, i0;
  payload_block(bpr, k, &row, &i0);
  float* er = err + row * L;
#pragma unroll
  for (int u = 0; u < kPer; ++u) {
    const int64_t i = i0 + u * kT + threadIdx.x;
    if (i >= k) break;
    const int64_t c = idx[row * k + i];
    if (c < 0 || c >= L) {
      vals[row * k + i] = 0.0f;
      continue;
    }
    vals[row * k + i] = er[c];
    er[c] = 0.0f;
  }
}

int blocks_per_row(int64_t k) { return static_cast<int>((k + kT * kPer - 1) / (kT * kPer)); }

}  // namespace

cudaError_t launch_efmix_mark(float* err, const int32_t* idx, int64_t rows, int64_t L, int64_t k,
                              float* saved, int restore, cudaStream_t s) {
  if (rows <= 0 || k <= 0) return cudaSuccess;
  const int bpr = blocks_per_row(k);
  if (rows * bpr > 0x7fffffffLL) return cudaErrorInvalidValue;
  efmix_mark_kernel<<<static_cast<unsigned>(rows * bpr), kT, 0, s>>>(err, idx, L, k, bpr, saved,
                                                                      restore);
  return cudaGetLastError();
}

cudaError_t launch_efmix_add(const float* x, float* err, int64_t n, int num_sms, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int vec = (n % 4 == 0) && (reinterpret_cast<uintptr_t>(x) % 16 == 0) &&
                  (reinterpret_cast<uintptr_t>(err) % 16 == 0);
  const int64_t want = ((vec ? n / 4 : n) + kT - 1) / kT;
  const int64_t cap = static_cast<int64_t>(num_sms) * 16;
  efmix_add_kernel<<<static_cast<unsigned>(want < cap ? want : cap), kT, 0, s>>>(x, err, n, vec);
  return cudaGetLastError();
}

cudaError_t launch_efmix_send(float* err, const int32_t* idx, int64_t rows, int64_t L, int64_t k,
                              float* vals, cudaStream_t s) {
  if (rows <= 0 || k <= 0) return cudaSuccess;
  const int bpr = blocks_per_row(k);
  if (rows * bpr > 0x7fffffffLL) return cudaErrorInvalidValue;
  efmix_send_kernel<<<static_cast<unsigned>(rows * bpr), kT, 0, s>>>(err, idx, L, k, bpr, vals);
  return cudaGetLastError();
}

}  // namespace mpc
