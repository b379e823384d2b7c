// topk_decompress.cu -- TopK decompression (§2.3: the kept values are put back
// at their indices and every other entry is zero) and the AQ-SGD receiver's
// buffer update (§2.5).
//
// Rows of up to 65536 entries: one CTA owns whole rows, zero-fills them with
// 16-byte stores and, after a block barrier, stores the kept values over the
// zeros; both writes of a line meet in L2, so HBM sees each output byte once.
// Longer rows: each output tile is built in shared memory (zero fill, scatter
// of the tile's kept entries, found by a block-parallel search of the row's
// ascending indices) and written once.
//
// Also here: the gather of TopK index reuse (§3.2), the payload of a second
// tensor at the indices kept for the first.
#include "common.cuh"
#include "kernels.h"
#include "launch_util.h"

namespace mpc {
namespace {

constexpr int kTile = 16384;  // floats per output tile (64 KiB of shared memory)
constexpr int kDecThreads = 256;

// Number of entries of idx[0..n) that are < target, for ascending idx;
// every thread of the block returns the same value.
__device__ int64_t block_lower_bound(const int32_t* idx, int64_t n, int64_t target) {
  int64_t lo = 0, hi = n;
  while (lo < hi) {
    const int64_t span = hi - lo;
    const int64_t stride = (span + kDecThreads - 1) / kDecThreads;
    const int64_t p = lo + static_cast<int64_t>(threadIdx.x) * stride;
    const bool pred = p < hi && static_cast<int64_t>(idx[p]) < target;
    const int c = __syncthreads_count(pred);
    if (c == 0) {
      hi = lo;
    } else {
      const int64_t last = lo + static_cast<int64_t>(c - 1) * stride;
      hi = min(hi, lo + static_cast<int64_t>(c) * stride);
      lo = last + 1;
    }
  }
  return lo;
}

// rpc rows per CTA when tpr == 1; tpr column tiles per row when rpc == 1.
__global__ void __launch_bounds__(kDecThreads)
    topk_decompress_kernel(const float* __restrict__ vals, const int32_t* __restrict__ idx,
                           int64_t rows, int64_t L, int64_t k, float* __restrict__ y,
                           int64_t rpc, int64_t tpr, int aligned) {
  pdl_begin();
  extern __shared__ __align__(16) float tile[];  // kTile floats
  const int tid = threadIdx.x;
  const int64_t g = blockIdx.x;
  int64_t r0, nrows, c0, ncols, e_begin, e_end;
  if (tpr == 1) {
    r0 = g * rpc;
    nrows = min(rpc, rows - r0);
    c0 = 0;
    ncols = L;
    e_begin = r0 * k;
    e_end = (r0 + nrows) * k;
  } else {
    r0 = g / tpr;
    nrows = 1;
    c0 = (g % tpr) * kTile;
    ncols = min64(kTile, L - c0);
    const int32_t* ri = idx + r0 * k;
    const int64_t lb0 = block_lower_bound(ri, k, c0);
    const int64_t lb1 = block_lower_bound(ri, k, c0 + ncols);
    e_begin = r0 * k + lb0;
    e_end = r0 * k + max(lb0, lb1);
  }
  const int64_t cells = nrows * ncols;  // <= kTile
  for (int64_t i = tid; i < (cells + 3) / 4; i += kDecThreads)
    reinterpret_cast<float4*>(tile)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  __syncthreads();
  for (int64_t e = e_begin + tid; e < e_end; e += kDecThreads) {
    // rpc * k <= kTile, so the 32-bit quotient is exact
    const int64_t lr =
        (tpr == 1) ? static_cast<uint32_t>(e - e_begin) / static_cast<uint32_t>(k) : 0u;
    const int64_t col = static_cast<int64_t>(idx[e]) - c0;
    if (col >= 0 && col < ncols) tile[lr * ncols + col] = vals[e];
  }
  __syncthreads();
  float* dst = y + r0 * L + c0;
  if (aligned) {
    const int64_t n4 = cells / 4;
    for (int64_t i = tid; i < n4; i += kDecThreads)
      reinterpret_cast<float4*>(dst)[i] = reinterpret_cast<const float4*>(tile)[i];
    for (int64_t i = n4 * 4 + tid; i < cells; i += kDecThreads) dst[i] = tile[i];
  } else {
    for (int64_t i = tid; i < cells; i += kDecThreads) dst[i] = tile[i];
  }
}

// Rows of up to 65536 entries: a CTA owns either whole rows [r0, r0 + nrows)
// (rpc rows, rpc * row_len <= kRowsPerCta) or the column range
// [part * pw, part * pw + pw) of one row (ppr parts per row).  It zero-fills
// its region, then stores the kept values that fall in it; a part brackets
// its own payload entries with one round of probes of the row's ascending
// indices and reads that range with 16-byte loads several deep.
constexpr int64_t kRowsPerCta = 16384;
constexpr int64_t kPartWidth = 8192;

__global__ void __launch_bounds__(kDecThreads)
    topk_decompress_rows_kernel(const float* __restrict__ vals, const int32_t* __restrict__ idx,
                                int64_t rows, int64_t L, int64_t k, float* __restrict__ y,
                                int64_t rpc, int64_t ppr, int64_t pw, int aligned, int vec) {
  pdl_begin();
  const int tid = threadIdx.x;
  int64_t r0, nrows, c0, ncols;
  if (ppr == 1) {
    r0 = static_cast<int64_t>(blockIdx.x) * rpc;
    nrows = min64(rpc, rows - r0);
    c0 = 0;
    ncols = L;
  } else {
    r0 = blockIdx.x / ppr;
    nrows = 1;
    c0 = (blockIdx.x % ppr) * pw;
    ncols = min64(pw, L - c0);
  }
  float* dst = y + r0 * L + c0;
  if (ppr == 1) {
    const int64_t cells = nrows * L;
    if (aligned) {
      const int64_t n4 = cells / 4;
      float4* d4 = reinterpret_cast<float4*>(dst);
      for (int64_t i = tid; i < n4; i += kDecThreads) d4[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int64_t i = n4 * 4 + tid; i < cells; i += kDecThreads) dst[i] = 0.0f;
    } else {
      for (int64_t i = tid; i < cells; i += kDecThreads) dst[i] = 0.0f;
    }
  } else {
    if (aligned) {
      const int64_t n4 = ncols / 4;
      float4* d4 = reinterpret_cast<float4*>(dst);
      for (int64_t i = tid; i < n4; i += kDecThreads) d4[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int64_t i = n4 * 4 + tid; i < ncols; i += kDecThreads) dst[i] = 0.0f;
    } else {
      for (int64_t i = tid; i < ncols; i += kDecThreads) dst[i] = 0.0f;
    }
  }
  __syncthreads();  // the zeros of this block precede its kept values
  const int64_t e_begin = r0 * k;
  const uint32_t nk = static_cast<uint32_t>(nrows * k);  // <= 65536
  const uint32_t k32 = static_cast<uint32_t>(k);
  const float* vr = vals + e_begin;
  const int32_t* ir = idx + e_begin;
  // A part of a long row needs the payload entries of its columns only: one
  // round of evenly spaced probes of the ascending indices brackets them (to
  // within one probe spacing each side; the column test drops the rest).
  uint32_t e_lo = 0, e_hi = nk;
  if (ppr > 1 && nk >= 4 * kDecThreads) {
    const uint32_t stride = (nk + kDecThreads - 1) / kDecThreads;
    const uint32_t p = static_cast<uint32_t>(tid) * stride;
    const bool in = p < nk;
    const int64_t v = in ? static_cast<int64_t>(ir[p]) : 0;
    const uint32_t c_lo = static_cast<uint32_t>(__syncthreads_count(in && v < c0));
    const uint32_t c_hi = static_cast<uint32_t>(__syncthreads_count(in && v < c0 + ncols));
    e_lo = c_lo > 0 ? (c_lo - 1) * stride : 0u;
    e_hi = min(nk, c_hi * stride);
  }
  if (vec) {
    // 4 entries per 16-byte load, kU loads in flight per thread
    constexpr int kU = 4;
    const uint32_t n4 = min(nk / 4, (e_hi + 3) / 4);
    for (uint32_t b = e_lo / 4 + tid; b < n4; b += kDecThreads * kU) {
      int4 iv[kU];
      float4 fv[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const uint32_t q = b + u * kDecThreads;
        if (q < n4) {
          iv[u] = reinterpret_cast<const int4*>(ir)[q];
          fv[u] = reinterpret_cast<const float4*>(vr)[q];
        }
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const uint32_t q = b + u * kDecThreads;
        if (q < n4) {
          const int ci[4] = {iv[u].x, iv[u].y, iv[u].z, iv[u].w};
          const float cv[4] = {fv[u].x, fv[u].y, fv[u].z, fv[u].w};
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const uint32_t e = 4 * q + t;
            const uint32_t lr = (ppr == 1) ? e / k32 : 0u;
            const int64_t col = static_cast<int64_t>(ci[t]) - c0;
            if (col >= 0 && col < ncols) dst[static_cast<int64_t>(lr) * L + col] = cv[t];
          }
        }
      }
    }
    for (uint32_t e = 4 * (nk / 4) + tid; e < e_hi; e += kDecThreads) {
      const uint32_t lr = (ppr == 1) ? e / k32 : 0u;
      const int64_t col = static_cast<int64_t>(ir[e]) - c0;
      if (col >= 0 && col < ncols) dst[static_cast<int64_t>(lr) * L + col] = vr[e];
    }
  } else {
    for (uint32_t e = e_lo + tid; e < e_hi; e += kDecThreads) {
      const uint32_t lr = (ppr == 1) ? e / k32 : 0u;
      const int64_t col = static_cast<int64_t>(ir[e]) - c0;
      if (col >= 0 && col < ncols) dst[static_cast<int64_t>(lr) * L + col] = vr[e];
    }
  }
}

// TopK index reuse (§3.2, Table 5): vals[r][i] = g[r][idx[r][i]].  A block
// covers kGU x 4 x 256 consecutive payload entries of one row (bpr blocks per
// row): 16-byte index loads and value stores when every row's payload starts
// 16-byte aligned, the gathered values fetched by independent 4-byte loads
// (ascending within a row, so neighbouring lanes mostly share sectors).  An
// index outside [0, L) reads nothing: its value is +0 and STATUS_BAD_INDEX is
// recorded.
constexpr int kGU = 4;

__global__ void __launch_bounds__(kDecThreads)
    topk_gather_kernel(const float* __restrict__ g, const int32_t* __restrict__ idx,
                       int64_t L, int64_t k, int bpr, float* __restrict__ vals, int vec,
                       unsigned* status) {
  pdl_begin();
  const int64_t row = blockIdx.x / bpr;
  const int64_t q0 = static_cast<int64_t>(blockIdx.x % bpr) * (kDecThreads * kGU);
  const float* gr = g + row * L;
  const int32_t* ir = idx + row * k;
  float* vr = vals + row * k;
  bool bad = false;
  if (vec) {
    const int64_t n4 = k / 4;
    int4 iv[kGU];
#pragma unroll
    for (int u = 0; u < kGU; ++u) {
      const int64_t q = q0 + u * kDecThreads + threadIdx.x;
      iv[u] = (q < n4) ? reinterpret_cast<const int4*>(ir)[q] : make_int4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < kGU; ++u) {
      const int64_t q = q0 + u * kDecThreads + threadIdx.x;
      if (q < n4) {
        const int c[4] = {iv[u].x, iv[u].y, iv[u].z, iv[u].w};
        float o[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const bool ok = c[t] >= 0 && c[t] < L;
          o[t] = ok ? gr[c[t]] : 0.0f;
          bad |= !ok;
        }
        reinterpret_cast<float4*>(vr)[q] = make_float4(o[0], o[1], o[2], o[3]);
      }
    }
  } else {
    for (int u = 0; u < 4 * kGU; ++u) {
      const int64_t i = 4 * q0 + u * kDecThreads + threadIdx.x;
      if (i < k) {
        const int c = ir[i];
        const bool ok = c >= 0 && c < L;
        vr[i] = ok ? gr[c] : 0.0f;
        bad |= !ok;
      }
    }
  }
  if (bad) set_status(status, STATUS_BAD_INDEX);
}

// One CTA per logical payload row: buf_recv[s][r][idx] += vals.
__global__ void __launch_bounds__(kDecThreads)
    aqsgd_decompress_kernel(const float* __restrict__ vals, const int32_t* __restrict__ idx,
                            float* __restrict__ buf, int64_t num_samples,
                            const int64_t* __restrict__ ids, int64_t rps, int64_t L, int64_t k,
                            unsigned* status) {
  pdl_begin();
  const int64_t lr = blockIdx.x;
  const int64_t sid = ids[lr / rps];
  if (sid < 0 || sid >= num_samples) {
    if (threadIdx.x == 0) set_status(status, STATUS_BAD_SAMPLE);
    return;
  }
  float* brow = buf + (sid * rps + lr % rps) * L;
  const float* v = vals + lr * k;
  const int32_t* ix = idx + lr * k;
  for (int64_t i = threadIdx.x; i < k; i += kDecThreads) {
    const int64_t c = ix[i];
    if (c >= 0 && c < L) brow[c] = fadd(brow[c], v[i]);
  }
}

}  // namespace

cudaError_t launch_topk_decompress(const float* vals, const int32_t* idx, int64_t rows,
                                   int64_t L, int64_t k, float* y, int aligned, int num_sms,
                                   cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (L <= 65536) {
    int64_t rpc = 1, ppr = 1, pw = kPartWidth, blocks;
    if (L <= kRowsPerCta) {
      rpc = max64(1, min64(rows, kRowsPerCta / L));
      blocks = (rows + rpc - 1) / rpc;
    } else {
      ppr = (L + kPartWidth - 1) / kPartWidth;
      blocks = rows * ppr;
    }
    // Too few blocks for the GPU: rows of 4096 entries or more split into
    // narrower parts (at least 2048 columns, multiples of 4) up to about two
    // blocks per SM.
    if (blocks < 2 * num_sms && L >= 4096) {
      const int64_t want = min64((L + 2047) / 2048, (2 * num_sms + rows - 1) / rows);
      if (want > ppr) {
        rpc = 1;
        pw = ((L + want - 1) / want + 3) / 4 * 4;
        ppr = (L + pw - 1) / pw;
        blocks = rows * ppr;
      }
    }
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
    // 16-byte payload loads when every block's payload range is 16-byte aligned
    const int vec = (k % 4 == 0) && (reinterpret_cast<uintptr_t>(vals) % 16 == 0) &&
                    (reinterpret_cast<uintptr_t>(idx) % 16 == 0);
    return launch_kernel(topk_decompress_rows_kernel, dim3(static_cast<unsigned>(blocks)),
                         dim3(kDecThreads), 0, s, 0u, vals, idx, rows, L, k, y, rpc, ppr, pw,
                         aligned, vec);
  }
  int64_t rpc = 1, tpr = 1, blocks;
  if (L <= kTile) {
    rpc = kTile / L;
    if (rpc > rows) rpc = rows;
    blocks = (rows + rpc - 1) / rpc;
  } else {
    tpr = (L + kTile - 1) / kTile;
    blocks = rows * tpr;
  }
  if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
  const int smem = kTile * 4;
  cudaError_t err = ensure_dynamic_smem(topk_decompress_kernel, smem);
  if (err != cudaSuccess) return err;
  topk_decompress_kernel<<<static_cast<unsigned>(blocks), kDecThreads, smem, s>>>(
      vals, idx, rows, L, k, y, rpc, tpr, aligned);
  return cudaGetLastError();
}

cudaError_t launch_topk_gather(const float* g, const int32_t* idx, int64_t rows, int64_t L,
                              int64_t k, float* vals, unsigned* status, cudaStream_t s) {
  if (rows <= 0 || k <= 0) return cudaSuccess;
  const int vec = (k % 4 == 0) && (reinterpret_cast<uintptr_t>(idx) % 16 == 0) &&
                  (reinterpret_cast<uintptr_t>(vals) % 16 == 0);
  const int64_t per_block = static_cast<int64_t>(kDecThreads) * kGU * 4;
  const int64_t bpr = (k + per_block - 1) / per_block;
  if (rows * bpr > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_kernel(topk_gather_kernel, dim3(static_cast<unsigned>(rows * bpr)),
                       dim3(kDecThreads), 0, s, 0u, g, idx, L, k, static_cast<int>(bpr), vals, vec,
                       status);
}

cudaError_t launch_aqsgd_decompress(const float* vals, const int32_t* idx, float* buf,
                                    int64_t num_samples, const int64_t* ids, int64_t n_ids,
                                    int64_t rps, int64_t L, int64_t k, unsigned* status,
                                    int num_sms, cudaStream_t s) {
  (void)num_sms;
  const int64_t rows = n_ids * rps;
  if (rows <= 0) return cudaSuccess;
  if (rows > 0x7fffffffLL) return cudaErrorInvalidValue;
  aqsgd_decompress_kernel<<<static_cast<unsigned>(rows), kDecThreads, 0, s>>>(
      vals, idx, buf, num_samples, ids, rps, L, k, status);
  return cudaGetLastError();
}

}  // namespace mpc
