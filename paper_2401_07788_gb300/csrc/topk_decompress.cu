// topk_decompress.cu -- TopK decompression (§2.3: the kept values are put back
// at their indices and every other entry is zero) and the AQ-SGD receiver's
// buffer update (§2.5).
//
// Every output tile (up to 8192 floats: whole short rows, or consecutive
// columns of a long row) is built in shared memory: zero fill, the kept values
// scattered in, then one coalesced copy to the output.
//
// Also here: the gather of TopK index reuse (§3.2), the payload of a second
// tensor at the indices kept for the first.
#include "common.cuh"
#include "kernels.h"
#include "launch_util.h"

namespace mpc {
namespace {

constexpr int kDecThreads = 256;
constexpr int kDT = 8192;  // floats per output tile (32 KiB of shared memory)

// Lower bound of target in the ascending a[0..n), by one warp: 32 probes a
// round narrow the range 32-fold.  Every lane returns the same value (some
// position in [0, n] if a is not ascending).
__device__ int64_t warp_lower_bound(const int32_t* a, int64_t n, int64_t target, int lane) {
  int64_t lo = 0, hi = n;  // the bound lies in [lo, hi]
  while (hi - lo > 32) {
    const int64_t step = (hi - lo + 31) / 32;
    const int64_t q = lo + (lane + 1) * step - 1;
    const bool below = q < hi && static_cast<int64_t>(a[q]) < target;
    const int c = __popc(__ballot_sync(kFull, below));
    const int64_t nlo = lo + c * step;
    hi = min64(hi, lo + (c + 1) * step - 1);
    lo = nlo;
  }
  const int64_t q = lo + lane;
  const bool below = q < hi && static_cast<int64_t>(a[q]) < target;
  return lo + __popc(__ballot_sync(kFull, below));
}

// Decompression by output tiles of kDT floats built in shared memory: zero
// fill, the kept values scattered into the tile, then one coalesced copy of
// the tile to y (so every output byte is written once, with whole lines).
// Rows of at most kDT entries: a tile holds rpt whole rows, whose payload is
// the contiguous range [r0 * k, (r0 + rpt) * k).  Longer rows: tpr tiles of
// consecutive columns per row; the payload entries of a tile are the next ones
// of the row's ascending indices below the tile's end.  Persistent CTAs each
// take a contiguous range of tiles and carry the payload position from tile to
// tile, so only a CTA whose first tile starts inside a row searches for it.
template <bool SHORT>
__global__ void __launch_bounds__(kDecThreads)
    topk_decompress_tiles_kernel(const float* __restrict__ vals, const int32_t* __restrict__ idx,
                                 int64_t rows, int64_t L, int64_t k, float* __restrict__ y,
                                 int64_t rpt, int64_t tpr, int64_t ntiles, int aligned) {
  pdl_begin();
  extern __shared__ __align__(16) float tile[];  // kDT floats
  __shared__ int64_t s_pos;
  __shared__ int s_cnt[2][kDecThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t per = (ntiles + gridDim.x - 1) / gridDim.x;
  const int64_t t0 = static_cast<int64_t>(blockIdx.x) * per;
  const int64_t t1 = min64(ntiles, t0 + per);
  constexpr int kB = 8;  // short rows: payload entries a thread per batch
  constexpr int kU = 4;  // long rows: payload entries a thread per round
  const uint32_t Lu = static_cast<uint32_t>(L);
  const uint32_t magic = static_cast<uint32_t>(0xffffffffu / static_cast<uint32_t>(k)) + 1u;
  // Short rows: the first batch of a tile's payload is loaded while the previous
  // tile is copied out (pcol, pv: those loads).
  int32_t pcol[kB];
  float pv[kB];
  auto fetch_short = [&](int64_t t, uint32_t j0, int32_t* col, float* v) {
    const int64_t r0 = t * rpt;
    const uint32_t n = static_cast<uint32_t>(min64(rpt, rows - r0) * k);
    const int64_t e0 = r0 * k;
#pragma unroll
    for (int b = 0; b < kB; ++b) {
      const uint32_t j = j0 + b * kDecThreads;
      col[b] = j < n ? idx[e0 + j] : -1;
      v[b] = j < n ? vals[e0 + j] : 0.0f;
    }
  };
  // long rows: entries pos .. of row r0, columns relative to c0
  auto fetch_long = [&](int64_t r0, int64_t c0, int64_t pos, int64_t* col, float* v) {
    const int32_t* ir = idx + r0 * k;
    const float* vr = vals + r0 * k;
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t e = pos + u * kDecThreads + tid;
      col[u] = e < k ? static_cast<int64_t>(ir[e]) - c0 : -1;
      v[u] = e < k ? vr[e] : 0.0f;
    }
  };
  int64_t pos = 0;  // payload entry of the row where the current tile's entries start
  bool have = false;  // the current tile's first batch is in pcol, pv
  for (int64_t t = t0; t < t1; ++t) {
    int64_t r0, nrows, c0, ncols;
    if (SHORT) {
      r0 = t * rpt;
      nrows = min64(rpt, rows - r0);
      c0 = 0;
      ncols = L;
    } else {
      r0 = t / tpr;
      nrows = 1;
      c0 = (t % tpr) * kDT;
      ncols = min64(kDT, L - c0);
      if (c0 == 0) {
        pos = 0;
      } else if (t == t0) {  // this CTA starts inside the row
        if (warp == 0) {
          const int64_t lb = warp_lower_bound(idx + r0 * k, k, c0, lane);
          if (lane == 0) s_pos = lb;
        }
        __syncthreads();
        pos = s_pos;
      }
    }
    const int64_t cells = nrows * ncols;  // <= kDT
    for (int64_t i = tid; i < (cells + 3) / 4; i += kDecThreads)
      reinterpret_cast<float4*>(tile)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    __syncthreads();
    if (SHORT) {
      // whole rows: the payload range of rows r0 .. r0 + nrows - 1; the local row of
      // entry j is j / k, taken as the high half of j * ceil(2^32 / k) (exact for j and
      // k up to 2^13; k = 1 needs no division).  Batches of kB entries a thread, all of
      // a batch's loads in flight together.
      const uint32_t n = static_cast<uint32_t>(nrows * k);  // <= kDT
      for (uint32_t j0 = tid; j0 < n; j0 += kB * kDecThreads) {
        int32_t col[kB];
        float v[kB];
        if (have && j0 == static_cast<uint32_t>(tid)) {
#pragma unroll
          for (int b = 0; b < kB; ++b) {
            col[b] = pcol[b];
            v[b] = pv[b];
          }
        } else {
          fetch_short(t, j0, col, v);
        }
#pragma unroll
        for (int b = 0; b < kB; ++b) {
          const uint32_t j = j0 + b * kDecThreads;
          const uint32_t lr = k == 1 ? j : __umulhi(j, magic);
          if (col[b] >= 0 && static_cast<uint32_t>(col[b]) < Lu) tile[lr * Lu + col[b]] = v[b];
        }
      }
    } else {
      // a column tile of a long row: the row's next payload entries below c0 + ncols
      // (ascending indices, so they are a prefix of the entries read from pos on)
      for (int it = 0;; ++it) {
        int64_t col[kU];
        float v[kU];
        fetch_long(r0, c0, pos, col, v);
        int cnt = 0;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int64_t e = pos + u * kDecThreads + tid;
          const bool in = e < k && col[u] < ncols;
          if (in && col[u] >= 0) tile[col[u]] = v[u];
          cnt += __popc(__ballot_sync(kFull, in));
        }
        if (lane == 0) s_cnt[it & 1][warp] = cnt;
        __syncthreads();
        int total = 0;
#pragma unroll
        for (int w = 0; w < kDecThreads / 32; ++w) total += s_cnt[it & 1][w];
        pos += total;
        if (total < kU * kDecThreads) break;
      }
    }
    __syncthreads();
    // short rows: the next tile's first payload loads go out before this tile's copy
    // (for long rows this measured slower: the extra registers cost more occupancy
    // than the overlap gains)
    have = false;
    if (SHORT && t + 1 < t1) {
      fetch_short(t + 1, tid, pcol, pv);
      have = true;
    }
    float* dst = y + r0 * L + c0;
    if (aligned) {
      const int64_t n4 = cells / 4;
      for (int64_t i = tid; i < n4; i += kDecThreads)
        reinterpret_cast<float4*>(dst)[i] = reinterpret_cast<const float4*>(tile)[i];
      for (int64_t i = n4 * 4 + tid; i < cells; i += kDecThreads) dst[i] = tile[i];
    } else {
      for (int64_t i = tid; i < cells; i += kDecThreads) dst[i] = tile[i];
    }
    __syncthreads();  // the tile is free for the next one
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
  int64_t rpt = 1, tpr = 1, ntiles;
  if (L <= kDT) {
    rpt = min64(rows, kDT / L);
    ntiles = (rows + rpt - 1) / rpt;
  } else {
    tpr = (L + kDT - 1) / kDT;
    if (rows > INT64_MAX / tpr) return cudaErrorInvalidValue;
    ntiles = rows * tpr;
  }
  constexpr int smem = kDT * 4;
  auto kernel = tpr == 1 ? topk_decompress_tiles_kernel<true> : topk_decompress_tiles_kernel<false>;
  cudaError_t err = ensure_dynamic_smem(kernel, smem);
  if (err != cudaSuccess) return err;
  const int occ = resident_blocks(kernel, kDecThreads, smem);
  const int64_t grid = min64(ntiles, static_cast<int64_t>(num_sms) * occ);
  return launch_kernel(kernel, dim3(static_cast<unsigned>(grid)), dim3(kDecThreads), smem, s, 0u,
                       vals, idx, rows, L, k, y, rpt, tpr, ntiles, aligned);
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
