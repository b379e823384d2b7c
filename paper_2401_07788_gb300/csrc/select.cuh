// select.cuh -- building blocks of the exact per-row TopK selection.
//
// The selection finds, for one row, the key T of the k-th largest magnitude
// and the number `need` of entries with key T that are kept (lowest columns
// first), so that the kept set is {key > T} plus the first `need` entries
// with key == T (§2.3; equal magnitudes go to the lower column).
//
// It narrows T down in rounds, each a histogram over bins that are monotone
// in the key, so that every bin above the chosen one is kept whole and every
// bin below it is dropped whole:
//   1. bins linear in |x| between 0 and the row's largest magnitude (or the
//      largest of a fixed sample of the row), which spreads typical
//      activations over many bins; magnitudes above the scale share the top bin;
//   2. then bins of equal width over the key range [lo, hi] that is left,
//      256 per round, until one key remains or a bin is taken whole.
// Keys are int: |x| bit pattern (>= 0), or -1 for a slot past the row end.
#pragma once

#include "common.cuh"

namespace mpc {

constexpr int kRoundBins = 256;

// Scale for the first (|x|-linear) histogram of nb bins: nb / max|x|, or 0
// when the row is all zero or its largest magnitude is not a finite normal
// number (then every key is a candidate and only integer rounds are used).
__device__ __forceinline__ float bucket_scale(int maxkey, int nb) {
  if (maxkey <= 0 || maxkey >= 0x7f800000) return 0.0f;
  float s = fdiv(static_cast<float>(nb), __int_as_float(maxkey));
  return (__float_as_uint(s) < 0x7f800000u) ? s : 0.0f;
}

// Bin of a key (>= 0) in the |x|-linear histogram.  Monotone in the key:
// |x| * scale rounds monotonically and truncation is monotone.
__device__ __forceinline__ int bucket_of(int key, float scale, int nb) {
  int b = __float2int_rz(fmul(__int_as_float(key), scale));
  return min(b, nb - 1);
}

// Shift that maps the key range [lo, hi] (hi > lo) onto at most 256 bins.
__device__ __forceinline__ int round_shift(int lo, int hi) {
  uint32_t span = static_cast<uint32_t>(hi - lo);
  return max(0, 24 - __clz(span));
}

struct BinPick {
  int bin;         // chosen bin
  uint32_t above;  // elements in bins above it
  uint32_t count;  // elements in it
};

// One warp: among 256 bins ranked from high to low, find the bin holding the
// kr-th element (1 <= kr <= total).  Lane l scans bins 255-8l down to 248-8l.
__device__ __forceinline__ BinPick warp_pick_bin(const uint32_t* hist, uint32_t kr, int lane) {
  uint32_t c[8];
  uint32_t tsum = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    c[j] = hist[kRoundBins - 1 - (lane * 8 + j)];
    tsum += c[j];
  }
  uint32_t incl = warp_inclusive_scan(tsum, lane);
  uint32_t excl = incl - tsum;
  bool mine = excl < kr && kr <= incl;
  unsigned who = __ballot_sync(kFull, mine);
  int src = who ? __ffs(who) - 1 : 0;
  int b = 0;
  uint32_t ab = 0, cb = 0;
  if (mine) {
    uint32_t run = excl;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (run + c[j] >= kr) {
        b = kRoundBins - 1 - (lane * 8 + j);
        ab = run;
        cb = c[j];
        break;
      }
      run += c[j];
    }
  }
  BinPick p;
  p.bin = __shfl_sync(kFull, b, src);
  p.above = __shfl_sync(kFull, ab, src);
  p.count = __shfl_sync(kFull, cb, src);
  return p;
}

// Result of a selection: kept = {key > T} + first `need` of {key == T}.
struct Threshold {
  int T;
  uint32_t need;
};

// One warp, m <= 64 keys (>= 0) in shared memory: the kr-th largest by
// counting, for each key, how many keys are larger and how many are at least
// as large (T is the key with #greater < kr <= #at-least).
__device__ __forceinline__ Threshold warp_small_select(const int* keys, uint32_t m, uint32_t kr,
                                                       int lane) {
  const int k0 = static_cast<uint32_t>(lane) < m ? keys[lane] : -1;
  const int k1 = static_cast<uint32_t>(lane) + 32u < m ? keys[lane + 32] : -1;
  uint32_t gt0 = 0, ge0 = 0, gt1 = 0, ge1 = 0;
  if (m <= 32) {
#pragma unroll 8
    for (int j = 0; j < 32; ++j) {
      const int a = __shfl_sync(kFull, k0, j);
      gt0 += a > k0;
      ge0 += a >= k0;
    }
  } else {
#pragma unroll 4
    for (int j = 0; j < 32; ++j) {
      const int a = __shfl_sync(kFull, k0, j);
      const int b = __shfl_sync(kFull, k1, j);
      gt0 += (a > k0) + (b > k0);
      ge0 += (a >= k0) + (b >= k0);
      gt1 += (a > k1) + (b > k1);
      ge1 += (a >= k1) + (b >= k1);
    }
  }
  const bool ok0 = static_cast<uint32_t>(lane) < m && gt0 < kr && kr <= ge0;
  const bool ok1 = static_cast<uint32_t>(lane) + 32u < m && gt1 < kr && kr <= ge1;
  const unsigned b0 = __ballot_sync(kFull, ok0);
  const unsigned b1 = __ballot_sync(kFull, ok1);
  Threshold t;
  if (b0) {
    const int src = __ffs(b0) - 1;
    t.T = __shfl_sync(kFull, k0, src);
    t.need = kr - __shfl_sync(kFull, gt0, src);
  } else {
    const int src = b1 ? __ffs(b1) - 1 : 0;
    t.T = __shfl_sync(kFull, k1, src);
    t.need = kr - __shfl_sync(kFull, gt1, src);
  }
  return t;
}

// One warp: among m keys (>= 0) in shared memory, find the kr-th largest
// (1 <= kr <= m) by integer rounds.  whist: 256 words of warp-private scratch.
__device__ __forceinline__ Threshold warp_list_select(const int* keys, uint32_t m, uint32_t kr,
                                                      uint32_t* whist, int lane) {
  int lo = 0x7fffffff, hi = -1;
  for (uint32_t j = lane; j < m; j += 32) {
    int key = keys[j];
    lo = min(lo, key);
    hi = max(hi, key);
  }
  lo = __reduce_min_sync(kFull, lo);
  hi = __reduce_max_sync(kFull, hi);
  Threshold t;
  for (;;) {
    if (lo >= hi) {
      t.T = lo;
      t.need = kr;
      return t;
    }
    const int sh = round_shift(lo, hi);
#pragma unroll
    for (int j = 0; j < 8; ++j) whist[lane * 8 + j] = 0;
    __syncwarp();
    for (uint32_t j = lane; j < m; j += 32) {
      int key = keys[j];
      if (key >= lo && key <= hi) atomicAdd(&whist[static_cast<uint32_t>(key - lo) >> sh], 1u);
    }
    __syncwarp();
    BinPick p = warp_pick_bin(whist, kr, lane);
    __syncwarp();
    kr -= p.above;
    int nlo = lo + (p.bin << sh);
    int nhi = static_cast<int>(min(static_cast<uint32_t>(hi),
                                   static_cast<uint32_t>(nlo) + ((1u << sh) - 1u)));
    if (p.count == kr) {  // the whole bin is kept: threshold just below it
      t.T = nlo - 1;
      t.need = 0;
      return t;
    }
    lo = nlo;
    hi = nhi;
  }
}

// One warp: the kr-th largest of m keys in shared memory.
__device__ __forceinline__ Threshold warp_select(const int* keys, uint32_t m, uint32_t kr,
                                                 uint32_t* whist, int lane) {
  if (m <= 64) return warp_small_select(keys, m, kr, lane);
  return warp_list_select(keys, m, kr, whist, lane);
}

}  // namespace mpc
