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

// The key if it is that of a finite number, else -1: the bin scale comes from
// the largest finite magnitude, and infinities (TopK marks entries with them)
// or NaNs then fall in the top bin.
__device__ __forceinline__ int finite_key(int key) { return key < 0x7f800000 ? key : -1; }

// Bin of a key (>= 0) in the |x|-linear histogram.  Monotone in the key:
// |x| * scale rounds monotonically and truncation is monotone.
__device__ __forceinline__ int bucket_of(int key, float scale, int nb) {
  int b = __float2int_rz(fmul(__int_as_float(key), scale));
  return min(b, nb - 1);
}

// The smallest key of bin b (b >= 1) of an |x|-linear histogram (bucket_of, or
// any bin rule that floors |x| * scale): the least c >= 0 with
// |x(c)| * scale >= b.  `inv` = 1 / scale, rounded; the start point it gives
// is a few units off at most and is corrected step by step, with bisection as
// the bound-free fallback.
__device__ __forceinline__ int bin_first_key(int b, float scale, float inv) {
  const float fb = static_cast<float>(b);
  auto reaches = [&](int c) { return fmul(__int_as_float(c), scale) >= fb; };
  int c = min(__float_as_int(fmul(fb, inv)), 0x7f800000);
  for (int i = 0; i < 8 && c > 0 && reaches(c - 1); ++i) --c;
  for (int i = 0; i < 8 && !reaches(c); ++i) ++c;
  if (!reaches(c) || (c > 0 && reaches(c - 1))) {
    int lo = 0, hi = 0x7f800000;  // reaches(hi), !reaches(lo)
    while (hi - lo > 1) {
      const int mid = lo + (hi - lo) / 2;
      if (reaches(mid)) hi = mid;
      else lo = mid;
    }
    c = hi;
  }
  return c;
}

// w |= bit when |v| >= t: one compare and one predicated OR, no branch.
__device__ __forceinline__ void or_if_ge(uint32_t& w, float v, float t, uint32_t bit) {
  asm("{\n .reg .pred p;\n setp.ge.f32 p, %1, %2;\n @p or.b32 %0, %0, %3;\n}"
      : "+r"(w)
      : "f"(fabsf(v)), "f"(t), "r"(bit));
}

// w |= bit when |v| > t, and when |v| == t: as or_if_ge.
__device__ __forceinline__ void or_if_gt(uint32_t& w, float v, float t, uint32_t bit) {
  asm("{\n .reg .pred p;\n setp.gt.f32 p, %1, %2;\n @p or.b32 %0, %0, %3;\n}"
      : "+r"(w)
      : "f"(fabsf(v)), "f"(t), "r"(bit));
}
__device__ __forceinline__ void or_if_eq(uint32_t& w, float v, float t, uint32_t bit) {
  asm("{\n .reg .pred p;\n setp.eq.f32 p, %1, %2;\n @p or.b32 %0, %0, %3;\n}"
      : "+r"(w)
      : "f"(fabsf(v)), "f"(t), "r"(bit));
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

// Rank test of one candidate key ki against the m keys: it is T when fewer than
// kr keys are larger and at least kr are at least as large.  Then *t is the
// threshold: {ki, kr - #larger}, or {ki - 1, 0} when every key equal to ki is
// kept anyway (no tie has to be ranked by index).
__device__ __forceinline__ bool rank_is_threshold(const int* keys, uint32_t m, uint32_t kr, int ki,
                                                  Threshold* t) {
  uint32_t gt = 0, ge = 0;
  uint32_t j = 0;
  for (; j + 4 <= m; j += 4) {
    const int a0 = keys[j], a1 = keys[j + 1], a2 = keys[j + 2], a3 = keys[j + 3];
    gt += (a0 > ki) + (a1 > ki) + (a2 > ki) + (a3 > ki);
    ge += (a0 >= ki) + (a1 >= ki) + (a2 >= ki) + (a3 >= ki);
  }
  for (; j < m; ++j) {
    const int a0 = keys[j];
    gt += a0 > ki;
    ge += a0 >= ki;
  }
  if (!(gt < kr && kr <= ge)) return false;
  const uint32_t need = kr - gt;
  *t = (need == ge - gt) ? Threshold{ki - 1, 0u} : Threshold{ki, need};
  return true;
}

// One warp, m <= 64 keys in shared memory: each lane ranks its candidates
// against all m keys (a loop of length m); the lane holding T reports it.
__device__ __forceinline__ Threshold warp_rank_select(const int* keys, uint32_t m, uint32_t kr,
                                                      int lane) {
  Threshold t = {-1, 0u};
  bool found = false;
  for (uint32_t i = lane; i < m; i += 32) {
    Threshold ti;
    if (rank_is_threshold(keys, m, kr, keys[i], &ti)) {
      t = ti;
      found = true;
    }
  }
  const unsigned who = __ballot_sync(kFull, found);
  const int src = who ? __ffs(who) - 1 : 0;
  t.T = __shfl_sync(kFull, t.T, src);
  t.need = __shfl_sync(kFull, t.need, src);
  return t;
}

// One warp: the kr-th largest of m keys in shared memory.
__device__ __forceinline__ Threshold warp_select(const int* keys, uint32_t m, uint32_t kr,
                                                 uint32_t* whist, int lane) {
  if (m <= 64) return warp_rank_select(keys, m, kr, lane);
  return warp_list_select(keys, m, kr, whist, lane);
}

}  // namespace mpc
