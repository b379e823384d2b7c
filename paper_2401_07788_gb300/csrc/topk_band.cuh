// topk_band.cuh -- exact per-row TopK (§2.3), fused with error feedback (§2.4,
// Seide et al.) or the EF21 / AQ-SGD buffer update (§2.4, §2.5), for rows of
// 1025..8192 entries.  One CTA per row.  The work per entry is kept small: at
// HBM speed an SM has about 20 instruction slots per fp32 entry, so the
// selection classifies every entry once and spends more only on the few
// entries near the threshold.
//
// The row is staged in shared memory by bulk copies, one 1024-entry chunk per
// warp.  Thread t owns the 32 consecutive entries [32t, 32t + 32) and describes
// them by 32-bit words (bit j <-> entry 32t + j):
//  1. thresholds from a sample: 256 entries of the row (64 float4 groups spread
//     over it, read from global memory while the chunks land) are binned by
//     their magnitude keys (256 bins of 1/32 octave below the largest finite
//     sample magnitude); the band [t_lo, t_hi) reaches 3 standard deviations of
//     the sample count on either side of the k-th, so that it holds the row's
//     k-th largest magnitude unless the sample is unusually off;
//  2. one classification pass: per entry |x| >= t_hi ("sure") and |x| >= t_lo,
//     as two words per thread; block sums give the sure and the band counts;
//  3. if the band holds the k-th entry (sure < k <= sure + band), each thread
//     walks the set bits of its band word, listing the band's columns in index
//     order and counting them in a 256-bin histogram of their keys; the bin
//     holding the k-th is then resolved by ranking its entries against each
//     other (integer rounds when it is crowded);
//  4. the kept band entries join the sure ones in the kept words; a block scan
//     of the per-thread counts gives each thread its payload positions, each
//     thread walks the set bits of its kept word and stages the columns, and
//     the payload leaves with coalesced stores (values read back from the row).
// When the band misses (degenerate data: many equal magnitudes, no finite
// non-zero magnitude in the sample, a far outlier), an exact selection by
// integer rounds over the whole staged row replaces steps 1-3.
//
// Error feedback writes err' = s over the whole row with coalesced stores while
// forming s = x + err, then +0 at the kept entries; EF21 / AQ-SGD add d to the
// state at the kept entries only (the state is read again there, from L2).
#pragma once

#include "common.cuh"
#include "kernels.h"
#include "launch_util.h"
#include "select.cuh"

namespace mpc {
namespace band {

constexpr int kSample = 256;   // sample entries (64 threads x one float4)
constexpr int kCandCap = 256;  // candidates of the chosen bin ranked against each other
constexpr float kZ = 3.0f;     // band half-width, in standard deviations of the sample count
constexpr int kMaxNT = 256;    // threads per CTA (rows of up to 32 x 256 entries)
constexpr int kOctaveShift = 18;  // sample bins: 2^18 keys, 1/32 of an octave
constexpr uint32_t kNoSure = 0x7f800001u;  // a t_hi no magnitude reaches (NaN bits)

template <int NT>
struct Shared {
  static constexpr int NW = NT / 32;
  uint32_t keptw[NT];  // per thread: kept entries of its 32
  union {
    int skey[kSample];  // sample keys (-1: no entry)
    int cand[kCandCap];  // keys of the chosen bin's entries
  } u;
  uint32_t hist[kRoundBins];
  uint32_t r[2][3][NW];  // block sums, two alternating sets
  uint32_t t_lo, t_hi;  // the band of keys [t_lo, t_hi); t_hi = kNoSure: nothing is sure
  int fsh;              // band histogram: bin = min((key - t_lo) >> fsh, 255)
  int T;
  uint32_t need;
  uint32_t ccount;
  int fallback;
  int resolve;  // how the threshold is found: 0 resolved by warp 0, 1 rank on the block, 2 rounds
  int pick_bin;
  uint32_t pick_above, pick_count;
  uint64_t bars[kMaxNT / 32];  // one per 1024-entry chunk
};

// Dynamic shared memory: the row (fp32), then 16-bit columns: the band list,
// and later, in the same place, the staged payload columns (k <= half a row).
__host__ __device__ constexpr int row_cap(int NT) { return 32 * NT; }
__host__ __device__ constexpr int list_cap(int NT) { return row_cap(NT) * 3 / 8; }
__host__ __device__ constexpr int stage_cap(int NT) { return row_cap(NT) / 2; }
__host__ __device__ constexpr int smem_bytes(int NT) { return row_cap(NT) * 4 + stage_cap(NT) * 2; }

template <int MODE>
__device__ __forceinline__ float ranked(float x, float a) {
  if (MODE == kEF) return fadd(x, a);
  if (MODE == kDelta) return fsub(x, a);
  return x;
}

__device__ __forceinline__ uint32_t ukey(float v) { return __float_as_uint(v) & 0x7fffffffu; }

// Two bins of a 256-bin histogram (bins ranked from high to low) from one scan:
// the bins holding the r1-th and the r2-th elements (r = 0 or r past the total:
// bin -1).
__device__ __forceinline__ void warp_pick_two(const uint32_t* hist, uint32_t r1, uint32_t r2,
                                              int lane, int* b1, int* b2) {
  uint32_t c[8];
  uint32_t tsum = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    c[j] = hist[kRoundBins - 1 - (lane * 8 + j)];
    tsum += c[j];
  }
  const uint32_t incl = warp_inclusive_scan(tsum, lane);
  const uint32_t excl = incl - tsum;
  int out[2] = {-1, -1};
  const uint32_t rs[2] = {r1, r2};
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const uint32_t r = rs[q];
    const bool mine = r > 0 && excl < r && r <= incl;
    const unsigned who = __ballot_sync(kFull, mine);
    int b = -1;
    if (mine) {
      uint32_t run = excl;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (b < 0 && run + c[j] >= r) b = kRoundBins - 1 - (lane * 8 + j);
        run += c[j];
      }
    }
    out[q] = who ? __shfl_sync(kFull, b, __ffs(who) - 1) : -1;
  }
  *b1 = out[0];
  *b2 = out[1];
}

// Block sums of a and b, and the exclusive prefix and sum of c, through the
// scratch set `set` (alternate the set between consecutive calls: the next
// call's writes then never meet this call's reads, so one barrier suffices).
template <int NT, class SH>
__device__ __forceinline__ void block_sums(uint32_t a, uint32_t b, uint32_t c, SH& sh,
                                           int set, int lane, int warp, uint32_t* sa,
                                           uint32_t* sb, uint32_t* pc, uint32_t* sc) {
  constexpr int NW = NT / 32;
  const uint32_t ci = warp_inclusive_scan(c, lane);
  const uint32_t as = __reduce_add_sync(kFull, a);
  const uint32_t bs = __reduce_add_sync(kFull, b);
  if (lane == 31) sh.r[set][0][warp] = ci;
  if (lane == 0) {
    sh.r[set][1][warp] = as;
    sh.r[set][2][warp] = bs;
  }
  __syncthreads();
  uint32_t wb = 0, ta = 0, tb = 0, tc = 0;
#pragma unroll
  for (int w = 0; w < NW; ++w) {
    const uint32_t cw = sh.r[set][0][w];
    wb += (w < warp) ? cw : 0u;
    tc += cw;
    ta += sh.r[set][1][w];
    tb += sh.r[set][2][w];
  }
  *sa = ta;
  *sb = tb;
  *pc = wb + ci - c;
  *sc = tc;
}

// Exact threshold by integer rounds over `count` keys key_at(i) within [lo, hi]
// (keys outside the range, and -1, are passed over): the kr-th largest of them.
// Each round a 256-bin histogram of the keys still in the range, the bin
// holding the kr-th, until one key remains or a bin is taken whole.  Every
// thread of the block calls it.
template <int NT, class SH, class KeyAt>
__device__ Threshold select_rounds(KeyAt key_at, int count, int lo, int hi, uint32_t kr, SH& sh,
                                   int tid, int lane, int warp) {
  for (;;) {
    if (lo >= hi) return Threshold{lo, kr};
    const int sft = round_shift(lo, hi);
    __syncthreads();
    for (int i = tid; i < kRoundBins; i += NT) sh.hist[i] = 0;
    __syncthreads();
    for (int i = tid; i < count; i += NT) {
      const int key = key_at(i);
      if (key >= lo && key <= hi) atomicAdd(&sh.hist[static_cast<uint32_t>(key - lo) >> sft], 1u);
    }
    __syncthreads();
    if (warp == 0) {
      const BinPick p = warp_pick_bin(sh.hist, kr, lane);
      if (lane == 0) {
        sh.pick_bin = p.bin;
        sh.pick_above = p.above;
        sh.pick_count = p.count;
      }
    }
    __syncthreads();
    const int bin = sh.pick_bin;
    const uint32_t above = sh.pick_above, cnt = sh.pick_count;
    kr -= above;
    const int nlo = lo + (bin << sft);
    const int nhi = static_cast<int>(
        min(static_cast<uint32_t>(hi), static_cast<uint32_t>(nlo) + ((1u << sft) - 1u)));
    if (cnt == kr) return Threshold{nlo - 1, 0u};
    lo = nlo;
    hi = nhi;
  }
}

// The kr-th largest (1 <= kr <= cnt) of the cnt keys cand[] as a threshold:
// each key ranked against all others by P threads, partial counts joined by
// shuffles.  The thread that finds it writes *T (keep keys above it) and *need
// (how many keys equal to T are kept as well, in index order; 0 when the
// threshold sits just below a key taken with all its copies).
template <int NT>
__device__ void rank_block(const int* cand, uint32_t cnt, uint32_t kr, int* T, uint32_t* need,
                           int tid) {
  uint32_t P = 1;
  while (P < 32 && cnt * P * 2 <= static_cast<uint32_t>(NT)) P *= 2;
  const uint32_t part = static_cast<uint32_t>(tid) & (P - 1);
  for (uint32_t c0 = 0; c0 < cnt; c0 += NT / P) {
    const uint32_t ci = c0 + static_cast<uint32_t>(tid) / P;
    uint32_t gt = 0, ge = 0;
    int ki = 0;
    if (ci < cnt) {
      ki = cand[ci];
      for (uint32_t j = part; j < cnt; j += P) {
        const int aj = cand[j];
        gt += aj > ki;
        ge += aj >= ki;
      }
    }
    for (uint32_t o = P >> 1; o > 0; o >>= 1) {
      gt += __shfl_xor_sync(kFull, gt, o);
      ge += __shfl_xor_sync(kFull, ge, o);
    }
    if (ci < cnt && part == 0 && gt < kr && kr <= ge) {
      const uint32_t nd = kr - gt;
      *T = (nd == ge - gt) ? ki - 1 : ki;
      *need = (nd == ge - gt) ? 0u : nd;
    }
  }
}

template <int MODE, int NT>
__global__ void __launch_bounds__(NT, NT == 64 ? 16 : (NT == 128 ? 10 : 5))
    topk_band_kernel(const TopkRowArgs a) {
  pdl_begin();
  constexpr int NW = NT / 32;
  constexpr int CAP = row_cap(NT);
  constexpr int LCAP = list_cap(NT);
  constexpr int SCAP = stage_cap(NT);
  static_assert(NT % 32 == 0 && NT <= kMaxNT, "threads");
  __shared__ Shared<NT> sh;
  extern __shared__ __align__(16) float4 dyn4[];
  float* srow = reinterpret_cast<float*>(dyn4);
  uint16_t* cols = reinterpret_cast<uint16_t*>(srow + CAP);  // band list, then staging

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t row = blockIdx.x;
  const int n = static_cast<int>(a.L);
  const int64_t k = a.k;

  float* arow = nullptr;
  if (MODE != kPlain) {
    int64_t srow_idx = row;
    if (MODE == kDelta && a.ids != nullptr) {
      const int64_t sid = a.ids[row / a.rps];
      if (sid < 0 || sid >= a.num_samples) {
        if (tid == 0) set_status(a.status, STATUS_BAD_SAMPLE);
        return;
      }
      srow_idx = sid * a.rps + row % a.rps;
    }
    arow = a.aux + srow_idx * a.L;
  }
  const float* xrow = a.x + row * a.L;

  // ---- loads: one bulk copy per 1024-entry chunk (chunk w <-> warp w) -------
  if (a.aligned && warp == 0 && lane < NW && 1024 * lane < n) {
    const int c0 = 1024 * lane;
    const uint32_t bytes = static_cast<uint32_t>(min(1024, n - c0)) * 4u;
    if (MODE != kPlain) bulk_prefetch_l2(arow + c0, bytes);
    mbar_init(&sh.bars[lane], 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(&sh.bars[lane], bytes);
    bulk_g2s(srow + c0, xrow + c0, bytes, &sh.bars[lane]);
  }
  // the sample, from global memory: entries [p, p + 4) for 64 points p
  if (tid < kSample / 4) {
    const int sp = (n / (kSample / 4)) * tid / 4 * 4;
    float sx[4] = {0.f, 0.f, 0.f, 0.f}, sa[4] = {0.f, 0.f, 0.f, 0.f};
    if (a.aligned && sp + 4 <= n) {
      const float4 v = *reinterpret_cast<const float4*>(xrow + sp);
      sx[0] = v.x, sx[1] = v.y, sx[2] = v.z, sx[3] = v.w;
      if (MODE != kPlain) {
        const float4 w = *reinterpret_cast<const float4*>(arow + sp);
        sa[0] = w.x, sa[1] = w.y, sa[2] = w.z, sa[3] = w.w;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (sp + i < n) {
          sx[i] = xrow[sp + i];
          if (MODE != kPlain) sa[i] = arow[sp + i];
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      sh.u.skey[4 * tid + i] = (sp + i < n) ? static_cast<int>(ukey(ranked<MODE>(sx[i], sa[i]))) : -1;
  }
  for (int i = tid; i < kRoundBins; i += NT) sh.hist[i] = 0;
  if (!a.aligned) {
    for (int e = tid; e < n; e += NT) {
      const float s = ranked<MODE>(xrow[e], MODE != kPlain ? arow[e] : 0.0f);
      srow[e] = s;
      if (MODE == kEF) arow[e] = s;  // err' = s; +0 at the kept entries later
    }
  }
  __syncthreads();

  // ---- thresholds from the sample (warp 0) ------------------------------------
  if (warp == 0) {
    int kk[8];
    int smax = -1;
    uint32_t nvalid = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      kk[j] = sh.u.skey[lane * 8 + j];
      nvalid += kk[j] >= 0;
      smax = max(smax, kk[j] >= 0 ? finite_key(kk[j]) : -1);
    }
    smax = __reduce_max_sync(kFull, smax);
    nvalid = __reduce_add_sync(kFull, nvalid);
    int fb = (smax > 0 && k < n) ? 0 : 1;
    uint32_t t_lo = 0, t_hi = kNoSure;
    int fsh = 0;
    if (!fb) {
      // 256 bins of 2^18 keys ending at the largest finite sample key: bin 0
      // takes everything below base, bin 255 everything above smax
      const int base = max(0, smax - (255 << kOctaveShift));
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (kk[j] >= 0)
          atomicAdd(&sh.hist[min(max(kk[j] - base, 0) >> kOctaveShift, kRoundBins - 1)], 1u);
      __syncwarp();
      // the expected sample count above the k-th largest, and its spread (only
      // the width of the band depends on these, so approximations serve)
      const float mu = __fdividef(static_cast<float>(k) * static_cast<float>(nvalid),
                                  static_cast<float>(n));
      const float sd = mu * rsqrtf(mu);
      const int r_hi = static_cast<int>(floorf(mu - kZ * sd));
      const int r_lo = static_cast<int>(ceilf(mu + kZ * sd)) + 1;
      int b_hi, b_lo;
      warp_pick_two(sh.hist, r_hi >= 1 ? static_cast<uint32_t>(r_hi) : 0u,
                    r_lo <= static_cast<int>(nvalid) ? static_cast<uint32_t>(r_lo) : 0u, lane,
                    &b_hi, &b_lo);
      if (b_hi >= 0 && b_hi < kRoundBins - 1)
        t_hi = static_cast<uint32_t>(base + ((b_hi + 1) << kOctaveShift));
      if (b_lo > 0) t_lo = static_cast<uint32_t>(base + (b_lo << kOctaveShift));
      if (t_lo > t_hi) t_lo = t_hi;
      // the band histogram spans [t_lo, t_hi), or, with nothing sure, up to one
      // octave above the sample's largest magnitude (larger keys share the top bin)
      const uint32_t fhi = t_hi != kNoSure ? t_hi - 1u
                                           : min(static_cast<uint32_t>(smax) + (1u << 23), 0x7f7fffffu);
      fsh = round_shift(static_cast<int>(t_lo), static_cast<int>(max(fhi, t_lo)));
      __syncwarp();
      for (int i = lane; i < kRoundBins; i += 32) sh.hist[i] = 0;  // for the band histogram
    }
    if (lane == 0) {
      sh.t_lo = t_lo;
      sh.t_hi = t_hi;
      sh.fsh = fsh;
      sh.fallback = fb;
    }
  }

  // ---- each warp waits for its chunk; error feedback / EF21 form s or d -------
  bool failed = false;
  const int cbase = 1024 * warp;
  if (a.aligned && cbase < n) {
    if (!mbar_wait_bounded(&sh.bars[warp], 0, a.spin_limit, a.status)) {
      mbar_wait_bounded(&sh.bars[warp], 0, kDrainPolls, nullptr);
      failed = true;
    }
    if (MODE != kPlain) {
      // striped over the chunk: consecutive lanes consecutive float4 groups
      const int nq = (min(1024, n - cbase)) / 4;
      float4* c4 = reinterpret_cast<float4*>(srow + cbase);
      const float4* a4 = reinterpret_cast<const float4*>(arow + cbase);
#pragma unroll 4
      for (int q = lane; q < nq; q += 32) {
        const float4 xv = c4[q];
        const float4 av = a4[q];
        const float4 sv = make_float4(ranked<MODE>(xv.x, av.x), ranked<MODE>(xv.y, av.y),
                                      ranked<MODE>(xv.z, av.z), ranked<MODE>(xv.w, av.w));
        c4[q] = sv;
        if (MODE == kEF) reinterpret_cast<float4*>(arow + cbase)[q] = sv;
      }
      __syncwarp();
    }
  }
  failed = __syncthreads_or(failed);
  if (failed) return;  // the status word reports the timeout; outputs unspecified

  // ---- classification: sure (key >= t_hi) and band (t_lo <= key < t_hi) -------
  const int e0 = 32 * tid;
  const int nv = max(0, min(32, n - e0));  // valid entries of this thread
  const uint32_t vmask = nv >= 32 ? 0xffffffffu : ((1u << nv) - 1u);
  bool fallback = sh.fallback != 0;
  uint32_t sure_w = 0, band_w = 0;
  uint32_t n_sure = 0, n_ge = 0, boff = 0, m = 0;
  if (!fallback) {
    // magnitudes compared as floats: for finite values the order of |x| is the
    // order of the keys, and kNoSure (a NaN) is reached by no |x|
    const float f_lo = __uint_as_float(sh.t_lo), f_hi = __uint_as_float(sh.t_hi);
    uint32_t hw = 0, gw = 0;
    if (nv > 0) {
      // 8 float4 groups, rotated by lane so that 8 consecutive lanes read 8
      // different bank groups
      const float4* my4 = reinterpret_cast<const float4*>(srow + e0);
      if (sh.t_hi == kNoSure) {
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const float4 v = my4[(u + lane) & 7];
          or_if_ge(gw, v.x, f_lo, 1u << (4 * u + 0));
          or_if_ge(gw, v.y, f_lo, 1u << (4 * u + 1));
          or_if_ge(gw, v.z, f_lo, 1u << (4 * u + 2));
          or_if_ge(gw, v.w, f_lo, 1u << (4 * u + 3));
        }
      } else {
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const float4 v = my4[(u + lane) & 7];
          or_if_ge(hw, v.x, f_hi, 1u << (4 * u + 0));
          or_if_ge(hw, v.y, f_hi, 1u << (4 * u + 1));
          or_if_ge(hw, v.z, f_hi, 1u << (4 * u + 2));
          or_if_ge(hw, v.w, f_hi, 1u << (4 * u + 3));
          or_if_ge(gw, v.x, f_lo, 1u << (4 * u + 0));
          or_if_ge(gw, v.y, f_lo, 1u << (4 * u + 1));
          or_if_ge(gw, v.z, f_lo, 1u << (4 * u + 2));
          or_if_ge(gw, v.w, f_lo, 1u << (4 * u + 3));
        }
      }
      const uint32_t rot = 4u * static_cast<uint32_t>(lane & 7);
      hw = __funnelshift_l(hw, hw, rot) & vmask;
      gw = __funnelshift_l(gw, gw, rot) & vmask;
    }
    sure_w = hw;
    band_w = gw & ~hw;
    block_sums<NT>(__popc(hw), __popc(gw), __popc(band_w), sh, 0, lane, warp, &n_sure, &n_ge,
                   &boff, &m);
    fallback = !(static_cast<int64_t>(n_sure) < k && k <= static_cast<int64_t>(n_ge) &&
                 m <= static_cast<uint32_t>(LCAP));
  }

  int T = -1;
  uint32_t need = 0;
  if (!fallback) {
    // ---- the band's columns in index order, and the histogram of their keys --
    const int t_lo = static_cast<int>(sh.t_lo);
    const int fsh = sh.fsh;
    {
      uint32_t w = band_w;
      uint32_t p = boff;
      while (w) {
        const int j = __ffs(w) - 1;
        w &= w - 1;
        const int e = e0 + j;
        const int key = static_cast<int>(ukey(srow[e]));
        cols[p++] = static_cast<uint16_t>(e);
        atomicAdd(&sh.hist[min(static_cast<uint32_t>(key - t_lo) >> fsh, kRoundBins - 1u)], 1u);
      }
    }
    __syncthreads();
    const uint32_t kr = static_cast<uint32_t>(k - n_sure);  // 1 <= kr <= m
    auto key_at = [&](int i) { return static_cast<int>(ukey(srow[cols[i]])); };
    // warp 0 finds the bin holding the kr-th band entry and, when the bin is
    // taken whole or holds at most 64 entries, the threshold itself
    constexpr uint32_t kWarpRank = 64;
    if (warp == 0) {
      const BinPick p = warp_pick_bin(sh.hist, kr, lane);
      const uint32_t kr2 = kr - p.above;
      const int bl = t_lo + (p.bin << fsh);
      // the top bin also takes every larger key
      const int bh = p.bin == kRoundBins - 1
                         ? 0x7fffffff
                         : static_cast<int>(min(static_cast<uint32_t>(bl) + ((1u << fsh) - 1u),
                                                0x7fffffffu));
      int Tw = bl - 1;  // the bin kept whole
      uint32_t nw = 0;
      int state = 0;    // 0: resolved; 1: rank on the block; 2: integer rounds
      if (p.count != kr2) {
        if (p.count <= kWarpRank && m <= 8 * 32) {
          // the bin's keys, compacted by ballots, then each ranked against all
          const unsigned lt = lanemask_lt();
          uint32_t c = 0;
          for (uint32_t i0 = 0; i0 < m; i0 += 32) {
            const uint32_t i = i0 + lane;
            const int key = i < m ? key_at(static_cast<int>(i)) : -1;
            const bool in = key >= bl && key <= bh;
            const unsigned b = __ballot_sync(kFull, in);
            if (in) sh.u.cand[c + __popc(b & lt)] = key;
            c += __popc(b);
          }
          __syncwarp();
          bool found = false;
          for (uint32_t ci = lane; ci < p.count; ci += 32) {
            const int ki = sh.u.cand[ci];
            uint32_t gt = 0, ge = 0;
            for (uint32_t j = 0; j < p.count; ++j) {
              const int aj = sh.u.cand[j];
              gt += aj > ki;
              ge += aj >= ki;
            }
            if (gt < kr2 && kr2 <= ge) {
              const uint32_t nd = kr2 - gt;
              Tw = (nd == ge - gt) ? ki - 1 : ki;
              nw = (nd == ge - gt) ? 0u : nd;
              found = true;
            }
          }
          const unsigned who = __ballot_sync(kFull, found);
          Tw = __shfl_sync(kFull, Tw, who ? __ffs(who) - 1 : 0);
          nw = __shfl_sync(kFull, nw, who ? __ffs(who) - 1 : 0);
        } else {
          state = p.count > static_cast<uint32_t>(kCandCap) ? 2 : 1;
        }
      }
      if (lane == 0) {
        sh.T = Tw;
        sh.need = nw;
        sh.resolve = state;
        sh.pick_bin = p.bin;
        sh.pick_above = p.above;
        sh.pick_count = p.count;
        sh.ccount = 0;
      }
    }
    __syncthreads();
    T = sh.T;
    need = sh.need;
    if (sh.resolve != 0) {
      const uint32_t kr2 = kr - sh.pick_above;
      const uint32_t cnt = sh.pick_count;
      const int bl = t_lo + (sh.pick_bin << fsh);
      const int bh = sh.pick_bin == kRoundBins - 1
                         ? 0x7fffffff
                         : static_cast<int>(min(static_cast<uint32_t>(bl) + ((1u << fsh) - 1u),
                                                0x7fffffffu));
      if (sh.resolve == 2) {
        const Threshold th = select_rounds<NT>(
            [&](int i) {
              const int key = key_at(i);
              return (key >= bl && key <= bh) ? key : -1;
            },
            static_cast<int>(m), bl, bh, kr2, sh, tid, lane, warp);
        T = th.T;
        need = th.need;
      } else {
        // the bin's entries ranked against each other on the block
        for (uint32_t i = tid; i < m; i += NT) {
          const int key = key_at(static_cast<int>(i));
          if (key >= bl && key <= bh) sh.u.cand[atomicAdd(&sh.ccount, 1u)] = key;
        }
        __syncthreads();
        rank_block<NT>(sh.u.cand, cnt, kr2, &sh.T, &sh.need, tid);
        __syncthreads();
        T = sh.T;
        need = sh.need;
      }
    }

    // ---- kept words: the sure entries, and the band entries above T or tied ---
    if (need == 0 && m <= 2 * NT) {
      // a small band: each thread tests its own band entries, so no other
      // thread's words are touched
      uint32_t w = band_w, kb = 0;
      while (w) {
        const int j = __ffs(w) - 1;
        w &= w - 1;
        if (static_cast<int>(ukey(srow[e0 + j])) > T) kb |= 1u << j;
      }
      sh.keptw[tid] = sure_w | kb;
    } else if (need == 0) {
      // a larger one: the band list split evenly over the block
      sh.keptw[tid] = sure_w;
      __syncthreads();
      for (uint32_t i = tid; i < m; i += NT) {
        const uint32_t e = cols[i];
        if (static_cast<int>(ukey(srow[e])) > T) atomicOr(&sh.keptw[e >> 5], 1u << (e & 31));
      }
    } else {
      sh.keptw[tid] = sure_w;
      __syncthreads();
      if (warp == 0) {
        // ties are taken in index order: the list is in index order
        const unsigned lt = lanemask_lt();
        uint32_t seen = 0;
        for (uint32_t i0 = 0; i0 < m; i0 += 32) {
          const uint32_t i = i0 + lane;
          const uint32_t e = i < m ? cols[i] : 0u;
          const int key = i < m ? static_cast<int>(ukey(srow[e])) : -1;
          const bool eq = key == T;
          const unsigned be = __ballot_sync(kFull, eq);
          const uint32_t rank = seen + __popc(be & lt);
          seen += __popc(be);
          if (key > T || (eq && rank < need)) atomicOr(&sh.keptw[e >> 5], 1u << (e & 31));
        }
      }
    }
    __syncthreads();
  } else {
    // ---- exact selection over the whole row by integer rounds ---------------
    int lo = 0x7fffffff, hi = -1;
    for (int e = tid; e < n; e += NT) {
      const int key = static_cast<int>(ukey(srow[e]));
      lo = min(lo, key);
      hi = max(hi, key);
    }
    lo = __reduce_min_sync(kFull, lo);
    hi = __reduce_max_sync(kFull, hi);
    if (lane == 0) {
      sh.r[1][0][warp] = static_cast<uint32_t>(lo);
      sh.r[1][1][warp] = static_cast<uint32_t>(hi);
    }
    __syncthreads();
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      lo = min(lo, static_cast<int>(sh.r[1][0][w]));
      hi = max(hi, static_cast<int>(sh.r[1][1][w]));
    }
    Threshold th{-1, 0u};
    if (k < n)
      th = select_rounds<NT>([&](int e) { return static_cast<int>(ukey(srow[e])); }, n, lo, hi,
                             static_cast<uint32_t>(k), sh, tid, lane, warp);
    T = th.T;
    need = th.need;
    // kept words: entries above T, and the first `need` entries equal to T
    uint32_t gtw = 0, eqw = 0;
    for (int i = 0; i < 32; ++i) {
      const int j = (i + lane) & 31;  // lanes on different banks
      const int key = j < nv ? static_cast<int>(ukey(srow[e0 + j])) : -1;
      gtw |= static_cast<uint32_t>(key > T) << j;
      eqw |= static_cast<uint32_t>(key == T) << j;
    }
    uint32_t d0, d1, eq_before, d2;
    block_sums<NT>(0u, 0u, __popc(eqw), sh, 0, lane, warp, &d0, &d1, &eq_before, &d2);
    uint32_t take = need > eq_before ? min(need - eq_before, 32u) : 0u;
    while (eqw && take) {
      gtw |= eqw & (~eqw + 1u);  // the lowest remaining tie
      eqw &= eqw - 1;
      --take;
    }
    sh.keptw[tid] = gtw;
    __syncthreads();
  }

  // ---- the payload: kept entries by ascending column ----------------------------
  uint32_t kw = sh.keptw[tid];
  uint32_t base, d0, d1, total;
  block_sums<NT>(0u, 0u, __popc(kw), sh, 1, lane, warp, &d0, &d1, &base, &total);
  pdl_end();
  float* vrow = a.vals + row * k;
  int32_t* irow = a.idx + row * k;
  if (k <= SCAP) {
    // columns staged at their payload positions (the band list is dead), then
    // values and columns written out with coalesced stores, and the buffers
    // updated at the kept columns (independent accesses, many in flight)
    uint32_t p = base;
    while (kw) {
      const int j = __ffs(kw) - 1;
      kw &= kw - 1;
      if (p < static_cast<uint32_t>(k)) cols[p] = static_cast<uint16_t>(e0 + j);
      ++p;
    }
    __syncthreads();
    const int kk = static_cast<int>(k);
    // payload positions [h, kk) in groups of 4 with 16-byte stores, where the
    // payload rows allow it; the first h singly
    const uintptr_t av = reinterpret_cast<uintptr_t>(vrow), ai = reinterpret_cast<uintptr_t>(irow);
    const int h = ((av & 15) == (ai & 15) && (av & 3) == 0)
                      ? min(kk, static_cast<int>(((16 - (av & 15)) & 15) >> 2))
                      : kk;
    for (int i = tid; i < h; i += NT) {
      const int e = cols[i];
      const float v = srow[e];
      vrow[i] = v;
      irow[i] = e;
      if (MODE == kEF) arow[e] = 0.0f;                 // err' = s - C(s): +0 where sent
      if (MODE == kDelta) arow[e] = fadd(arow[e], v);  // state + d, where sent
    }
    for (int i = h + 4 * tid; i < kk; i += 4 * NT) {
      int e[4];
      float v[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        e[q] = i + q < kk ? cols[i + q] : 0;
        v[q] = srow[e[q]];
      }
      if (i + 4 <= kk) {
        *reinterpret_cast<float4*>(vrow + i) = make_float4(v[0], v[1], v[2], v[3]);
        *reinterpret_cast<int4*>(irow + i) = make_int4(e[0], e[1], e[2], e[3]);
      } else {
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (i + q < kk) {
            vrow[i + q] = v[q];
            irow[i + q] = e[q];
          }
      }
      if (MODE == kDelta) {
        // the kept columns are distinct: all four state loads go out first
        float g[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) g[q] = i + q < kk ? arow[e[q]] : 0.0f;
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (i + q < kk) arow[e[q]] = fadd(g[q], v[q]);
      }
      if (MODE == kEF) {
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (i + q < kk) arow[e[q]] = 0.0f;
      }
    }
  } else {
    uint32_t p = base;
    while (kw) {
      const int j = __ffs(kw) - 1;
      kw &= kw - 1;
      const int e = e0 + j;
      const float v = srow[e];
      if (p < static_cast<uint32_t>(k)) {
        vrow[p] = v;
        irow[p] = e;
      }
      if (MODE == kEF) arow[e] = 0.0f;
      if (MODE == kDelta) arow[e] = fadd(arow[e], v);
      ++p;
    }
  }
}

template <int MODE, int NT>
cudaError_t run(const TopkRowArgs& a, cudaStream_t s) {
  auto kernel = topk_band_kernel<MODE, NT>;
  const int smem = smem_bytes(NT);
  cudaError_t err = ensure_dynamic_smem(kernel, smem);
  if (err != cudaSuccess) return err;
  if (a.rows > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_kernel(kernel, dim3(static_cast<unsigned>(a.rows)), dim3(NT), smem, s, 0u, a);
}

// Rows of 1025..8192 entries (one CTA of L/32 threads rounded up to 64, 128 or 256).
inline bool fits(int64_t L) { return L > 1024 && L <= 32 * kMaxNT; }

template <int MODE>
cudaError_t run_mode(const TopkRowArgs& a, cudaStream_t s) {
  if (a.L <= 2048) return run<MODE, 64>(a, s);
  if (a.L <= 4096) return run<MODE, 128>(a, s);
  return run<MODE, 256>(a, s);
}

}  // namespace band
}  // namespace mpc
