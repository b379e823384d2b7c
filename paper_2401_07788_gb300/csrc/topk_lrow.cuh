// topk_lrow.cuh -- exact per-row TopK (§2.3), fused with error feedback (§2.4,
// Seide et al.) or the EF21 / AQ-SGD buffer update (§2.4, §2.5), for rows of
// 8193..65536 entries that start 16-byte aligned.  One CTA of 512 threads per
// row.
//
//  0. the row's chunks (8192 entries, 32 KiB) are prefetched into L2 by bulk
//     prefetches, two chunks ahead of the first pass;
//  1. thresholds from a sample: 2048 entries of the row (one float4 group per
//     thread, spread evenly) binned by magnitude key (256 bins of 1/32 octave
//     below the largest finite sample key); the band [t_lo, t_hi) reaches 3.5
//     binomial standard deviations of the sample count on either side of the
//     k-th.  When the sample puts few enough entries at or above t_lo, the row
//     is done in one pass ("list mode"), else in two;
//  2. first pass: every entry compared with t_hi ("sure") and t_lo; the sure
//     entries counted per 512-entry sub-chunk; the band's entries (list mode:
//     every entry >= t_lo) listed in shared memory with their columns, each
//     sub-chunk's as one segment in index order, and the band's keys counted in
//     a 256-bin histogram on the way;
//  3. if the band holds the k-th entry, the histogram bin holding it is found
//     and its entries ranked against each other (integer rounds when it is
//     crowded): the threshold T, and how many keys equal to T are kept; the
//     list then gives each sub-chunk its listed entries above T and equal to
//     T.  Otherwise (degenerate data) an exact selection by integer rounds over
//     the whole row, read again from L2, and a counting pass;
//  4. the payload offset of every sub-chunk and its quota of ties (the first
//     `need` keys equal to T over the row, in index order) by one warp scan;
//  5. list mode: each warp writes the kept entries of its sub-chunks' segments
//     (coalesced), error feedback zeroes err' and EF21 / AQ-SGD update the state
//     at the kept columns.  Two-pass mode: a second pass over the row (from
//     L2), each warp on its own sub-chunks with no block barrier: the kept
//     entries (|s| > T, and the sub-chunk's quota of ties) of two 128-entry
//     groups at a time staged in shared memory in index order by predicated
//     stores and written out with coalesced stores (a sub-chunk with nothing
//     kept is not read again); error
//     feedback rewrites err' (+0 where kept), EF21 / AQ-SGD the state (state + d
//     where kept), a 16-byte group at a time.
//
// Layout: chunk c, warp w and group u (0..3) cover entries
// c * 8192 + w * 512 + u * 128 + [0, 128) (sub-chunk 16c + w), lane l the four
// entries from 4l on.  The first pass writes err' = s under error feedback.
// Loads and stores carry L2 priorities: what is read or written again later in
// the kernel is kept, what the kernel is done with is dropped first.
#pragma once

#include "topk_band.cuh"

namespace mpc {
namespace lrow {

constexpr int NT = 512;
constexpr int NW = NT / 32;
constexpr int kU = 4;                  // float4 groups per lane per sub-chunk
constexpr int kSub = 32 * kU * 4;      // entries per warp sub-chunk (512)
constexpr int kChunk = NW * kSub;      // entries per chunk (8192)
constexpr int kSample = 4 * NT;        // sample entries (2048)
constexpr int kListCap = 12288;        // entries listed (value bits and column)
constexpr int kCandCap = 512;          // keys of the chosen bin ranked on the block
constexpr int kMinL = 8193;
constexpr int kMaxL = 65536;
constexpr int kAhead = 2;              // chunks prefetched ahead of the first pass
constexpr int kMaxSub = kMaxL / kSub;  // sub-chunks of a row (128)
constexpr float kZ = 3.5f;
constexpr float kListShare = 0.25f;    // list mode up to this share of the row listed

struct Shared {
  uint32_t hist[kRoundBins];
  uint32_t r[2][3][NW];   // block sums (band::select_rounds scratch, reductions)
  int cand[kCandCap];
  // per 512-entry sub-chunk: sure entries, listed entries above T and equal to
  // T, ties kept, entries kept, the payload position of the first, and the
  // sub-chunk's segment of the list
  uint32_t sc_sure[kMaxSub], sc_gt[kMaxSub], sc_eq[kMaxSub];
  uint32_t sc_tie[kMaxSub], sc_kept[kMaxSub], sc_base[kMaxSub];
  uint32_t seg_start[kMaxSub], seg_cnt[kMaxSub];
  int smax[NW];
  uint32_t t_lo, t_hi;
  int fsh;
  int lmode;              // every entry >= t_lo listed: one pass
  int T;
  uint32_t need;
  uint32_t mcount;        // entries listed
  uint32_t ccount;
  int resolve;
  int pick_bin;
  uint32_t pick_above, pick_count;
};

// dynamic shared memory: the stage (kU float4 per thread in the first pass,
// the per-warp output buffers in the second), the listed values, their columns
constexpr int kStageBytes = kU * NT * 16;
constexpr int kSmemBytes = kStageBytes + kListCap * 6;

__device__ __forceinline__ uint32_t fld(uint32_t packed, int u) { return (packed >> (8 * u)) & 0xffu; }

// Per-group counts of a 16-bit word (bits 4u..4u+3 <-> group u) packed in bytes.
__device__ __forceinline__ uint32_t pack_counts(uint32_t w) {
  uint32_t p = 0;
#pragma unroll
  for (int u = 0; u < kU; ++u) p |= static_cast<uint32_t>(__popc((w >> (4 * u)) & 0xfu)) << (8 * u);
  return p;
}

template <int MODE>
__global__ void __launch_bounds__(NT, 2) topk_lrow_kernel(const TopkRowArgs a) {
  pdl_begin();
  __shared__ Shared sh;
  extern __shared__ __align__(16) float4 dyn4[];
  float4* stage = dyn4;
  uint32_t* lval = reinterpret_cast<uint32_t*>(dyn4 + kU * NT);  // value bits
  uint16_t* lcol = reinterpret_cast<uint16_t*>(lval + kListCap);

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
  const int nch = (n + kChunk - 1) / kChunk;
  const int nsc = (n + kSub - 1) / kSub;
  const uint64_t keep = l2_evict_last(), drop = l2_evict_first();
  auto prefetch = [&](int c) {
    if (c < nch) {
      const uint32_t bytes = static_cast<uint32_t>(min(kChunk, n - c * kChunk)) * 4u;
      const float* xs = xrow + static_cast<int64_t>(c) * kChunk;
      if (MODE == kEF) {
        bulk_prefetch_l2(xs, bytes);
        bulk_prefetch_l2(arow + static_cast<int64_t>(c) * kChunk, bytes);
      } else {
        bulk_prefetch_l2(xs, bytes, keep);
        if (MODE == kDelta) bulk_prefetch_l2(arow + static_cast<int64_t>(c) * kChunk, bytes, keep);
      }
    }
  };
  if (tid == 0)
    for (int c = 0; c < kAhead; ++c) prefetch(c);
  // a float4 group as this lane sees it: s = x + err (error feedback),
  // d = x - state (EF21 / AQ-SGD), else x
  auto load = [&](int q, float4* g, uint64_t px, uint64_t pa) -> float4 {
    const float4 xv = ld_f4(xrow + q, px);
    if (MODE == kPlain) return xv;
    const float4 av = ld_f4(arow + q, pa);
    if (g) *g = av;
    return make_float4(band::ranked<MODE>(xv.x, av.x), band::ranked<MODE>(xv.y, av.y),
                       band::ranked<MODE>(xv.z, av.z), band::ranked<MODE>(xv.w, av.w));
  };

  const bool keep_all = k >= n;
  // ---- the sample -----------------------------------------------------------------
  if (tid < kRoundBins) sh.hist[tid] = 0;
  if (tid == 0) sh.mcount = 0;
  int kk[4];
  {
    const int sp = (n / 4 / NT) * tid * 4;  // n > 8192: sp + 4 <= n
    const float4 v = load(sp, nullptr, keep, keep);
    kk[0] = static_cast<int>(band::ukey(v.x));
    kk[1] = static_cast<int>(band::ukey(v.y));
    kk[2] = static_cast<int>(band::ukey(v.z));
    kk[3] = static_cast<int>(band::ukey(v.w));
    int mx = max(max(finite_key(kk[0]), finite_key(kk[1])), max(finite_key(kk[2]), finite_key(kk[3])));
    mx = __reduce_max_sync(kFull, mx);
    if (lane == 0) sh.smax[warp] = mx;
  }
  __syncthreads();
  int smax = -1;
#pragma unroll
  for (int w = 0; w < NW; ++w) smax = max(smax, sh.smax[w]);
  const int base = max(0, smax - (255 << band::kOctaveShift));
  if (smax > 0 && !keep_all) {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      atomicAdd(&sh.hist[min(max(kk[j] - base, 0) >> band::kOctaveShift, kRoundBins - 1)], 1u);
  }
  __syncthreads();
  if (warp == 0) {
    uint32_t t_lo = band::kNoSure, t_hi = band::kNoSure;  // nothing classified
    int fsh = 0, lmode = 0;
    if (smax > 0 && !keep_all) {
      const float pk = static_cast<float>(k) / static_cast<float>(n);
      const float mu = pk * static_cast<float>(kSample);
      const float sd = sqrtf(fmaxf(mu * (1.0f - pk), 1.0f));
      const int r_hi = static_cast<int>(floorf(mu - kZ * sd));
      const int r_lo = static_cast<int>(ceilf(mu + kZ * sd)) + 1;
      int b_hi, b_lo;
      band::warp_pick_two(sh.hist, r_hi >= 1 ? static_cast<uint32_t>(r_hi) : 0u,
                          r_lo <= kSample ? static_cast<uint32_t>(r_lo) : 0u, lane, &b_hi, &b_lo);
      t_lo = b_lo > 0 ? static_cast<uint32_t>(base + (b_lo << band::kOctaveShift)) : 0u;
      if (b_hi >= 0 && b_hi < kRoundBins - 1)
        t_hi = static_cast<uint32_t>(base + ((b_hi + 1) << band::kOctaveShift));
      if (t_lo > t_hi) t_lo = t_hi;
      const uint32_t fhi = t_hi != band::kNoSure
                               ? t_hi - 1u
                               : min(static_cast<uint32_t>(smax) + (1u << 23), 0x7f7fffffu);
      fsh = round_shift(static_cast<int>(t_lo), static_cast<int>(max(fhi, t_lo)));
      // list mode when the sample's count at or above t_lo, scaled to the row with
      // a margin, fits the list
      uint32_t ge = 0;
      if (b_lo > 0) {
#pragma unroll
        for (int j = 0; j < 8; ++j) ge += (lane * 8 + j >= b_lo) ? sh.hist[lane * 8 + j] : 0u;
      }
      ge = __reduce_add_sync(kFull, ge);
      const float est = static_cast<float>(ge) * static_cast<float>(n) / static_cast<float>(kSample);
      lmode = b_lo > 0 && est * 1.25f + 512.0f <= static_cast<float>(kListCap) &&
              est <= kListShare * static_cast<float>(n);
    }
    __syncwarp();
    for (int i = lane; i < kRoundBins; i += 32) sh.hist[i] = 0;  // the band histogram
    if (lane == 0) {
      sh.t_lo = t_lo;
      sh.t_hi = t_hi;
      sh.fsh = fsh;
      sh.lmode = lmode;
    }
  }
  __syncthreads();

  int T = -1;
  uint32_t need = 0;
  bool use_list = false;
  if (!keep_all) {
    // ---- first pass: classification, the list and the band's histogram ------------
    const float f_lo = __uint_as_float(sh.t_lo), f_hi = __uint_as_float(sh.t_hi);
    const uint32_t t_lo = sh.t_lo, t_hi = sh.t_hi;
    const int fsh = sh.fsh;
    const bool lmode = sh.lmode != 0;
    // x is read again only by the second pass (and, under error feedback, not at all)
    const uint64_t px = (MODE == kEF || lmode) ? drop : keep;
    const uint64_t pa = MODE == kEF ? drop : keep;
    const float* st = reinterpret_cast<const float*>(stage);
    uint32_t n_sure = 0;  // this thread's sure entries (list mode), or its warp's
    for (int c = 0; c < nch; ++c) {
      if (tid == 0) prefetch(c + kAhead);
      const int sc = c * NW + warp;
      const int sb = sc * kSub;
      const int q0 = sb + lane * 4;
      float4 v[kU];
      uint32_t vm = 0xffffu;
      if (sb + kSub <= n) {
#pragma unroll
        for (int u = 0; u < kU; ++u) v[u] = load(q0 + u * 128, nullptr, px, pa);
      } else {
        vm = 0;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
          if (q0 + u * 128 < n) {
            v[u] = load(q0 + u * 128, nullptr, px, pa);
            vm |= 0xfu << (4 * u);
          }
        }
      }
      if (MODE == kEF) {
#pragma unroll
        for (int u = 0; u < kU; ++u)
          if ((vm >> (4 * u)) & 1u) st_f4(arow + q0 + u * 128, v[u], keep);  // err' = s for now
      }
      // |s| >= t_lo for every entry; |s| >= t_hi too in two-pass mode (list mode
      // tells the sure entries apart among the listed ones)
      uint32_t gw = 0;
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        gw |= (static_cast<uint32_t>(fabsf(v[u].x) >= f_lo) << (4 * u + 0)) |
              (static_cast<uint32_t>(fabsf(v[u].y) >= f_lo) << (4 * u + 1)) |
              (static_cast<uint32_t>(fabsf(v[u].z) >= f_lo) << (4 * u + 2)) |
              (static_cast<uint32_t>(fabsf(v[u].w) >= f_lo) << (4 * u + 3));
      }
      gw &= vm;
      uint32_t lw = gw;  // listed
      if (!lmode) {
        uint32_t hw = 0;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          hw |= (static_cast<uint32_t>(fabsf(v[u].x) >= f_hi) << (4 * u + 0)) |
                (static_cast<uint32_t>(fabsf(v[u].y) >= f_hi) << (4 * u + 1)) |
                (static_cast<uint32_t>(fabsf(v[u].z) >= f_hi) << (4 * u + 2)) |
                (static_cast<uint32_t>(fabsf(v[u].w) >= f_hi) << (4 * u + 3));
        }
        hw &= vm;
        const uint32_t ns = __reduce_add_sync(kFull, static_cast<uint32_t>(__popc(hw)));
        if (lane == 0) sh.sc_sure[sc] = ns;
        n_sure += ns;
        lw = gw & ~hw;  // the band
      }
      // the sub-chunk's segment in index order: (group, lane, entry)
      const uint32_t pl = pack_counts(lw);
      const uint32_t il = warp_inclusive_scan(pl, lane);
      const uint32_t tl = __shfl_sync(kFull, il, 31);
      const uint32_t wt = fld(tl, 0) + fld(tl, 1) + fld(tl, 2) + fld(tl, 3);
      uint32_t p0 = 0;
      if (lane == 0) {
        if (wt != 0) p0 = atomicAdd(&sh.mcount, wt);
        sh.seg_start[sc] = p0;
        sh.seg_cnt[sc] = wt;
      }
      if (wt != 0) {
        p0 = __shfl_sync(kFull, p0, 0);
        if (lw != 0) {
          // the values come back from this thread's own stage slots
#pragma unroll
          for (int u = 0; u < kU; ++u) stage[u * NT + tid] = v[u];
          const uint32_t q0 = p0 + fld(il, 0) - fld(pl, 0);
          const uint32_t q1 = p0 + fld(tl, 0) + fld(il, 1) - fld(pl, 1);
          const uint32_t q2 = p0 + fld(tl, 0) + fld(tl, 1) + fld(il, 2) - fld(pl, 2);
          const uint32_t q3 = p0 + fld(tl, 0) + fld(tl, 1) + fld(tl, 2) + fld(il, 3) - fld(pl, 3);
          const uint32_t all = lw;
          while (lw) {
            const int b = __ffs(lw) - 1;
            lw &= lw - 1;
            const int u = b >> 2;
            const uint32_t qu = u == 0 ? q0 : (u == 1 ? q1 : (u == 2 ? q2 : q3));
            const uint32_t p = qu + __popc(all & ((1u << b) - 1u) & (0xffffffffu << (4 * u)));
            const uint32_t bits = __float_as_uint(st[(u * NT + tid) * 4 + (b & 3)]);
            if (p < static_cast<uint32_t>(kListCap)) {
              lval[p] = bits;
              lcol[p] = static_cast<uint16_t>(sb + u * 128 + lane * 4 + (b & 3));
            }
            const uint32_t key = bits & 0x7fffffffu;
            if (lmode && key >= t_hi) {
              ++n_sure;
            } else {
              atomicAdd(&sh.hist[min((key - t_lo) >> fsh, static_cast<uint32_t>(kRoundBins - 1))], 1u);
            }
          }
        }
      }
    }
    if (lmode) n_sure = __reduce_add_sync(kFull, n_sure);
    // n_sure is warp-uniform: the block total from the per-warp sums
    if (lane == 0) sh.r[0][0][warp] = n_sure;
    __syncthreads();
    n_sure = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) n_sure += sh.r[0][0][w];
    const uint32_t m = sh.mcount;
    const uint32_t n_ge = lmode ? m : n_sure + m;  // entries >= t_lo
    const bool fallback = !(static_cast<int64_t>(n_sure) < k && k <= static_cast<int64_t>(n_ge) &&
                            m <= static_cast<uint32_t>(kListCap));
    use_list = lmode && !fallback;
    if (!fallback) {
      // ---- the threshold inside the band ------------------------------------------
      const uint32_t kr = static_cast<uint32_t>(k - n_sure);  // 1 <= kr <= band entries
      if (warp == 0) {
        const BinPick p = warp_pick_bin(sh.hist, kr, lane);
        const uint32_t kr2 = kr - p.above;
        const int bl = static_cast<int>(t_lo) + (p.bin << fsh);
        if (lane == 0) {
          sh.T = bl - 1;  // the bin taken whole
          sh.need = 0;
          sh.resolve = p.count == kr2 ? 0 : (p.count <= static_cast<uint32_t>(kCandCap) ? 1 : 2);
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
        const int bl = static_cast<int>(t_lo) + (sh.pick_bin << fsh);
        // the bin's keys; the top bin takes every larger band key (none reaches t_hi)
        int bh = sh.pick_bin == kRoundBins - 1
                     ? 0x7fffffff
                     : static_cast<int>(min(static_cast<uint32_t>(bl) + ((1u << fsh) - 1u), 0x7fffffffu));
        if (t_hi != band::kNoSure) bh = min(bh, static_cast<int>(t_hi) - 1);
        if (sh.resolve == 2) {
          const Threshold th = band::select_rounds<NT>(
              [&](int i) {
                const int key = static_cast<int>(lval[i] & 0x7fffffffu);
                return (key >= bl && key <= bh) ? key : -1;
              },
              static_cast<int>(m), bl, bh, kr2, sh, tid, lane, warp);
          T = th.T;
          need = th.need;
        } else {
          for (uint32_t i = tid; i < m; i += NT) {
            const int key = static_cast<int>(lval[i] & 0x7fffffffu);
            if (key >= bl && key <= bh) sh.cand[atomicAdd(&sh.ccount, 1u)] = key;
          }
          __syncthreads();
          band::rank_block<NT>(sh.cand, cnt, kr2, &sh.T, &sh.need, tid);
          __syncthreads();
          T = sh.T;
          need = sh.need;
        }
      }
      // ---- kept entries per sub-chunk: the sure ones (two-pass mode), and the
      // listed ones above T or tied, counted by one warp per segment
      for (int sc = warp; sc < nsc; sc += NW) {
        const uint32_t s0 = sh.seg_start[sc], cnt = sh.seg_cnt[sc];
        uint32_t gt = 0, eq = 0;
        for (uint32_t i = lane; i < cnt; i += 32) {
          const int key = static_cast<int>(lval[s0 + i] & 0x7fffffffu);
          gt += key > T;
          eq += key == T;
        }
        gt = __reduce_add_sync(kFull, gt);
        eq = __reduce_add_sync(kFull, eq);
        if (lane == 0) {
          sh.sc_gt[sc] = gt;
          sh.sc_eq[sc] = eq;
          if (lmode) sh.sc_sure[sc] = 0;  // the sure entries are listed
        }
      }
    } else {
      // ---- exact selection over the whole row by integer rounds (from L2) ---------
      auto key_of = [&](int e) -> int {
        float v;
        if (MODE == kEF) v = arow[e];  // s, written by the first pass
        else if (MODE == kDelta) v = fsub(xrow[e], arow[e]);
        else v = xrow[e];
        return static_cast<int>(band::ukey(v));
      };
      // the key range over every entry but NaN (+inf counts: EF-mixed TopK marks
      // entries with it)
      int lo = 0x7fffffff, hi = -1;
      for (int e = tid; e < n; e += NT) {
        const int key = key_of(e);
        if (key <= 0x7f800000) {
          lo = min(lo, key);
          hi = max(hi, key);
        }
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
      const Threshold th = band::select_rounds<NT>(key_of, n, lo, hi, static_cast<uint32_t>(k),
                                                   sh, tid, lane, warp);
      T = th.T;
      need = th.need;
      // kept entries per sub-chunk, counted over the row (sure counts are void here)
      const float tf = __uint_as_float(static_cast<uint32_t>(T));  // T >= 0: k < n
      for (int c = 0; c < nch; ++c) {
        const int sb = c * kChunk + warp * kSub;
        uint32_t gt = 0, eq = 0;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int q = sb + u * 128 + lane * 4;
          if (q < n) {
            const float4 v = MODE == kEF ? ld_f4(arow + q, keep) : load(q, nullptr, keep, keep);
            or_if_gt(gt, v.x, tf, 1u << (4 * u + 0));
            or_if_gt(gt, v.y, tf, 1u << (4 * u + 1));
            or_if_gt(gt, v.z, tf, 1u << (4 * u + 2));
            or_if_gt(gt, v.w, tf, 1u << (4 * u + 3));
            or_if_eq(eq, v.x, tf, 1u << (4 * u + 0));
            or_if_eq(eq, v.y, tf, 1u << (4 * u + 1));
            or_if_eq(eq, v.z, tf, 1u << (4 * u + 2));
            or_if_eq(eq, v.w, tf, 1u << (4 * u + 3));
          }
        }
        const uint32_t ngt = __reduce_add_sync(kFull, static_cast<uint32_t>(__popc(gt)));
        const uint32_t neq = __reduce_add_sync(kFull, static_cast<uint32_t>(__popc(eq)));
        if (lane == 0) {
          sh.sc_sure[c * NW + warp] = 0;
          sh.sc_gt[c * NW + warp] = ngt;
          sh.sc_eq[c * NW + warp] = neq;
        }
      }
    }
    __syncthreads();
    // ---- payload offsets per sub-chunk (index order), ties allotted in index order --
    if (warp == 0) {
      constexpr int kPer = kMaxSub / 32;
      uint32_t eq[kPer], kc[kPer], es = 0;
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        const int sc = lane * kPer + i;
        eq[i] = sc < nsc ? sh.sc_eq[sc] : 0u;
        kc[i] = sc < nsc ? sh.sc_sure[sc] + sh.sc_gt[sc] : 0u;
        es += eq[i];
      }
      uint32_t eb = warp_inclusive_scan(es, lane) - es;  // ties before this lane's sub-chunks
      uint32_t ks = 0;
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        const uint32_t tie = need > eb ? min(need - eb, eq[i]) : 0u;
        eb += eq[i];
        sh.sc_tie[lane * kPer + i] = tie;
        kc[i] += tie;
        ks += kc[i];
      }
      uint32_t kb = warp_inclusive_scan(ks, lane) - ks;
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        sh.sc_base[lane * kPer + i] = kb;
        sh.sc_kept[lane * kPer + i] = kc[i];
        kb += kc[i];
      }
    }
  } else {
    // every entry kept
    for (int sc = tid; sc < kMaxSub; sc += NT) {
      sh.sc_base[sc] = static_cast<uint32_t>(sc * kSub);
      sh.sc_kept[sc] = sc < nsc ? static_cast<uint32_t>(min(kSub, n - sc * kSub)) : 0u;
      sh.sc_tie[sc] = 0;
    }
  }
  __syncthreads();  // the stage is free; the offsets are in place
  pdl_end();

  float* vrow = a.vals + row * k;
  int32_t* irow = a.idx + row * k;
  if (use_list) {
    // ---- list mode: the payload from each sub-chunk's segment -----------------------
    const unsigned lt = lanemask_lt();
    for (int sc = warp; sc < nsc; sc += NW) {
      if (sh.sc_kept[sc] == 0) continue;
      const uint32_t s0 = sh.seg_start[sc], cnt = sh.seg_cnt[sc], tq = sh.sc_tie[sc];
      uint32_t pos = sh.sc_base[sc], eqseen = 0;
      for (uint32_t i0 = 0; i0 < cnt; i0 += 32) {
        const uint32_t i = i0 + lane;
        const bool in = i < cnt;
        const uint32_t bits = in ? lval[s0 + i] : 0u;
        const int col = in ? static_cast<int>(lcol[s0 + i]) : 0;
        const int key = static_cast<int>(bits & 0x7fffffffu);
        const bool eq = in && key == T;
        const unsigned be = __ballot_sync(kFull, eq);
        const bool kp = (in && key > T) || (eq && eqseen + __popc(be & lt) < tq);
        eqseen += __popc(be);
        const unsigned bk = __ballot_sync(kFull, kp);
        if (kp) {
          const uint32_t p = pos + __popc(bk & lt);
          const float v = __uint_as_float(bits);
          if (p < static_cast<uint32_t>(k)) {
            st_f32(vrow + p, v, drop);
            st_s32(irow + p, col, drop);
          }
          if (MODE == kEF) st_f32(arow + col, 0.0f, drop);                   // err' = s - C(s)
          if (MODE == kDelta) st_f32(arow + col, fadd(arow[col], v), drop);  // state + d
        }
        pos += __popc(bk);
      }
    }
    return;
  }

  // ---- two-pass mode: the second pass ------------------------------------------------
  // Each warp on its own sub-chunks: kept entries |s| > T (all finite entries when T
  // is -1), and the sub-chunk's quota of ties |s| == T, first in index order.
  // this warp's share of the stage: (value, column) pairs of two 128-entry groups
  const uint2* op = reinterpret_cast<const uint2*>(stage) + warp * 256;
  const uint32_t op_s = static_cast<uint32_t>(__cvta_generic_to_shared(op));
  const float tf = T >= 0 ? __uint_as_float(static_cast<uint32_t>(T)) : -1.0f;
  for (int c = 0; c < nch; ++c) {
    const int sc = c * NW + warp;
    if (sh.sc_kept[sc] == 0) continue;  // nothing sent; err' = s and the state stand
    const uint32_t tq = sh.sc_tie[sc];
    uint32_t ubase = sh.sc_base[sc];
    const int sb = sc * kSub;
    float4 v[kU], g[kU];
    uint32_t vm = 0;
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int q = sb + u * 128 + lane * 4;
      v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      g[u] = v[u];
      if (q < n) {
        if (MODE == kEF && !keep_all) v[u] = ld_f4(arow + q, drop);  // s
        else v[u] = load(q, &g[u], drop, drop);
        vm |= 0xfu << (4 * u);
      }
    }
    uint32_t kw = 0;
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      or_if_gt(kw, v[u].x, tf, 1u << (4 * u + 0));
      or_if_gt(kw, v[u].y, tf, 1u << (4 * u + 1));
      or_if_gt(kw, v[u].z, tf, 1u << (4 * u + 2));
      or_if_gt(kw, v[u].w, tf, 1u << (4 * u + 3));
    }
    kw &= vm;
    if (tq != 0) {
      // this sub-chunk's first tq ties in (group, lane, entry) order
      uint32_t ew = 0;
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        or_if_eq(ew, v[u].x, tf, 1u << (4 * u + 0));
        or_if_eq(ew, v[u].y, tf, 1u << (4 * u + 1));
        or_if_eq(ew, v[u].z, tf, 1u << (4 * u + 2));
        or_if_eq(ew, v[u].w, tf, 1u << (4 * u + 3));
      }
      ew &= vm;
      const uint32_t pe = pack_counts(ew);
      const uint32_t ie = warp_inclusive_scan(pe, lane);
      const uint32_t te = __shfl_sync(kFull, ie, 31);
      uint32_t before = 0;
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        uint32_t nib = (ew >> (4 * u)) & 0xfu;
        const uint32_t b = before + fld(ie, u) - fld(pe, u);
        uint32_t take = tq > b ? min(tq - b, static_cast<uint32_t>(__popc(nib))) : 0u;
        while (nib && take) {
          kw |= (nib & (~nib + 1u)) << (4 * u);
          nib &= nib - 1;
          --take;
        }
        before += fld(te, u);
      }
    }
    const uint32_t pk = pack_counts(kw);
    const uint32_t ik = warp_inclusive_scan(pk, lane);
    const uint32_t tk = __shfl_sync(kFull, ik, 31);
#pragma unroll
    for (int u0 = 0; u0 < kU; u0 += 2) {
      // the kept entries of groups u0 and u0 + 1 staged in index order by
      // predicated stores, then out with coalesced stores
      const uint32_t ta = fld(tk, u0), tr = ta + fld(tk, u0 + 1);
      if (tr != 0) {
        uint32_t at = op_s + 8u * (fld(ik, u0) - fld(pk, u0));
        stage_kept4((kw >> (4 * u0)) & 0xfu, at, v[u0], sb + u0 * 128 + lane * 4);
        at = op_s + 8u * (ta + fld(ik, u0 + 1) - fld(pk, u0 + 1));
        stage_kept4((kw >> (4 * (u0 + 1))) & 0xfu, at, v[u0 + 1], sb + (u0 + 1) * 128 + lane * 4);
        __syncwarp();
        const uint32_t lim = static_cast<int64_t>(ubase) < k
                                 ? static_cast<uint32_t>(min(static_cast<int64_t>(tr), k - ubase))
                                 : 0u;
        for (uint32_t i = lane; i < lim; i += 32) {
          const uint2 e = op[i];
          st_f32(vrow + ubase + i, __uint_as_float(e.x), drop);
          st_s32(irow + ubase + i, static_cast<int32_t>(e.y), drop);
        }
        __syncwarp();
        ubase += tr;
      }
#pragma unroll
      for (int u = u0; u < u0 + 2; ++u) {
        const uint32_t nib = (kw >> (4 * u)) & 0xfu;
        const int col0 = sb + u * 128 + lane * 4;
        if (MODE != kPlain && nib != 0) {
          float4 w4;
          if (MODE == kEF) {  // err' = s - C(s): +0 where sent
            w4 = make_float4((nib & 1u) ? 0.0f : v[u].x, (nib & 2u) ? 0.0f : v[u].y,
                             (nib & 4u) ? 0.0f : v[u].z, (nib & 8u) ? 0.0f : v[u].w);
          } else {  // state + d where sent
            w4 = make_float4((nib & 1u) ? fadd(g[u].x, v[u].x) : g[u].x,
                             (nib & 2u) ? fadd(g[u].y, v[u].y) : g[u].y,
                             (nib & 4u) ? fadd(g[u].z, v[u].z) : g[u].z,
                             (nib & 8u) ? fadd(g[u].w, v[u].w) : g[u].w);
          }
          st_f4(arow + col0, w4, drop);
        }
      }
    }
  }
}

// Rows this kernel takes: 8193..65536 entries, 16-byte aligned rows.
inline bool fits(const TopkRowArgs& a) { return a.aligned && a.L >= kMinL && a.L <= kMaxL; }

template <int MODE>
cudaError_t run_mode(const TopkRowArgs& a, cudaStream_t s) {
  auto kernel = topk_lrow_kernel<MODE>;
  cudaError_t err = ensure_dynamic_smem(kernel, kSmemBytes);
  if (err != cudaSuccess) return err;
  if (a.rows > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_kernel(kernel, dim3(static_cast<unsigned>(a.rows)), dim3(NT), kSmemBytes, s, 0u, a);
}

}  // namespace lrow
}  // namespace mpc
