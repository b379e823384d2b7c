// topk_rows.cuh -- exact per-row TopK (§2.3) for rows that fit on chip, fused
// with error feedback (§2.4, Seide et al.) and with the EF21 / AQ-SGD buffer
// update (§2.4, §2.5).  Kernel templates; topk_rows_{plain,ef,delta}.cu
// instantiate them, one fused variant per translation unit.
//
// Two kernels share the selection of select.cuh.  Both read x (and the error
// or state row) from HBM once, keep the ranked values (x, x + err or
// x - state) on chip, write the payload once, write err once (error
// feedback) or the state at the kept entries only (EF21 / AQ-SGD).
//
//  * topk_cta_kernel: rows longer than 1024 entries.  One thread-block cluster
//    of C CTAs per row, each CTA holding a slice of up to SCAP entries.  The
//    slice of x arrives by one bulk asynchronous copy completing on an
//    mbarrier; the error / state slice by 16-byte loads issued at the same
//    time.  Passes over the slice: ranked values with the histogram, count-and-collect
//    (entries above the chosen bin are counted per 128-entry chunk, entries in
//    it are appended to a candidate list), write.  The CTAs of a cluster push
//    histogram group sums, candidate lists and counts into each other's shared
//    memory (st.shared::cluster) before a cluster barrier and pull only the few
//    bins of the chosen group: two cluster barriers per row, none at exit.  The
//    bin scale comes from a sample of the row that every CTA of the cluster
//    reads identically, so the histogram is built in the same pass that forms
//    the ranked values and no barrier is spent on the row maximum.
//  * topk_warp_kernel: one warp per row for rows of at most 1024 entries,
//    persistent over rows; each warp double-buffers its rows with its own bulk
//    copies and mbarriers, so the next row loads while this one is selected.
//    The row stays in registers (plain TopK: the keys; the fused variants: the
//    ranked values), the selection's histogram and candidates in the warp's
//    scratch.  The write marks the kept entries, places each group of 128 by one
//    packed warp scan, stages the kept (value, column) pairs of two groups at a
//    time in the scratch with predicated stores, and copies them out with
//    coalesced stores.
//
// FULL instantiations drop the per-entry end-of-slice checks; they run when
// every 4-entry slot a thread processes lies inside the slice.
#pragma once

#include "common.cuh"
#include "kernels.h"
#include "launch_util.h"
#include "select.cuh"
#include "topk_band.cuh"
#include "topk_lrow.cuh"

namespace mpc {
namespace rows {

constexpr int kNB = 1024;   // bins of the first histogram, CTA kernel
constexpr int kLCAP = 256;  // candidate keys per row, CTA kernel (whole cluster)
constexpr int kLCAPW = 256;   // candidate keys per row, warp kernel
constexpr int kMaxCluster = 8;
constexpr int kSampleThreads = 64;  // threads that read the row sample (4 entries each)

// The value the selection ranks, for each fused variant.
template <int MODE>
__device__ __forceinline__ float ranked_value(float x, float a) {
  if (MODE == kEF) return fadd(x, a);     // s = x + err
  if (MODE == kDelta) return fsub(x, a);  // d = x - state
  return x;
}

template <int MODE>
__device__ __forceinline__ float4 ranked4(float4 x, float4 a) {
  return make_float4(ranked_value<MODE>(x.x, a.x), ranked_value<MODE>(x.y, a.y),
                     ranked_value<MODE>(x.z, a.z), ranked_value<MODE>(x.w, a.w));
}

// Keys of the 4 entries base..base+3 (-1 past the slice end n, unless FULL).
template <bool FULL>
__device__ __forceinline__ void keys4(const float4 v, int base, int n, int k[4]) {
  if (FULL) {
    k[0] = mag_key(v.x);
    k[1] = mag_key(v.y);
    k[2] = mag_key(v.z);
    k[3] = mag_key(v.w);
  } else {
    k[0] = (base + 0 < n) ? mag_key(v.x) : -1;
    k[1] = (base + 1 < n) ? mag_key(v.y) : -1;
    k[2] = (base + 2 < n) ? mag_key(v.z) : -1;
    k[3] = (base + 3 < n) ? mag_key(v.w) : -1;
  }
}

// Bin of a key (>= 0) in the first histogram of the CTA kernel: |x| * scale
// rounded down and capped at kNB - 1 (scale = kNB / the largest magnitude of
// a sample of the row), in FP32 operations only: the cap first, then the
// floor as the low mantissa bits of p + 2^23 rounded toward zero.  Monotone
// in the key.
__device__ __forceinline__ int lin_bin(int key, float scale) {
  const float p = fminf(fmul(__int_as_float(key), scale), static_cast<float>(kNB - 1));
  return __float_as_int(__fadd_rz(p, 8388608.0f)) & 0x7fffff;
}

// ---------------------------------------------------------------------------
// Block-level reductions and scans (NT threads)
// ---------------------------------------------------------------------------
template <int NT>
__device__ __forceinline__ int block_max(int v, int* red, int lane, int warp) {
  v = __reduce_max_sync(kFull, v);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  const int r = __reduce_max_sync(kFull, lane < NT / 32 ? red[lane] : red[0]);
  __syncthreads();
  return r;
}

template <int NT>
__device__ __forceinline__ int block_min(int v, int* red, int lane, int warp) {
  v = __reduce_min_sync(kFull, v);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  const int r = __reduce_min_sync(kFull, lane < NT / 32 ? red[lane] : red[0]);
  __syncthreads();
  return r;
}

template <int NT>
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* red, int lane, int warp) {
  const uint32_t inc = warp_inclusive_scan(v, lane);
  if (lane == 31) red[warp] = inc;
  __syncthreads();
  // the warps' totals, one per lane, scanned: this warp's base is the sum before it
  const uint32_t t = lane < NT / 32 ? red[lane] : 0u;
  const uint32_t base = __shfl_sync(kFull, warp_inclusive_scan(t, lane) - t, warp);
  __syncthreads();
  return base + inc - v;
}

// ---------------------------------------------------------------------------
// CTA / cluster kernel
// ---------------------------------------------------------------------------
// The first pick of the CTA kernel: bin B, the entries above it and in it
// (whole row), its first and last keys, this CTA's entries in it and those of
// the CTAs before it.
struct PickOut {
  int B;
  uint32_t above, m;
  int kl, kh;
  uint32_t own, off;
};

template <int NT, int SCAP>
struct CtaShared {
  static constexpr int NW = NT / 32;
  static constexpr int NCH = SCAP / 128;  // chunks of 128 consecutive entries
  // The first histogram; dead once it has been packed and pushed, after which
  // the same words hold the row's candidate keys, this CTA's candidate chunks
  // and the histograms of the integer rounds.
  union {
    uint32_t hist[kNB + 64];  // + 32 zero spill counters, + 32 past-the-end ones
    struct {
      int cand[kLCAP];        // the row's candidates, CTA by CTA (pushed)
      uint16_t lch[kLCAP];    // chunk of each of this CTA's candidates
    } c;
    uint32_t rhist[2][kRoundBins];
  } u;
  uint32_t cgt[NCH];     // per chunk: entries kept for being above T (or bin B)
  uint32_t ceq[NCH];     // per chunk: entries equal to T
  uint32_t gbins[128];
  uint32_t wtot[kMaxCluster][NW];  // per CTA and warp: entries above bin B (pushed)
  uint32_t tot_gt[kMaxCluster];    // pushed by the lower ranks of the cluster
  uint32_t tot_eq[kMaxCluster];
  int red[NW];
  uint32_t ured[NW];
  int sample_max[2];
  uint32_t lcount;
  uint32_t pick_t, pick_excl;
  int pub_lo, pub_hi;
  uint32_t before_gt, before_eq;
  uint8_t woff[NW][128];  // per warp: column offsets of a chunk's staged kept entries
  BinPick pick;
  PickOut pk;
  Threshold thr;
  uint64_t bars[8];  // one per slice chunk (one float4 slot of every thread)
};

// The bin holding the kr-th element of an NBINS-bin histogram (bins ranked
// high to low) summed over the cluster's C CTAs (integer rounds).  Each thread
// owns a group of G consecutive bins; group sums are pushed to every CTA
// (table `gsum`, C x NT words), scanned locally, and only the chosen group's
// bins are pulled from the other CTAs.
template <int NT, int NBINS, class Sh>
__device__ __forceinline__ BinPick cluster_pick(const uint32_t* hist, uint32_t* gsum, uint32_t C,
                                                uint32_t crank, uint32_t kr, Sh& sh, int tid,
                                                int lane, int warp) {
  constexpr int NG = NT < NBINS ? NT : NBINS;  // bin groups: thread t < NG owns group t
  constexpr int G = NBINS / NG;
  static_assert(G * NG == NBINS && G * kMaxCluster <= 128, "bin groups");
  uint32_t gs = 0;
  if (tid < NG) {
#pragma unroll
    for (int b = 0; b < G; ++b) gs += hist[NBINS - 1 - (tid * G + b)];
  }
  uint32_t total = gs;
  if (C > 1) {
    uint32_t* mine = gsum + crank * NT + tid;
    for (uint32_t r = 0; r < C; ++r) dsmem_st_u32(dsmem_addr(mine, r), gs);
    cluster_sync();
    total = 0;
    for (uint32_t r = 0; r < C; ++r) total += gsum[r * NT + tid];
  }
  if (tid == 0) {
    sh.pick_t = 0;
    sh.pick_excl = 0;
  }
  const uint32_t excl = block_excl_scan<NT>(total, sh.ured, lane, warp);
  if (excl < kr && kr <= excl + total) {
    sh.pick_t = tid;
    sh.pick_excl = excl;
  }
  __syncthreads();
  const uint32_t tg = sh.pick_t;
  if (tid < G * static_cast<int>(C)) {
    const int r = tid / G, b = tid % G;
    const uint32_t* p = &hist[NBINS - 1 - (tg * G + b)];
    sh.gbins[tid] = (C > 1) ? dsmem_ld_u32(dsmem_addr(p, r)) : *p;
  }
  __syncthreads();
  if (tid == 0) {
    uint32_t run = sh.pick_excl;
    BinPick pk = {NBINS - 1 - static_cast<int>(tg * G), run, 0};
    for (int b = 0; b < G; ++b) {
      uint32_t cnt = 0;
      for (uint32_t r = 0; r < C; ++r) cnt += sh.gbins[r * G + b];
      pk = BinPick{NBINS - 1 - static_cast<int>(tg * G + b), run, cnt};
      if (run + cnt >= kr) break;
      run += cnt;
    }
    sh.pick = pk;
  }
  __syncthreads();
  return sh.pick;
}

// Warp 0: exclusive scan in place of per-chunk counts; returns the total.
template <int NCH>
__device__ __forceinline__ uint32_t scan_chunks1(uint32_t* c, int lane) {
  constexpr int PER = (NCH + 31) / 32;
  uint32_t g[PER], t = 0;
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int ch = lane * PER + j;
    g[j] = ch < NCH ? c[ch] : 0u;
    t += g[j];
  }
  uint32_t e = warp_inclusive_scan(t, lane) - t;
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int ch = lane * PER + j;
    if (ch < NCH) c[ch] = e;
    e += g[j];
  }
  return __shfl_sync(kFull, e, 31);
}

// Bytes of dynamic shared memory of the CTA kernel for cluster size C: the
// slice, and the packed histograms of the C CTAs (kNB / 2 words each; the
// group-sum tables of the integer rounds, 2 x C x NT words, reuse them).
constexpr int cta_smem_bytes(int NT, int SCAP, int C) {
  return SCAP * 4 + C * (kNB / 2 > 2 * NT ? kNB / 2 : 2 * NT) * 4;
}

// Barrier over the row: the cluster, or the CTA when the row has one CTA.
__device__ __forceinline__ void row_sync(uint32_t C) {
  if (C > 1) cluster_sync();
  else __syncthreads();
}

template <int MODE, int NT, int SCAP, bool FULL>
__global__ void __launch_bounds__(NT, (NT == 128 ? 6 : NT == 256 ? 4 : NT == 512 ? 2 : 1))
    topk_cta_kernel(const TopkRowArgs a) {
  pdl_begin();
  constexpr int NW = NT / 32;
  constexpr int NQ = SCAP / 4;     // float4 slots per slice
  constexpr int QPT = NQ / NT;     // float4 slots per thread
  constexpr int NCH = SCAP / 128;  // 128-entry chunks per slice
  constexpr int G = kNB / NT;      // bins of a thread's group in the first histogram
  constexpr int GW = G / 2;        // packed words of a group (two 16-bit counts each)
  // A wide CTA (512 or 1024 threads) holds a whole row: no cluster, and the
  // histogram is read where it was built.
  constexpr bool kWide = NT >= 512;
  static_assert(G == 4 || G == 8 || (kWide && (G == 1 || G == 2)), "bin groups");
  static_assert(SCAP < 65536, "per-CTA bin counts fit 16 bits");
  using Sh = CtaShared<NT, SCAP>;
  __shared__ Sh sh;
  extern __shared__ __align__(16) float4 dyn4[];

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t C = cluster_size();
  const uint32_t crank = cluster_rank();
  float4* s4 = dyn4;                                         // NQ float4: ranked values
  uint32_t* table = reinterpret_cast<uint32_t*>(dyn4 + NQ);  // C x NT x GW packed bins
  const int64_t row = blockIdx.x / C;
  const int64_t L = a.L;
  const int64_t k = a.k;
  const int64_t c0 = static_cast<int64_t>(crank) * a.slice;
  const int n = static_cast<int>(max64(0, min64(a.slice, L - c0)));

  // Row of the error (EF) or state (EF21 / AQ-SGD) buffer.  Every CTA of the
  // cluster reads the same id, so all of them leave together, before any
  // cluster barrier.
  float* arow = nullptr;
  if (MODE != kPlain) {
    int64_t srow = row;
    if (MODE == kDelta && a.ids != nullptr) {
      const int64_t sid = a.ids[row / a.rps];
      if (sid < 0 || sid >= a.num_samples) {
        if (tid == 0 && crank == 0) set_status(a.status, STATUS_BAD_SAMPLE);
        return;
      }
      srow = sid * a.rps + row % a.rps;
    }
    arow = a.aux + srow * L;
  }
  const float* xrow = a.x + row * L;

  // ---- issue the loads: a sample of the row, x by bulk copies, err / state ----
  // The bin placement comes from a sample of the row, entries [p, p+4) spread
  // over it, read identically by every CTA of the cluster; it is requested
  // first, so that it is not queued behind the slices.
  float sx[4] = {0.f, 0.f, 0.f, 0.f}, sa[4] = {0.f, 0.f, 0.f, 0.f};
  const int64_t sp = (L / kSampleThreads) * tid / 4 * 4;
  if (tid < kSampleThreads) {
    if (a.aligned && sp + 4 <= L) {
      const float4 v = *reinterpret_cast<const float4*>(xrow + sp);
      sx[0] = v.x, sx[1] = v.y, sx[2] = v.z, sx[3] = v.w;
      if (MODE != kPlain) {
        const float4 w = *reinterpret_cast<const float4*>(arow + sp);
        sa[0] = w.x, sa[1] = w.y, sa[2] = w.z, sa[3] = w.w;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (sp + i < L) {
          sx[i] = xrow[sp + i];
          if (MODE != kPlain) sa[i] = arow[sp + i];
        }
    }
  }
  // The slice of x arrives in chunks of one float4 slot per thread (4*NT
  // entries), each completing on its own mbarrier and issued by its own lane,
  // so the first pass starts on chunk 0 while the others are in flight.
  static_assert(QPT <= 8, "one mbarrier per chunk");
  const int jmax = (n + 4 * NT - 1) / (4 * NT);  // float4 slots of each thread in use
  // The matching chunks of the error / state slice are prefetched into L2 by
  // the same lanes and read from there chunk by chunk in the first pass.
  if (a.aligned && warp == 0 && lane < jmax) {
    const uint32_t bytes = static_cast<uint32_t>(min(4 * NT, n - 4 * NT * lane)) * 4u;
    if (MODE != kPlain) bulk_prefetch_l2(arow + c0 + 4 * NT * lane, bytes);
    mbar_init(&sh.bars[lane], 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(&sh.bars[lane], bytes);
    bulk_g2s(s4 + lane * NT, xrow + c0 + 4 * NT * lane, bytes, &sh.bars[lane]);
  }
  auto aux4 = [&](int j) {
    const int q = j * NT + tid;
    return (a.aligned && MODE != kPlain && j < QPT && 4 * q < n)
               ? *reinterpret_cast<const float4*>(arow + c0 + 4 * q)
               : make_float4(0.f, 0.f, 0.f, 0.f);
  };
  float4 anext = aux4(0);
  for (int i = tid; i < kNB + 64; i += NT) sh.u.hist[i] = 0;
  if (tid == 0) {
    sh.lcount = 0;
    sh.thr = Threshold{0x7fffffff, 0};
  }
  if (tid < kSampleThreads) {
    int smax = -1;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (sp + i < L) smax = max(smax, finite_key(mag_key(ranked_value<MODE>(sx[i], sa[i]))));
    smax = __reduce_max_sync(kFull, smax);
    if (lane == 0) sh.sample_max[warp] = smax;
  }
  if (!a.aligned) {
    float* s = reinterpret_cast<float*>(s4);
    for (int e = tid; e < n; e += NT)
      s[e] = ranked_value<MODE>(xrow[c0 + e], (MODE != kPlain) ? arow[c0 + e] : 0.0f);
  }
  __syncthreads();
  const int smax = max(sh.sample_max[0], sh.sample_max[1]);
  const float scale = bucket_scale(smax, kNB);
  const bool binned = k < L && scale > 0.0f;

  // ---- ranked values into shared memory and the first histogram -------------
  bool failed = false;
#pragma unroll
  for (int j = 0; j < QPT; ++j) {
    if (j < jmax) {
      const float4 acur = anext;
      if (MODE != kPlain && j + 1 < QPT) anext = aux4(j + 1);
      if (a.aligned && !mbar_wait_bounded(&sh.bars[j], 0, a.spin_limit, a.status)) {
        mbar_wait_bounded(&sh.bars[j], 0, kDrainPolls, nullptr);
        failed = true;
      }
      const int q = j * NT + tid;
      float4 v = s4[q];
      if (MODE != kPlain && a.aligned) {
        v = ranked4<MODE>(v, acur);
        s4[q] = v;
      }
      if (binned) {
        int kk[4];
        keys4<FULL>(v, 4 * q, n, kk);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          // one atomic per entry and no branch: zeros (common after ReLU) go to
          // this lane's own spill counter rather than all to bin 0 (folded into
          // bin 0 when the histogram is packed), slots past the slice end to a
          // second spill counter that is never read
          const int b = lin_bin(kk[i], scale);
          const int slot = kk[i] > 0 ? b : ((FULL || kk[i] == 0) ? kNB + lane : kNB + 32 + lane);
          atomicAdd(&sh.u.hist[slot], 1u);
        }
      }
    }
  }
  failed = __syncthreads_or(failed);
  // A slice whose copy timed out takes part in the rest as an empty one (the
  // status word reports the timeout; the row's outputs are then unspecified).
  const int nv = failed ? 0 : n;
  const int jv = failed ? 0 : jmax;

  // ---- select T and need -----------------------------------------------------
  int T = -1;
  uint32_t need = 0;
  bool counted = false;  // per-chunk counts of kept entries are in place (fast path)
  uint32_t own = 0, off = 0;  // this CTA's candidates and those of the CTAs before it
  uint32_t gt_before = 0, eq_before = 0;  // kept / tied entries of the earlier CTAs
  if (k < L) {
    uint32_t kr = static_cast<uint32_t>(k);
    int B = 0;
    uint32_t m = static_cast<uint32_t>(L);  // with scale 0 every entry is a candidate
    int kl = 0, kh = 0x7fffffff;            // the keys of bin B
    if (scale > 0.0f) {
      // Every CTA pushes its histogram, packed two 16-bit counts to a word, to
      // every CTA of the row; thread t owns group t of G bins (groups ranked
      // high to low).  A wide CTA folds the zeros into bin 0 and reads its
      // histogram in place.
      if constexpr (kWide) {
        if (warp == 0) {
          const uint32_t z = __reduce_add_sync(kFull, sh.u.hist[kNB + lane]);
          if (lane == 0) sh.u.hist[0] += z;
        }
      } else {
        const int b0 = kNB - G * (tid + 1);
        uint32_t w[GW];
#pragma unroll
        for (int i = 0; i < GW; ++i) w[i] = sh.u.hist[b0 + 2 * i] | (sh.u.hist[b0 + 2 * i + 1] << 16);
        if (b0 == 0) {
          // the zeros, from the spill counters, into bin 0
          uint32_t z = 0;
          for (int l = 0; l < 32; ++l) z += sh.u.hist[kNB + l];
          w[0] += z;
        }
        uint32_t* dst = table + (crank * NT + tid) * GW;
        if (C > 1) {
          for (uint32_t r = 0; r < C; ++r) {
            if (GW == 2) dsmem_st_u32x2(dsmem_addr(dst, r), make_uint2(w[0], w[1]));
            else dsmem_st_u32x4(dsmem_addr(dst, r), make_uint4(w[0], w[1], w[GW > 2 ? 2 : 0], w[GW > 3 ? 3 : 0]));
          }
        } else {
#pragma unroll
          for (int i = 0; i < GW; ++i) dst[i] = w[i];
        }
      }
      row_sync(C);
      // counts of group g's bins (ascending) summed over the row
      auto group_bins = [&](int g, uint32_t (&cnt)[G]) {
        if constexpr (kWide) {
#pragma unroll
          for (int b = 0; b < G; ++b) cnt[b] = sh.u.hist[kNB - G * (g + 1) + b];
        } else {
#pragma unroll
          for (int b = 0; b < G; ++b) cnt[b] = 0;
          for (uint32_t r = 0; r < C; ++r) {
            const uint32_t* src = table + (r * NT + g) * GW;
#pragma unroll
            for (int i = 0; i < GW; ++i) {
              const uint32_t wv = src[i];
              cnt[2 * i] += wv & 0xffffu;
              cnt[2 * i + 1] += wv >> 16;
            }
          }
        }
      };
      uint32_t cnt[G];
      group_bins(tid, cnt);
      uint32_t total = 0;
#pragma unroll
      for (int b = 0; b < G; ++b) total += cnt[b];
      const uint32_t incl = warp_inclusive_scan(total, lane);
      if (lane == 31) sh.ured[warp] = incl;
      __syncthreads();
      // the warp whose groups hold the kr-th entry (every warp finds the same):
      // a scan of the warps' totals, one per lane
      const uint32_t wu = lane < NW ? sh.ured[lane] : 0u;
      const uint32_t wi = warp_inclusive_scan(wu, lane);
      const unsigned reach = __ballot_sync(kFull, lane < NW - 1 && wi >= kr);
      const int ws = reach ? __ffs(reach) - 1 : NW - 1;
      const uint32_t wbase = __shfl_sync(kFull, wi - wu, ws);
      if (warp == ws) {
        // that warp finds the bin, this CTA's entries in it and those of the
        // CTAs before it, and the bin's first and last keys
        const uint32_t ex = wbase + incl - total;
        const unsigned who = __ballot_sync(kFull, ex < kr && kr <= ex + total);
        const int src = who ? __ffs(who) - 1 : 31;
        const int gb0 = kNB - G * (tid + 1);
        int pb = gb0;
        uint32_t pab = ex, pc = cnt[0];
        {
          uint32_t run = ex;
          bool done = false;
#pragma unroll
          for (int b = G - 1; b >= 0; --b) {
            if (!done && run + cnt[b] >= kr) {
              pb = gb0 + b;
              pab = run;
              pc = cnt[b];
              done = true;
            }
            if (!done) run += cnt[b];
          }
        }
        const int Bw = __shfl_sync(kFull, pb, src);
        const uint32_t above = __shfl_sync(kFull, pab, src);
        const uint32_t mw = __shfl_sync(kFull, pc, src);
        const int gB = (kNB - 1 - Bw) / G;
        const int ib = Bw - (kNB - G * (gB + 1));
        uint32_t cr = 0;
        if constexpr (kWide) {
          (void)gB;
          (void)ib;
          cr = lane == 0 ? mw : 0u;
        } else if (lane < static_cast<int>(C)) {
          const uint32_t wv = table[(lane * NT + gB) * GW + ib / 2];
          cr = (ib & 1) ? (wv >> 16) : (wv & 0xffffu);
        }
        const uint32_t offw = __reduce_add_sync(kFull, lane < static_cast<int>(crank) ? cr : 0u);
        const uint32_t ownw = __shfl_sync(kFull, cr, crank);
        // lanes 0 and 1 find the first keys of bins B and B + 1 side by side
        const int bb = Bw + (lane & 1);
        const float inv = fmul(__int_as_float(smax), 1.0f / kNB);
        const int fk = (bb >= 1 && bb < kNB) ? bin_first_key(bb, scale, inv) : 0;
        const int klw = (Bw == 0) ? 0 : __shfl_sync(kFull, fk, 0);
        const int khw = (Bw == kNB - 1) ? 0x7fffffff : __shfl_sync(kFull, fk, 1) - 1;
        if (lane == 0) sh.pk = PickOut{Bw, above, mw, klw, khw, ownw, offw};
      }
      __syncthreads();
      B = sh.pk.B;
      kr -= sh.pk.above;
      m = sh.pk.m;
      kl = sh.pk.kl;
      kh = sh.pk.kh;
      own = sh.pk.own;
      off = sh.pk.off;
    }

    if (scale > 0.0f && m <= static_cast<uint32_t>(kLCAP)) {
      // ---- count and collect: entries above bin B are kept; the m entries in
      // it are the candidates for T, pushed to every CTA of the row at their
      // place in the row's candidate table ------------------------------------
      uint32_t wab = 0;
#pragma unroll 1
      for (int j = 0; j < QPT; ++j) {
        uint32_t ab = 0;
        if (j < jv) {
          const int q = j * NT + tid;
          int kk[4];
          keys4<FULL>(s4[q], 4 * q, nv, kk);
          bool inb[4];
          bool anyb = false;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            ab += kk[i] > kh;
            inb[i] = static_cast<uint32_t>(kk[i] - kl) <= static_cast<uint32_t>(kh - kl);
            anyb |= inb[i];
          }
          if (__any_sync(kFull, anyb)) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              if (inb[i]) {
                const uint32_t at = atomicAdd(&sh.lcount, 1u);
                if (at < own) {
                  sh.u.c.lch[at] = static_cast<uint16_t>(j * NW + warp);
                  int* slot = &sh.u.c.cand[off + at];
                  if (C > 1) {
                    for (uint32_t r = 0; r < C; ++r)
                      dsmem_st_u32(dsmem_addr(slot, r), static_cast<uint32_t>(kk[i]));
                  } else {
                    *slot = kk[i];
                  }
                }
              }
            }
          }
          ab = __reduce_add_sync(kFull, ab);
        }
        if (lane == 0) {
          sh.cgt[j * NW + warp] = ab;
          sh.ceq[j * NW + warp] = 0;
        }
        wab += ab;
      }
      if (lane == 0) {
        uint32_t* slot = &sh.wtot[crank][warp];
        if (C > 1) {
          for (uint32_t r = 0; r < C; ++r) dsmem_st_u32(dsmem_addr(slot, r), wab);
        } else {
          *slot = wab;
        }
      }
      row_sync(C);  // the last cluster barrier: nothing is read remotely after it
      // P threads rank each candidate against the whole list (P a power of two,
      // m x P <= NT); the group holding T reports it (all such groups report
      // the same values)
      {
        uint32_t P = 1;
        while (P < 32 && m * P * 2 <= static_cast<uint32_t>(NT)) P *= 2;
        const uint32_t ci = static_cast<uint32_t>(tid) / P, part = static_cast<uint32_t>(tid) % P;
        uint32_t gt = 0, ge = 0;
        int ki = 0;
        if (ci < m) {
          ki = sh.u.c.cand[ci];
          for (uint32_t j = part; j < m; j += P) {
            const int aj = sh.u.c.cand[j];
            gt += aj > ki;
            ge += aj >= ki;
          }
        }
        for (uint32_t o = P >> 1; o > 0; o >>= 1) {
          gt += __shfl_xor_sync(kFull, gt, o);
          ge += __shfl_xor_sync(kFull, ge, o);
        }
        if (ci < m && part == 0 && gt < kr && kr <= ge) {
          const uint32_t nd = kr - gt;
          sh.thr = (nd == ge - gt) ? Threshold{ki - 1, 0u} : Threshold{ki, nd};
        }
      }
      __syncthreads();
      T = sh.thr.T;
      need = sh.thr.need;
      own = min(own, sh.lcount);
      // this CTA's candidates above T, or equal to it, join their chunks' counts
      for (uint32_t p = tid; p < own; p += NT) {
        const int key = sh.u.c.cand[off + p];
        const int ch = sh.u.c.lch[p];
        if (key > T) atomicAdd(&sh.cgt[ch], 1u);
        else if (key == T) atomicAdd(&sh.ceq[ch], 1u);
      }
      __syncthreads();
      if (warp == 0) {
        scan_chunks1<NCH>(sh.cgt, lane);
        if (need) scan_chunks1<NCH>(sh.ceq, lane);
        // the earlier CTAs' kept entries (above bin B, and candidates above T)
        // and their ties
        uint32_t gb = 0, eb = 0;
        for (uint32_t p = lane; p < off; p += 32) {
          const int key = sh.u.c.cand[p];
          gb += key > T;
          eb += key == T;
        }
        for (uint32_t i = lane; i < crank * NW; i += 32) gb += sh.wtot[i / NW][i % NW];
        gb = __reduce_add_sync(kFull, gb);
        eb = __reduce_add_sync(kFull, eb);
        if (lane == 0) {
          sh.before_gt = gb;
          sh.before_eq = eb;
        }
      }
      __syncthreads();
      gt_before = sh.before_gt;
      eq_before = sh.before_eq;
      counted = true;
    } else {
      // ---- too many candidates for the table: integer rounds over the slice --
      int lo = 0x7fffffff, hi = -1;
#pragma unroll 2
      for (int j = 0; j < jv; ++j) {
        const int q = j * NT + tid;
        int kk[4];
        keys4<FULL>(s4[q], 4 * q, nv, kk);
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (kk[i] >= kl && kk[i] <= kh) {
            lo = min(lo, kk[i]);
            hi = max(hi, kk[i]);
          }
      }
      lo = block_min<NT>(lo, sh.red, lane, warp);
      hi = block_max<NT>(hi, sh.red, lane, warp);
      if (C > 1) {
        if (tid == 0) {
          sh.pub_lo = lo;
          sh.pub_hi = hi;
        }
        // also the point after which no CTA reads the packed histograms, whose
        // words the round tables reuse
        cluster_sync();
        for (uint32_t r = 0; r < C; ++r) {
          lo = min(lo, dsmem_ld_s32(dsmem_addr(&sh.pub_lo, r)));
          hi = max(hi, dsmem_ld_s32(dsmem_addr(&sh.pub_hi, r)));
        }
      }
      int p = 0;
      for (;;) {
        if (lo >= hi) {
          T = lo;
          need = kr;
          break;
        }
        const int sft = round_shift(lo, hi);
        for (int i = tid; i < kRoundBins; i += NT) sh.u.rhist[p][i] = 0;
        __syncthreads();
#pragma unroll 2
        for (int j = 0; j < jv; ++j) {
          const int q = j * NT + tid;
          int kk[4];
          keys4<FULL>(s4[q], 4 * q, nv, kk);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (kk[i] >= lo && kk[i] <= hi)
              atomicAdd(&sh.u.rhist[p][static_cast<uint32_t>(kk[i] - lo) >> sft], 1u);
        }
        __syncthreads();
        // the group-sum table alternates from round to round, so a push never
        // lands on sums another CTA may still be reading
        const BinPick q = cluster_pick<NT, kRoundBins>(sh.u.rhist[p], table + p * C * NT, C,
                                                       crank, kr, sh, tid, lane, warp);
        kr -= q.above;
        const int nlo = lo + (q.bin << sft);
        const int nhi = static_cast<int>(
            min(static_cast<uint32_t>(hi), static_cast<uint32_t>(nlo) + ((1u << sft) - 1u)));
        if (q.count == kr) {
          T = nlo - 1;
          need = 0;
          break;
        }
        lo = nlo;
        hi = nhi;
        p ^= 1;
      }
    }
  }

  if (!counted) {
    // ---- count kept entries per 128-entry chunk ------------------------------
#pragma unroll 2
    for (int j = 0; j < QPT; ++j) {
      uint32_t g = 0, e = 0;
      if (j < jv) {
        const int q = j * NT + tid;
        int kk[4];
        keys4<FULL>(s4[q], 4 * q, nv, kk);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          g += kk[i] > T;
          e += kk[i] == T;
        }
        g = __reduce_add_sync(kFull, g);
        e = need ? __reduce_add_sync(kFull, e) : 0u;
      }
      if (lane == 0) {
        sh.cgt[j * NW + warp] = g;
        sh.ceq[j * NW + warp] = e;
      }
    }
    __syncthreads();
    if (warp == 0) {
      const uint32_t tg = scan_chunks1<NCH>(sh.cgt, lane);
      const uint32_t te = scan_chunks1<NCH>(sh.ceq, lane);
      if (C > 1 && lane == 31) {
        // push this slice's totals to every later CTA of the row
        for (uint32_t r = crank + 1; r < C; ++r) {
          dsmem_st_u32(dsmem_addr(&sh.tot_gt[crank], r), tg);
          dsmem_st_u32(dsmem_addr(&sh.tot_eq[crank], r), te);
        }
      }
    }
    row_sync(C);  // the last cluster barrier: nothing is read remotely after it
    for (uint32_t r = 0; r < crank; ++r) {
      gt_before += sh.tot_gt[r];
      eq_before += sh.tot_eq[r];
    }
  }

  // ---- write the payload (ascending column) and the buffers -----------------
  pdl_end();
  float* vrow = a.vals + row * k;
  int32_t* irow = a.idx + row * k;
  const uint32_t kk32 = static_cast<uint32_t>(min64(k, 0x7fffffff));
  const unsigned lt = lanemask_lt();
#pragma unroll 1
  for (int j = 0; j < jv; ++j) {
    const int q = j * NT + tid;
    const float4 v4 = s4[q];
    int kk[4];
    keys4<FULL>(v4, 4 * q, nv, kk);
    const int ch = j * NW + warp;
    const uint32_t eqt = eq_before + sh.ceq[ch];
    uint32_t pos = gt_before + sh.cgt[ch] + min(need, eqt);
    bool kp[4];
    if (need) {
      uint32_t r = eqt;
#pragma unroll
      for (int i = 0; i < 4; ++i) r += __popc(__ballot_sync(kFull, kk[i] == T) & lt);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const bool e = kk[i] == T;
        kp[i] = kk[i] > T || (e && r < need);
        r += e;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) kp[i] = kk[i] > T;
    }
    // this lane's first position among the chunk's kept entries, and their count
    uint32_t pre = 0, tot = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const unsigned b = __ballot_sync(kFull, kp[i]);
      pre += __popc(b & lt);
      tot += __popc(b);
    }
    const int e0 = 4 * q;
    const float val[4] = {v4.x, v4.y, v4.z, v4.w};
    const int col = static_cast<int>(c0) + e0;
    // The column offsets of the kept entries are staged in column order, then
    // the entries are read back from the chunk's slots and written out with
    // coalesced stores.
    const float* sval = reinterpret_cast<const float*>(s4 + j * NT + warp * 32);
    uint8_t* soff = sh.woff[warp];
    __syncwarp();
    {
      uint32_t r = pre;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (kp[i]) soff[r] = static_cast<uint8_t>(4 * lane + i);
        r += kp[i] ? 1u : 0u;
      }
    }
    __syncwarp();
    {
      // at most 128 kept entries a chunk: up to four warp-wide rounds, the
      // later ones only when the chunk keeps that many
      const int colbase = static_cast<int>(c0) + 4 * (j * NT + warp * 32);
      const uint32_t lim = min(tot, kk32 > pos ? kk32 - pos : 0u);
      float* vdst = vrow + pos;
      int32_t* idst = irow + pos;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (32u * u < lim) {
          const uint32_t t = 32u * u + lane;
          if (t < lim) {
            const uint32_t o = soff[t];
            vdst[t] = sval[o];
            idst[t] = colbase + static_cast<int>(o);
          }
        }
      }
    }
    if (MODE == kDelta) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (kp[i]) {
          // state + d, against the same state value d was formed from
          float* sp = arow + col + i;
          *sp = fadd(*sp, val[i]);
        }
    }
    if (MODE == kEF) {
      const float ne[4] = {kp[0] ? 0.0f : val[0], kp[1] ? 0.0f : val[1], kp[2] ? 0.0f : val[2],
                           kp[3] ? 0.0f : val[3]};
      if (a.aligned && (FULL || e0 + 4 <= nv)) {
        *reinterpret_cast<float4*>(arow + col) = make_float4(ne[0], ne[1], ne[2], ne[3]);
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (e0 + i < nv) arow[col + i] = ne[i];
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Warp-per-row kernel (rows of at most 128 * NVW entries, WPC warps per CTA)
// ---------------------------------------------------------------------------
struct WarpShared {
  union {
    struct {
      uint32_t hist[kRoundBins + 64];  // + 32 zero spill counters, + 32 past-the-end ones
      int lkey[kLCAPW];
    } sel;
    uint2 out[(kRoundBins + 64 + kLCAPW) / 2];  // the write stage: (value, column) pairs
  } u;
  uint32_t lcount;
  uint64_t bar[2];
};

// w |= bit when key > t: one compare and one predicated OR.
__device__ __forceinline__ void or_if_key_gt(uint32_t& w, int key, int t, uint32_t bit) {
  asm("{\n .reg .pred p;\n setp.gt.s32 p, %1, %2;\n @p or.b32 %0, %0, %3;\n}" : "+r"(w) : "r"(key), "r"(t), "r"(bit));
}

// Row of the error / state buffer for a logical row (nullptr for plain TopK);
// *ok = false for an AQ-SGD sample id out of range.
template <int MODE>
__device__ __forceinline__ float* state_row(const TopkRowArgs& a, int64_t row, bool* ok) {
  *ok = true;
  if (MODE == kPlain) return nullptr;
  int64_t srow = row;
  if (MODE == kDelta && a.ids != nullptr) {
    const int64_t sid = a.ids[row / a.rps];
    if (sid < 0 || sid >= a.num_samples) {
      *ok = false;
      return nullptr;
    }
    srow = sid * a.rps + row % a.rps;
  }
  return a.aux + srow * a.L;
}

// Rows staged per row buffer of the warp kernel: x, plus the err / state row
// except for rows of 513..768 entries (NVW 6), where that row is read through
// L2 (measured: with it staged one CTA fits an SM and the kernel runs ~25 %
// slower; for other lengths the staged row is faster).
__host__ __device__ constexpr int warp_row_buffers(int mode, int nvw) { return (mode == kPlain || nvw == 6) ? 1 : 2; }

// Warps per CTA: eight, four when a warp's two row buffers exceed 12 KiB.
__host__ __device__ constexpr int warp_wpc(int mode, int nvw) {
  return 2 * 128 * nvw * 4 * warp_row_buffers(mode, nvw) > 12 * 1024 ? 4 : 8;
}

// CTAs per SM the registers are held to: as many as the shared memory admits
// (row buffers and WarpShared), at most four; two for the fused variants on
// rows of 513..768 entries, which hold 24 ranked values a thread (measured: at
// three they spill and run ~5 % slower).
__host__ __device__ constexpr int warp_min_blocks(int mode, int nvw) {
  return (nvw == 6 && mode != kPlain) ? 2 : 227 * 1024 / (warp_wpc(mode, nvw) * (2 * 128 * nvw * 4 * warp_row_buffers(mode, nvw) +
                                              static_cast<int>(sizeof(WarpShared)))) < 4
             ? 227 * 1024 / (warp_wpc(mode, nvw) * (2 * 128 * nvw * 4 * warp_row_buffers(mode, nvw) +
                                                    static_cast<int>(sizeof(WarpShared))))
             : 4;
}

template <int MODE, int NVW, int WPC, bool FULL>
__global__ void __launch_bounds__(32 * WPC, warp_min_blocks(MODE, NVW)) topk_warp_kernel(const TopkRowArgs a) {
  pdl_begin();
  constexpr int RCAP = 128 * NVW;
  // x, and the err / state row, are staged per row in the warp's buffers;
  // rows of 513..768 entries instead prefetch the err / state row into L2 and
  // read it from there: staged, it would leave room for one CTA per SM
  constexpr int NBUF = warp_row_buffers(MODE, NVW);
  __shared__ WarpShared wsh[WPC];
  extern __shared__ __align__(16) float dyn[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  WarpShared& sh = wsh[warp];
  float* wbase = dyn + warp * (2 * RCAP * NBUF);  // two row buffers (double buffering)
  const int64_t L = a.L;
  const int64_t k = a.k;
  const int n = static_cast<int>(L);
  const unsigned lt = lanemask_lt();
  const int64_t stride = static_cast<int64_t>(gridDim.x) * WPC;
  const uint32_t bytes = static_cast<uint32_t>(n) * 4u;

  if (a.aligned && lane == 0) {
    mbar_init(&sh.bar[0], 1);
    mbar_init(&sh.bar[1], 1);
    fence_mbar_init();
  }
  __syncwarp();

  // Start the bulk copies of one row into buffer b; returns false (and does
  // nothing) for a row whose sample id is out of range.
  auto issue = [&](int64_t r, int b) -> bool {
    bool ok;
    float* ar = state_row<MODE>(a, r, &ok);
    if (!ok) return false;
    if (lane == 0) {
      float* buf = wbase + b * (RCAP * NBUF);
      fence_proxy_async_smem();
      mbar_arrive_expect_tx(&sh.bar[b], bytes * NBUF);
      bulk_g2s(buf, a.x + r * L, bytes, &sh.bar[b]);
      if (MODE != kPlain) {
        if (NBUF == 2) bulk_g2s(buf + RCAP, ar, bytes, &sh.bar[b]);
        else bulk_prefetch_l2(ar, bytes);
      }
    }
    return true;
  };

  int64_t row = static_cast<int64_t>(blockIdx.x) * WPC + warp;
  uint32_t phases = 0u;  // bit b: parity of buffer b's next phase
  uint32_t live = 0u;    // bit b: a copy into buffer b is in flight
  int b = 0;
  if (a.aligned && row < a.rows && issue(row, 0)) live |= 1u;
  for (; row < a.rows; row += stride, b ^= 1) {
    const int64_t next = row + stride;
    if (a.aligned && next < a.rows) {
      if (issue(next, b ^ 1)) live |= 2u >> b;
      else live &= ~(2u >> b);
    }
    bool ok;
    float* arow = state_row<MODE>(a, row, &ok);
    if (!ok) {
      if (lane == 0) set_status(a.status, STATUS_BAD_SAMPLE);
      continue;
    }
    float* xs = wbase + b * (RCAP * NBUF);
    if (a.aligned) {
      const uint32_t par = (phases >> b) & 1u;
      const bool got = mbar_wait_bounded(&sh.bar[b], par, a.spin_limit, a.status);
      if (__any_sync(kFull, !got)) {
        // give up on the remaining rows; drain the copies this warp started
        mbar_wait_bounded(&sh.bar[b], par, kDrainPolls, nullptr);
        if (next < a.rows && ((live >> (b ^ 1)) & 1u))
          mbar_wait_bounded(&sh.bar[b ^ 1], (phases >> (b ^ 1)) & 1u, kDrainPolls, nullptr);
        break;
      }
      phases ^= 1u << b;
    } else {
      const float* xrow = a.x + row * L;
      for (int e = lane; e < n; e += 32) {
        xs[e] = xrow[e];
        if (MODE != kPlain && NBUF == 2) xs[RCAP + e] = arow[e];
      }
      __syncwarp();
    }
    float4* x4 = reinterpret_cast<float4*>(xs);
    // the err / state entries 4q..4q+3 of this row (+0 past its end), from the
    // staged copy or through L2
    auto aux4 = [&](int q) -> float4 {
      if (NBUF == 2) return reinterpret_cast<const float4*>(xs + RCAP)[q];
      const int e0 = 4 * q;
      if (a.aligned && (FULL || e0 + 4 <= n)) return *reinterpret_cast<const float4*>(arow + e0);
      float t[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) t[i] = (e0 + i < n) ? arow[e0 + i] : 0.0f;
      return make_float4(t[0], t[1], t[2], t[3]);
    };

    // ---- ranked values and their keys; the largest key --------------------------
    // Plain TopK holds the keys in registers and reads the values again from the
    // row buffer; the fused variants hold the ranked values (x + err, x - state)
    // and derive the keys.
    constexpr bool kHoldKeys = MODE == kPlain;
    int kv[kHoldKeys ? NVW : 1][4];
    float4 sv[kHoldKeys ? 1 : NVW];
    auto keys_of = [&](int v, int kk[4]) {
      if constexpr (kHoldKeys) {
#pragma unroll
        for (int i = 0; i < 4; ++i) kk[i] = kv[v][i];
      } else {
        keys4<FULL>(sv[v], 4 * (v * 32 + lane), n, kk);
      }
    };
    auto value_of = [&](int v) -> float4 {
      if constexpr (kHoldKeys) return x4[v * 32 + lane];
      else return sv[v];
    };
    int kall = -1;
#pragma unroll
    for (int v = 0; v < NVW; ++v) {
      const int q = v * 32 + lane;
      int kk[4];
      if constexpr (kHoldKeys) {
        keys4<FULL>(x4[q], 4 * q, n, kv[v]);
#pragma unroll
        for (int i = 0; i < 4; ++i) kk[i] = kv[v][i];
      } else {
        sv[v] = ranked4<MODE>(x4[q], aux4(q));
        keys4<FULL>(sv[v], 4 * q, n, kk);
      }
      kall = max(kall, max(max(kk[0], kk[1]), max(kk[2], kk[3])));
    }
    kall = __reduce_max_sync(kFull, kall);
    // the bin scale comes from the largest finite magnitude (TopK marks entries
    // with +inf); a row with a NaN (outside the finite-input contract) takes the
    // integer rounds
    int kmax = kall;
    if (kall >= 0x7f800000) {
      kmax = -1;
#pragma unroll
      for (int v = 0; v < NVW; ++v) {
        int kk[4];
        keys_of(v, kk);
        kmax = max(kmax, max(max(finite_key(kk[0]), finite_key(kk[1])),
                             max(finite_key(kk[2]), finite_key(kk[3]))));
      }
      kmax = __reduce_max_sync(kFull, kmax);
      if (kall > 0x7f800000) kmax = 0;
    }

    // ---- select ---------------------------------------------------------------
    Threshold t;
    if (k >= L) {
      t.T = -1;
      t.need = 0;
    } else {
      const float scale = bucket_scale(kmax, kRoundBins);
      uint32_t kr = static_cast<uint32_t>(k);
      int B = 0;
      uint32_t m = static_cast<uint32_t>(n);  // with scale 0 every entry is a candidate
      if (scale > 0.0f) {
#pragma unroll
        for (int j = 0; j < 8; ++j) sh.u.sel.hist[lane * 8 + j] = 0;
        sh.u.sel.hist[kRoundBins + lane] = 0;
        sh.u.sel.hist[kRoundBins + 32 + lane] = 0;
        if (lane == 0) sh.lcount = 0;
        __syncwarp();
#pragma unroll
        for (int v = 0; v < NVW; ++v) {
          const int q = v * 32 + lane;
          int kk[4];
          keys_of(v, kk);
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            // one atomic per entry and no branch: zeros to this lane's spill
            // counter (folded into bin 0 below), past-the-end slots to another
            const int b = bucket_of(kk[i], scale, kRoundBins);
            const int slot = kk[i] > 0 ? b
                                       : ((FULL || kk[i] == 0) ? kRoundBins + lane
                                                               : kRoundBins + 32 + lane);
            atomicAdd(&sh.u.sel.hist[slot], 1u);
          }
        }
        __syncwarp();
        const uint32_t zc = __reduce_add_sync(kFull, sh.u.sel.hist[kRoundBins + lane]);
        if (lane == 0) sh.u.sel.hist[0] += zc;
        __syncwarp();
        const BinPick p = warp_pick_bin(sh.u.sel.hist, kr, lane);
        __syncwarp();
        B = p.bin;
        kr -= p.above;
        m = p.count;
      }
      if (scale > 0.0f && m <= static_cast<uint32_t>(kLCAPW)) {
        // the candidates are the m entries in bin B, appended where they occur
#pragma unroll
        for (int v = 0; v < NVW; ++v) {
          const int q = v * 32 + lane;
          int kk[4];
          keys_of(v, kk);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if ((FULL || kk[i] >= 0) && bucket_of(kk[i], scale, kRoundBins) == B) {
              const uint32_t at = atomicAdd(&sh.lcount, 1u);
              if (at < kLCAPW) sh.u.sel.lkey[at] = kk[i];
            }
        }
        __syncwarp();
        t = warp_select(sh.u.sel.lkey, min(sh.lcount, static_cast<uint32_t>(kLCAPW)), kr, sh.u.sel.hist, lane);
      } else {
        int lo = 0x7fffffff, hi = -1;
#pragma unroll
        for (int v = 0; v < NVW; ++v) {
          const int q = v * 32 + lane;
          int kk[4];
          keys_of(v, kk);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (kk[i] >= 0 && (scale == 0.0f || bucket_of(kk[i], scale, kRoundBins) == B)) {
              lo = min(lo, kk[i]);
              hi = max(hi, kk[i]);
            }
        }
        lo = __reduce_min_sync(kFull, lo);
        hi = __reduce_max_sync(kFull, hi);
        for (;;) {
          if (lo >= hi) {
            t.T = lo;
            t.need = kr;
            break;
          }
          const int sft = round_shift(lo, hi);
#pragma unroll
          for (int j = 0; j < 8; ++j) sh.u.sel.hist[lane * 8 + j] = 0;
          __syncwarp();
#pragma unroll
          for (int v = 0; v < NVW; ++v) {
            const int q = v * 32 + lane;
            int kk[4];
            keys_of(v, kk);
#pragma unroll
            for (int i = 0; i < 4; ++i)
              if (kk[i] >= lo && kk[i] <= hi)
                atomicAdd(&sh.u.sel.hist[static_cast<uint32_t>(kk[i] - lo) >> sft], 1u);
          }
          __syncwarp();
          const BinPick q = warp_pick_bin(sh.u.sel.hist, kr, lane);
          __syncwarp();
          kr -= q.above;
          const int nlo = lo + (q.bin << sft);
          const int nhi = static_cast<int>(
              min(static_cast<uint32_t>(hi), static_cast<uint32_t>(nlo) + ((1u << sft) - 1u)));
          if (q.count == kr) {
            t.T = nlo - 1;
            t.need = 0;
            break;
          }
          lo = nlo;
          hi = nhi;
        }
      }
    }
    const int T = t.T;
    const uint32_t need = t.need;

    // ---- write (one pass: the warp owns the whole row) ------------------------
    // kept entries: bit 4v + i of km for entry 4 (32 v + lane) + i
    uint32_t km = 0;
#pragma unroll
    for (int v = 0; v < NVW; ++v) {
      int kk[4];
      keys_of(v, kk);
#pragma unroll
      for (int i = 0; i < 4; ++i) or_if_key_gt(km, kk[i], T, 1u << (4 * v + i));
    }
    if (need) {
      // the first `need` entries with key T, in index order
      uint32_t seen = 0;
#pragma unroll
      for (int v = 0; v < NVW; ++v) {
        int kk[4];
        keys_of(v, kk);
        uint32_t em = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) em |= static_cast<uint32_t>(kk[i] == T) << i;
        const uint32_t c = __popc(em);
        const uint32_t inc = warp_inclusive_scan(c, lane);
        uint32_t r = seen + inc - c;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if ((em >> i) & 1u) {
            if (r < need) km |= 1u << (4 * v + i);
            ++r;
          }
        seen += __shfl_sync(kFull, inc, 31);
      }
    }
    float* vrow = a.vals + row * k;
    int32_t* irow = a.idx + row * k;
    // The kept entries of two groups at a time go to the warp's write stage (the
    // selection's scratch, free again) in index order, then out with coalesced
    // stores.
    auto fld = [](uint32_t w, int j) { return (w >> (8 * j)) & 0xffu; };
    const uint32_t out_s = static_cast<uint32_t>(__cvta_generic_to_shared(sh.u.out));
    uint32_t pos = 0;  // entries kept by the groups before
    __syncwarp();      // every lane is done with the selection's scratch
#pragma unroll
    for (int v0 = 0; v0 < NVW; v0 += 4) {
      // this lane's kept counts of four groups, a byte each (a group keeps at
      // most 128 entries of the warp): one scan gives all four offsets
      uint32_t pc = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (v0 + j < NVW) pc |= static_cast<uint32_t>(__popc((km >> (4 * (v0 + j))) & 0xfu)) << (8 * j);
      const uint32_t inc = warp_inclusive_scan(pc, lane);
      const uint32_t tot = __shfl_sync(kFull, inc, 31);
      const uint32_t exc = inc - pc;
#pragma unroll
      for (int j = 0; j < 4 && v0 + j < NVW; j += 2) {  // NVW is even
        const int va = v0 + j;
        const uint32_t ta = fld(tot, j), tr = ta + fld(tot, j + 1);
        uint32_t at = out_s + 8u * fld(exc, j);
        stage_kept4((km >> (4 * va)) & 0xfu, at, value_of(va), 4 * (va * 32 + lane));
        at = out_s + 8u * (ta + fld(exc, j + 1));
        stage_kept4((km >> (4 * (va + 1))) & 0xfu, at, value_of((va + 1)), 4 * ((va + 1) * 32 + lane));
        __syncwarp();
        const uint32_t lim = pos < static_cast<uint64_t>(k)
                                 ? static_cast<uint32_t>(min(static_cast<int64_t>(tr), k - pos))
                                 : 0u;
        float* vp = vrow + pos;
        int32_t* ip = irow + pos;
        for (uint32_t i = lane; i < lim; i += 32) {
          const uint2 e = sh.u.out[i];
          vp[i] = __uint_as_float(e.x);
          ip[i] = static_cast<int32_t>(e.y);
        }
        __syncwarp();
        pos += tr;
      }
    }
    if (MODE != kPlain) {
#pragma unroll
      for (int v = 0; v < NVW; ++v) {
        const int q = v * 32 + lane;
        const int e0 = 4 * q;
        const uint32_t nib = (km >> (4 * v)) & 0xfu;
        if (FULL || e0 < n) {
          const float4 s4 = value_of(v);
          const float val[4] = {s4.x, s4.y, s4.z, s4.w};
          if (MODE == kDelta && nib != 0) {  // state + d where kept
            const float4 g = aux4(q);
            const float st[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
              if ((nib >> i) & 1u) arow[e0 + i] = fadd(st[i], val[i]);
          }
          if (MODE == kEF) {  // err' = s - C(s): +0 where kept
            const float ne[4] = {(nib & 1u) ? 0.0f : val[0], (nib & 2u) ? 0.0f : val[1],
                                 (nib & 4u) ? 0.0f : val[2], (nib & 8u) ? 0.0f : val[3]};
            if (a.aligned && (FULL || e0 + 4 <= n)) {
              *reinterpret_cast<float4*>(arow + e0) = make_float4(ne[0], ne[1], ne[2], ne[3]);
            } else {
#pragma unroll
              for (int i = 0; i < 4; ++i)
                if (e0 + i < n) arow[e0 + i] = ne[i];
            }
          }
        }
      }
    }
    __syncwarp();  // this buffer is free for the bulk copy of a later row
  }
}

// ---------------------------------------------------------------------------
// Host-side launch
// ---------------------------------------------------------------------------
template <int MODE, int NVW, bool FULL>
cudaError_t run_warp(const TopkRowArgs& a, int num_sms, cudaStream_t s) {
  constexpr int NBUF = warp_row_buffers(MODE, NVW);
  constexpr int WBYTES = 2 * 128 * NVW * 4 * NBUF;
  constexpr int WPC = warp_wpc(MODE, NVW);
  auto kernel = topk_warp_kernel<MODE, NVW, WPC, FULL>;
  const int smem = WPC * WBYTES;
  cudaError_t err = ensure_dynamic_smem(kernel, smem);
  if (err != cudaSuccess) return err;
  const int occ = resident_blocks(kernel, 32 * WPC, smem);
  const int64_t want = (a.rows + WPC - 1) / WPC;
  const int64_t cap = static_cast<int64_t>(num_sms) * occ;
  const int blocks = static_cast<int>(want < cap ? want : cap);
  return launch_kernel(kernel, dim3(blocks), dim3(32 * WPC), smem, s, 0u, a);
}

template <int MODE, int NVW>
cudaError_t run_warp_any(const TopkRowArgs& a, int num_sms, cudaStream_t s) {
  if (a.L == 128 * NVW) return run_warp<MODE, NVW, true>(a, num_sms, s);
  return run_warp<MODE, NVW, false>(a, num_sms, s);
}

template <int MODE, int NT, int SCAP, bool FULL>
cudaError_t run_cta(const TopkRowArgs& a, int C, cudaStream_t s) {
  auto kernel = topk_cta_kernel<MODE, NT, SCAP, FULL>;
  const int smem = cta_smem_bytes(NT, SCAP, C);
  cudaError_t err = ensure_dynamic_smem(kernel, cta_smem_bytes(NT, SCAP, NT >= 512 ? 1 : kMaxCluster));
  if (err != cudaSuccess) return err;
  return launch_kernel(kernel, dim3(static_cast<unsigned>(a.rows * C)), dim3(NT), smem, s,
                       static_cast<unsigned>(C), a);
}

// FULL when every CTA's slice is a whole number of NT x 4-entry slots.
template <int MODE, int NT, int SCAP>
cudaError_t run_cta_any(const TopkRowArgs& a, int C, cudaStream_t s) {
  const bool full = (a.slice % (4 * NT) == 0) && (a.slice * C == a.L);
  if (full) return run_cta<MODE, NT, SCAP, true>(a, C, s);
  return run_cta<MODE, NT, SCAP, false>(a, C, s);
}

template <int MODE>
cudaError_t run_mode(const TopkRowArgs& a0, int num_sms, cudaStream_t s) {
  TopkRowArgs a = a0;
  const int64_t L = a.L;
  if (L <= 256) return run_warp_any<MODE, 2>(a, num_sms, s);
  if (L <= 512) return run_warp_any<MODE, 4>(a, num_sms, s);
  if (L <= 768) return run_warp_any<MODE, 6>(a, num_sms, s);
  if (L <= 1024) return run_warp_any<MODE, 8>(a, num_sms, s);
  // Rows of 1025..8192 entries take the band kernel (topk_band.cuh) unless the
  // knob keeps the kernels below.
  if (a.band && band::fits(L)) return band::run_mode<MODE>(a, s);
  // Aligned rows of 8193..65536 entries: one 512-thread CTA per row reading the
  // row twice, the second time from L2 (topk_lrow.cuh), unless the knob keeps
  // the kernels below.
  if (a.band && a.wide_cta && lrow::fits(a)) return lrow::run_mode<MODE>(a, s);
  // One CTA of 128 threads for rows up to 4096 entries, else clusters of
  // 256-thread CTAs holding up to 8192 entries each, split further (slices of
  // at least 2048 entries) while the grid has fewer than 2 CTAs per SM.
  if (L <= 2048) {
    a.slice = (L + 3) / 4 * 4;
    return run_cta_any<MODE, 128, 2048>(a, 1, s);
  }
  if (L <= 4096) {
    a.slice = (L + 3) / 4 * 4;
    return run_cta_any<MODE, 128, 4096>(a, 1, s);
  }
  // Rows up to 32768 entries take one wide CTA each (512 threads and 2 CTAs
  // per SM up to 16384, else 1024 threads and one CTA per SM) when that fills
  // most of the GPU in a single wave: no cluster barriers on the way.  With
  // more rows the smaller clustered CTAs of several waves pack better.
  if (a.wide_cta && L > 8192 && L <= 16384 && a.rows >= num_sms && a.rows <= 2 * num_sms) {
    a.slice = (L + 3) / 4 * 4;
    return run_cta_any<MODE, 512, 16384>(a, 1, s);
  }
  if (a.wide_cta && L > 8192 && L <= 32768 && 4 * a.rows >= 3 * num_sms && a.rows <= num_sms) {
    a.slice = (L + 3) / 4 * 4;
    return run_cta_any<MODE, 1024, 32768>(a, 1, s);
  }
  int64_t C = (L + 8191) / 8192;
  while (a.rows * C < 2 * num_sms && 2 * C <= kMaxCluster && L / (2 * C) >= 2048) C *= 2;
  if (C > kMaxCluster) return cudaErrorInvalidValue;
  a.slice = ((L + C - 1) / C + 3) / 4 * 4;
  return run_cta_any<MODE, 256, 8192>(a, static_cast<int>(C), s);
}

}  // namespace rows
}  // namespace mpc
