// topk_rows.cu -- exact per-row TopK (§2.3) for rows that fit on chip, fused
// with error feedback (§2.4, Seide et al.) and with the EF21 / AQ-SGD buffer
// update (§2.4, §2.5).
//
// Two kernels share the selection of select.cuh:
//  * topk_cta_kernel: one thread-block cluster of C CTAs per row.  Each CTA
//    stages its slice of the row (and of the error or state row) in shared
//    memory with one bulk asynchronous copy completing on an mbarrier, keeps
//    the magnitude keys in registers, and merges its histograms with the other
//    CTAs of the cluster through distributed shared memory.
//  * topk_warp_kernel: one warp per row for rows of at most 2048 entries;
//    each warp stages its row with its own bulk copy and mbarrier and walks
//    the rows of a persistent grid.
// Both read x (and err / state) from HBM once, write the payload once and,
// for error feedback, write err once; the EF21 / AQ-SGD state is written
// only at the kept entries.
#include "common.cuh"
#include "kernels.h"
#include "launch_util.h"
#include "select.cuh"

namespace mpc {

namespace {

constexpr int kNB = 2048;     // bins of the first histogram, CTA kernel
constexpr int kLCAP = 512;    // candidate keys gathered per cluster, CTA kernel
constexpr int kLCAPW = 256;   // candidate keys per warp, warp kernel
constexpr int kWPC = 8;       // warps per CTA, warp kernel

// The value that the selection ranks, for each fused variant.
template <int MODE>
__device__ __forceinline__ float ranked_value(float x, float a) {
  if (MODE == kEF) return fadd(x, a);    // s = x + err
  if (MODE == kDelta) return fsub(x, a); // d = x - state
  return x;
}

// ---------------------------------------------------------------------------
// Block-level reductions and scans (NT threads, NT/32 warps).
// ---------------------------------------------------------------------------
template <int NT>
__device__ __forceinline__ int block_max(int v, int* red, int lane, int warp) {
  v = __reduce_max_sync(kFull, v);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  int r = red[0];
#pragma unroll
  for (int i = 1; i < NT / 32; ++i) r = max(r, red[i]);
  __syncthreads();
  return r;
}

template <int NT>
__device__ __forceinline__ int block_min(int v, int* red, int lane, int warp) {
  v = __reduce_min_sync(kFull, v);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  int r = red[0];
#pragma unroll
  for (int i = 1; i < NT / 32; ++i) r = min(r, red[i]);
  __syncthreads();
  return r;
}

template <int NT>
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* red, int lane, int warp) {
  uint32_t inc = warp_inclusive_scan(v, lane);
  if (lane == 31) red[warp] = inc;
  __syncthreads();
  uint32_t base = 0;
#pragma unroll
  for (int i = 0; i < NT / 32; ++i)
    if (i < warp) base += red[i];
  __syncthreads();
  return base + inc - v;
}

// ---------------------------------------------------------------------------
// CTA / cluster kernel
// ---------------------------------------------------------------------------
template <int NT, int NV>
struct CtaShared {
  static constexpr int NW = NT / 32;
  static constexpr int NCH = NV * NW;  // chunks of 128 consecutive entries
  uint32_t hist[kNB];
  uint32_t rhist[2][kRoundBins];
  int lkey[kLCAP];
  int gkey[kLCAP];
  uint32_t cgt[NCH];
  uint32_t ceq[NCH];
  int red[NW];
  uint32_t ured[NW];
  // published to the other CTAs of the cluster (each written once per launch)
  int pub_max, pub_lo, pub_hi;
  uint32_t pub_lc, pub_gt, pub_eq;
  // block-wide broadcasts
  BinPick pick;
  Threshold thr;
  uint32_t lcount;
  uint64_t bar;
};

// Among NBINS bins ranked high to low, summed over the cluster's C CTAs,
// find the bin holding the kr-th element; result in sh.pick.
template <int NT, int NBINS, class Sh>
__device__ __forceinline__ BinPick cta_pick_bin(const uint32_t* hist, uint32_t C, uint32_t kr,
                                                Sh& sh, int tid, int lane, int warp) {
  constexpr int G = (NBINS + NT - 1) / NT;
  uint32_t c[G];
  uint32_t tsum = 0;
#pragma unroll
  for (int j = 0; j < G; ++j) {
    const int slot = tid * G + j;
    uint32_t cnt = 0;
    if (slot < NBINS) {
      const uint32_t* p = &hist[NBINS - 1 - slot];
      if (C == 1) {
        cnt = *p;
      } else {
        for (uint32_t r = 0; r < C; ++r) cnt += dsmem_ld_u32(dsmem_addr(p, r));
      }
    }
    c[j] = cnt;
    tsum += cnt;
  }
  if (tid == 0) sh.pick = BinPick{0, 0, 0};
  uint32_t excl = block_excl_scan<NT>(tsum, sh.ured, lane, warp);
  if (excl < kr && kr <= excl + tsum) {
    uint32_t run = excl;
#pragma unroll
    for (int j = 0; j < G; ++j) {
      if (run + c[j] >= kr) {
        sh.pick = BinPick{NBINS - 1 - (tid * G + j), run, c[j]};
        break;
      }
      run += c[j];
    }
  }
  __syncthreads();
  return sh.pick;
}

template <int MODE, int NT, int NV>
__global__ void __launch_bounds__(NT) topk_cta_kernel(const TopkRowArgs a) {
  constexpr int NW = NT / 32;
  constexpr int NCH = NV * NW;
  constexpr int SCAP = 4 * NT * NV;
  using Sh = CtaShared<NT, NV>;
  __shared__ Sh sh;
  extern __shared__ __align__(16) float dyn[];
  float* sx = dyn;
  float* sa = dyn + SCAP;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t C = cluster_size();
  const uint32_t crank = cluster_rank();
  const int64_t row = blockIdx.x / C;
  const int64_t L = a.L;
  const int64_t k = a.k;
  const int64_t c0 = static_cast<int64_t>(crank) * a.slice;
  const int n = static_cast<int>(max64(0, min64(a.slice, L - c0)));

  // Row of the error (EF) or state (EF21 / AQ-SGD) buffer.  The decision to
  // skip a row is the same in every CTA of the cluster, so all of them leave
  // together before the first cluster barrier.
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

  // ---- stage the slice in shared memory (one HBM read) ---------------------
  bool failed = false;
  if (a.aligned) {
    if (tid == 0) {
      mbar_init(&sh.bar, 1);
      fence_mbar_init();
    }
    __syncthreads();
    if (n > 0) {
      if (tid == 0) {
        const uint32_t bytes = static_cast<uint32_t>(n) * 4u;
        mbar_arrive_expect_tx(&sh.bar, MODE == kPlain ? bytes : 2u * bytes);
        bulk_g2s(sx, xrow + c0, bytes, &sh.bar);
        if (MODE != kPlain) bulk_g2s(sa, arow + c0, bytes, &sh.bar);
      }
      if (!mbar_wait_bounded(&sh.bar, 0, a.spin_limit, a.status)) {
        mbar_wait_bounded(&sh.bar, 0, kDrainPolls, nullptr);
        failed = true;
      }
    }
    failed = __syncthreads_or(failed);
  } else {
    for (int e = tid; e < n; e += NT) {
      sx[e] = xrow[c0 + e];
      if (MODE != kPlain) sa[e] = arow[c0 + e];
    }
    __syncthreads();
  }
  const int nv = failed ? 0 : n;  // a failed slice takes part as an empty one

  // ---- magnitude keys in registers ------------------------------------------
  int key[NV][4];
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const int q = v * NT + tid;
    const float4 xv = reinterpret_cast<const float4*>(sx)[q];
    float4 av = make_float4(0.f, 0.f, 0.f, 0.f);
    if (MODE != kPlain) av = reinterpret_cast<const float4*>(sa)[q];
    const float xs[4] = {xv.x, xv.y, xv.z, xv.w};
    const float as[4] = {av.x, av.y, av.z, av.w};
#pragma unroll
    for (int i = 0; i < 4; ++i)
      key[v][i] = (4 * q + i < nv) ? mag_key(ranked_value<MODE>(xs[i], as[i])) : -1;
  }

  // ---- select T and need -----------------------------------------------------
  int T;
  uint32_t need;
  if (k >= L) {
    T = -1;
    need = 0;
  } else {
    int kmax = -1;
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
      for (int i = 0; i < 4; ++i) kmax = max(kmax, key[v][i]);
    kmax = block_max<NT>(kmax, sh.red, lane, warp);
    if (C > 1) {
      if (tid == 0) sh.pub_max = kmax;
      cluster_sync();
      for (uint32_t r = 0; r < C; ++r) kmax = max(kmax, dsmem_ld_s32(dsmem_addr(&sh.pub_max, r)));
    }
    const float scale = bucket_scale(kmax, kNB);
    uint32_t kr = static_cast<uint32_t>(k);
    int B = 0;
    uint32_t m;
    if (scale > 0.0f) {
      for (int i = tid; i < kNB; i += NT) sh.hist[i] = 0;
      __syncthreads();
      uint32_t zc = 0;
#pragma unroll
      for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int kk = key[v][i];
          if (kk == 0) ++zc;
          else if (kk > 0) atomicAdd(&sh.hist[bucket_of(kk, scale, kNB)], 1u);
        }
      zc = __reduce_add_sync(kFull, zc);
      if (lane == 0 && zc) atomicAdd(&sh.hist[0], zc);
      if (C > 1) cluster_sync(); else __syncthreads();
      const BinPick p = cta_pick_bin<NT, kNB>(sh.hist, C, kr, sh, tid, lane, warp);
      B = p.bin;
      kr -= p.above;
      m = p.count;
    } else {
      m = static_cast<uint32_t>(L);  // every entry is a candidate
    }
    auto candidate = [&](int kk) {
      return kk >= 0 && (scale == 0.0f || bucket_of(kk, scale, kNB) == B);
    };

    if (m <= static_cast<uint32_t>(kLCAP)) {
      // Gather the candidates' keys and finish on the list (one warp).
      if (tid == 0) sh.lcount = 0;
      __syncthreads();
#pragma unroll
      for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const bool pr = candidate(key[v][i]);
          const unsigned bal = __ballot_sync(kFull, pr);
          if (bal) {
            uint32_t base = 0;
            if (lane == 0) base = atomicAdd(&sh.lcount, static_cast<uint32_t>(__popc(bal)));
            base = __shfl_sync(kFull, base, 0);
            if (pr) sh.lkey[base + __popc(bal & lanemask_lt())] = key[v][i];
          }
        }
      __syncthreads();
      const int* list = sh.lkey;
      uint32_t mt = sh.lcount;
      if (C > 1) {
        if (tid == 0) sh.pub_lc = mt;
        cluster_sync();
        uint32_t off = 0;
        for (uint32_t r = 0; r < C; ++r) {
          const uint32_t lr = dsmem_ld_u32(dsmem_addr(&sh.pub_lc, r));
          const uint32_t base = dsmem_addr(sh.lkey, r);
          for (uint32_t j = tid; j < lr && off + j < kLCAP; j += NT)
            sh.gkey[off + j] = dsmem_ld_s32(base + 4u * j);
          off += lr;
        }
        __syncthreads();
        list = sh.gkey;
        mt = min(off, static_cast<uint32_t>(kLCAP));
      }
      if (warp == 0) {
        const Threshold t = warp_list_select(list, mt, kr, sh.rhist[0], lane);
        if (lane == 0) sh.thr = t;
      }
      __syncthreads();
      T = sh.thr.T;
      need = sh.thr.need;
    } else {
      // Too many candidates for the list: integer rounds over the registers.
      int lo = 0x7fffffff, hi = -1;
#pragma unroll
      for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (candidate(key[v][i])) {
            lo = min(lo, key[v][i]);
            hi = max(hi, key[v][i]);
          }
      lo = block_min<NT>(lo, sh.red, lane, warp);
      hi = block_max<NT>(hi, sh.red, lane, warp);
      if (C > 1) {
        if (tid == 0) {
          sh.pub_lo = lo;
          sh.pub_hi = hi;
        }
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
        const int s = round_shift(lo, hi);
        for (int i = tid; i < kRoundBins; i += NT) sh.rhist[p][i] = 0;
        __syncthreads();
#pragma unroll
        for (int v = 0; v < NV; ++v)
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int kk = key[v][i];
            if (kk >= lo && kk <= hi)
              atomicAdd(&sh.rhist[p][static_cast<uint32_t>(kk - lo) >> s], 1u);
          }
        if (C > 1) cluster_sync(); else __syncthreads();
        const BinPick q = cta_pick_bin<NT, kRoundBins>(sh.rhist[p], C, kr, sh, tid, lane, warp);
        kr -= q.above;
        const int nlo = lo + (q.bin << s);
        const int nhi = static_cast<int>(
            min(static_cast<uint32_t>(hi), static_cast<uint32_t>(nlo) + ((1u << s) - 1u)));
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

  // ---- count kept entries per 128-entry chunk ------------------------------
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    uint32_t g = 0, q = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      g += key[v][i] > T;
      q += key[v][i] == T;
    }
    g = __reduce_add_sync(kFull, g);
    q = need ? __reduce_add_sync(kFull, q) : 0u;
    if (lane == 0) {
      sh.cgt[v * NW + warp] = g;
      sh.ceq[v * NW + warp] = q;
    }
  }
  __syncthreads();
  if (warp == 0) {
    constexpr int PER = (NCH + 31) / 32;
    uint32_t g[PER], q[PER], tg = 0, tq = 0;
#pragma unroll
    for (int j = 0; j < PER; ++j) {
      const int ch = lane * PER + j;
      g[j] = ch < NCH ? sh.cgt[ch] : 0u;
      q[j] = ch < NCH ? sh.ceq[ch] : 0u;
      tg += g[j];
      tq += q[j];
    }
    uint32_t eg = warp_inclusive_scan(tg, lane) - tg;
    uint32_t eq = warp_inclusive_scan(tq, lane) - tq;
#pragma unroll
    for (int j = 0; j < PER; ++j) {
      const int ch = lane * PER + j;
      if (ch < NCH) {
        sh.cgt[ch] = eg;
        sh.ceq[ch] = eq;
      }
      eg += g[j];
      eq += q[j];
    }
    if (lane == 31) {
      sh.pub_gt = eg;
      sh.pub_eq = eq;
    }
  }
  __syncthreads();
  uint32_t gt_before = 0, eq_before = 0;
  if (C > 1) {
    cluster_sync();
    for (uint32_t r = 0; r < crank; ++r) {
      gt_before += dsmem_ld_u32(dsmem_addr(&sh.pub_gt, r));
      eq_before += dsmem_ld_u32(dsmem_addr(&sh.pub_eq, r));
    }
  }

  // ---- write the payload (ascending column) and the buffers -----------------
  const int64_t pbase = row * k;
  const unsigned lt = lanemask_lt();
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const int ch = v * NW + warp;
    const uint32_t eqt = eq_before + sh.ceq[ch];
    uint32_t pos = gt_before + sh.cgt[ch] + min(need, eqt);
    bool kp[4];
    if (need) {
      uint32_t r = eqt;
#pragma unroll
      for (int i = 0; i < 4; ++i) r += __popc(__ballot_sync(kFull, key[v][i] == T) & lt);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const bool e = key[v][i] == T;
        kp[i] = key[v][i] > T || (e && r < need);
        r += e;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) kp[i] = key[v][i] > T;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) pos += __popc(__ballot_sync(kFull, kp[i]) & lt);

    const int q = v * NT + tid;
    const int e0 = 4 * q;
    if (e0 >= nv) continue;
    const float4 xv = reinterpret_cast<const float4*>(sx)[q];
    float4 av = make_float4(0.f, 0.f, 0.f, 0.f);
    if (MODE != kPlain) av = reinterpret_cast<const float4*>(sa)[q];
    const float xs[4] = {xv.x, xv.y, xv.z, xv.w};
    const float as[4] = {av.x, av.y, av.z, av.w};
    float val[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) val[i] = ranked_value<MODE>(xs[i], as[i]);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (kp[i]) {
        if (pos < static_cast<uint64_t>(k)) {
          a.vals[pbase + pos] = val[i];
          a.idx[pbase + pos] = static_cast<int32_t>(c0 + e0 + i);
        }
        if (MODE == kDelta) arow[c0 + e0 + i] = fadd(as[i], val[i]);
        ++pos;
      }
    }
    if (MODE == kEF) {
      float ne[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) ne[i] = kp[i] ? 0.0f : val[i];
      if (a.aligned && e0 + 4 <= nv) {
        *reinterpret_cast<float4*>(arow + c0 + e0) = make_float4(ne[0], ne[1], ne[2], ne[3]);
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (e0 + i < nv) arow[c0 + e0 + i] = ne[i];
      }
    }
  }
  if (C > 1) cluster_sync();  // no CTA leaves while another may read its shared memory
}

// ---------------------------------------------------------------------------
// Warp-per-row kernel (rows of at most 128 * NVW entries)
// ---------------------------------------------------------------------------
struct WarpShared {
  uint32_t hist[kRoundBins];
  int lkey[kLCAPW];
  uint64_t bar;
};

template <int MODE, int NVW>
__global__ void __launch_bounds__(32 * kWPC) topk_warp_kernel(const TopkRowArgs a) {
  constexpr int RCAP = 128 * NVW;
  constexpr int NBUF = (MODE == kPlain) ? 1 : 2;
  __shared__ WarpShared wsh[kWPC];
  extern __shared__ __align__(16) float dyn[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  WarpShared& sh = wsh[warp];
  float* sx = dyn + warp * (RCAP * NBUF);
  float* sa = sx + RCAP;
  const int64_t L = a.L;
  const int64_t k = a.k;
  const int n = static_cast<int>(L);
  const unsigned lt = lanemask_lt();

  if (a.aligned) {
    if (lane == 0) {
      mbar_init(&sh.bar, 1);
      fence_mbar_init();
    }
    __syncwarp();
  }
  uint32_t phase = 0;
  for (int64_t row = static_cast<int64_t>(blockIdx.x) * kWPC + warp; row < a.rows;
       row += static_cast<int64_t>(gridDim.x) * kWPC) {
    float* arow = nullptr;
    if (MODE != kPlain) {
      int64_t srow = row;
      if (MODE == kDelta && a.ids != nullptr) {
        const int64_t sid = a.ids[row / a.rps];
        if (sid < 0 || sid >= a.num_samples) {
          if (lane == 0) set_status(a.status, STATUS_BAD_SAMPLE);
          continue;
        }
        srow = sid * a.rps + row % a.rps;
      }
      arow = a.aux + srow * L;
    }
    const float* xrow = a.x + row * L;

    // ---- stage the row ------------------------------------------------------
    if (a.aligned) {
      if (lane == 0) {
        fence_proxy_async_smem();
        const uint32_t bytes = static_cast<uint32_t>(n) * 4u;
        mbar_arrive_expect_tx(&sh.bar, bytes * NBUF);
        bulk_g2s(sx, xrow, bytes, &sh.bar);
        if (MODE != kPlain) bulk_g2s(sa, arow, bytes, &sh.bar);
      }
      const bool ok = mbar_wait_bounded(&sh.bar, phase, a.spin_limit, a.status);
      if (__any_sync(kFull, !ok)) {
        mbar_wait_bounded(&sh.bar, phase, kDrainPolls, nullptr);
        break;  // leave the remaining rows; the status word reports the timeout
      }
      phase ^= 1u;
    } else {
      for (int e = lane; e < n; e += 32) {
        sx[e] = xrow[e];
        if (MODE != kPlain) sa[e] = arow[e];
      }
      __syncwarp();
    }

    int key[NVW][4];
#pragma unroll
    for (int v = 0; v < NVW; ++v) {
      const int q = v * 32 + lane;
      const float4 xv = reinterpret_cast<const float4*>(sx)[q];
      float4 av = make_float4(0.f, 0.f, 0.f, 0.f);
      if (MODE != kPlain) av = reinterpret_cast<const float4*>(sa)[q];
      const float xs[4] = {xv.x, xv.y, xv.z, xv.w};
      const float as[4] = {av.x, av.y, av.z, av.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
        key[v][i] = (4 * q + i < n) ? mag_key(ranked_value<MODE>(xs[i], as[i])) : -1;
    }

    // ---- select ---------------------------------------------------------------
    Threshold t;
    if (k >= L) {
      t.T = -1;
      t.need = 0;
    } else {
      int kmax = -1;
#pragma unroll
      for (int v = 0; v < NVW; ++v)
#pragma unroll
        for (int i = 0; i < 4; ++i) kmax = max(kmax, key[v][i]);
      kmax = __reduce_max_sync(kFull, kmax);
      const float scale = bucket_scale(kmax, kRoundBins);
      uint32_t kr = static_cast<uint32_t>(k);
      int B = 0;
      uint32_t m;
      if (scale > 0.0f) {
#pragma unroll
        for (int j = 0; j < 8; ++j) sh.hist[lane * 8 + j] = 0;
        __syncwarp();
        uint32_t zc = 0;
#pragma unroll
        for (int v = 0; v < NVW; ++v)
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int kk = key[v][i];
            if (kk == 0) ++zc;
            else if (kk > 0) atomicAdd(&sh.hist[bucket_of(kk, scale, kRoundBins)], 1u);
          }
        zc = __reduce_add_sync(kFull, zc);
        if (lane == 0 && zc) atomicAdd(&sh.hist[0], zc);
        __syncwarp();
        const BinPick p = warp_pick_bin(sh.hist, kr, lane);
        __syncwarp();
        B = p.bin;
        kr -= p.above;
        m = p.count;
      } else {
        m = static_cast<uint32_t>(n);
      }
      auto candidate = [&](int kk) {
        return kk >= 0 && (scale == 0.0f || bucket_of(kk, scale, kRoundBins) == B);
      };
      if (m <= static_cast<uint32_t>(kLCAPW)) {
        uint32_t cnt = 0;
#pragma unroll
        for (int v = 0; v < NVW; ++v)
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const bool pr = candidate(key[v][i]);
            const unsigned bal = __ballot_sync(kFull, pr);
            if (pr) {
              const uint32_t at = cnt + __popc(bal & lt);
              if (at < kLCAPW) sh.lkey[at] = key[v][i];
            }
            cnt += __popc(bal);
          }
        __syncwarp();
        t = warp_list_select(sh.lkey, min(cnt, static_cast<uint32_t>(kLCAPW)), kr, sh.hist, lane);
      } else {
        int lo = 0x7fffffff, hi = -1;
#pragma unroll
        for (int v = 0; v < NVW; ++v)
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (candidate(key[v][i])) {
              lo = min(lo, key[v][i]);
              hi = max(hi, key[v][i]);
            }
        lo = __reduce_min_sync(kFull, lo);
        hi = __reduce_max_sync(kFull, hi);
        for (;;) {
          if (lo >= hi) {
            t.T = lo;
            t.need = kr;
            break;
          }
          const int s = round_shift(lo, hi);
#pragma unroll
          for (int j = 0; j < 8; ++j) sh.hist[lane * 8 + j] = 0;
          __syncwarp();
#pragma unroll
          for (int v = 0; v < NVW; ++v)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int kk = key[v][i];
              if (kk >= lo && kk <= hi)
                atomicAdd(&sh.hist[static_cast<uint32_t>(kk - lo) >> s], 1u);
            }
          __syncwarp();
          const BinPick q = warp_pick_bin(sh.hist, kr, lane);
          __syncwarp();
          kr -= q.above;
          const int nlo = lo + (q.bin << s);
          const int nhi = static_cast<int>(
              min(static_cast<uint32_t>(hi), static_cast<uint32_t>(nlo) + ((1u << s) - 1u)));
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

    // ---- write (one pass: the warp owns the whole row) ----------------------
    const int64_t pbase = row * k;
    uint32_t pos = 0, eq_seen = 0;
#pragma unroll
    for (int v = 0; v < NVW; ++v) {
      bool kp[4];
      uint32_t slot_kept = 0;
      if (need) {
        unsigned be[4];
        uint32_t r = eq_seen;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          be[i] = __ballot_sync(kFull, key[v][i] == T);
          r += __popc(be[i] & lt);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const bool e = key[v][i] == T;
          kp[i] = key[v][i] > T || (e && r < need);
          r += e;
          eq_seen += __popc(be[i]);
        }
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) kp[i] = key[v][i] > T;
      }
      uint32_t p = pos;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const unsigned bk = __ballot_sync(kFull, kp[i]);
        p += __popc(bk & lt);
        slot_kept += __popc(bk);
      }
      const int q = v * 32 + lane;
      const int e0 = 4 * q;
      if (e0 < n) {
        const float4 xv = reinterpret_cast<const float4*>(sx)[q];
        float4 av = make_float4(0.f, 0.f, 0.f, 0.f);
        if (MODE != kPlain) av = reinterpret_cast<const float4*>(sa)[q];
        const float xs[4] = {xv.x, xv.y, xv.z, xv.w};
        const float as[4] = {av.x, av.y, av.z, av.w};
        float val[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) val[i] = ranked_value<MODE>(xs[i], as[i]);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          if (kp[i]) {
            if (p < static_cast<uint64_t>(k)) {
              a.vals[pbase + p] = val[i];
              a.idx[pbase + p] = e0 + i;
            }
            if (MODE == kDelta) arow[e0 + i] = fadd(as[i], val[i]);
            ++p;
          }
        }
        if (MODE == kEF) {
          float ne[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) ne[i] = kp[i] ? 0.0f : val[i];
          if (a.aligned && e0 + 4 <= n) {
            *reinterpret_cast<float4*>(arow + e0) = make_float4(ne[0], ne[1], ne[2], ne[3]);
          } else {
#pragma unroll
            for (int i = 0; i < 4; ++i)
              if (e0 + i < n) arow[e0 + i] = ne[i];
          }
        }
      }
      pos += slot_kept;
    }
    __syncwarp();  // the row's shared memory is free for the next bulk copy
  }
}

// ---------------------------------------------------------------------------
// Host-side launch
// ---------------------------------------------------------------------------
template <int MODE, int NVW>
cudaError_t run_warp(const TopkRowArgs& a, int num_sms, cudaStream_t s) {
  auto kernel = topk_warp_kernel<MODE, NVW>;
  const int smem = kWPC * 128 * NVW * 4 * ((MODE == kPlain) ? 1 : 2);
  cudaError_t err = ensure_dynamic_smem(kernel, smem);
  if (err != cudaSuccess) return err;
  const int occ = resident_blocks(kernel, 32 * kWPC, smem);
  const int64_t want = (a.rows + kWPC - 1) / kWPC;
  const int64_t cap = static_cast<int64_t>(num_sms) * occ;
  const int blocks = static_cast<int>(want < cap ? want : cap);
  kernel<<<blocks, 32 * kWPC, smem, s>>>(a);
  return cudaGetLastError();
}

template <int MODE, int NT, int NV>
cudaError_t run_cta(const TopkRowArgs& a, int C, cudaStream_t s) {
  auto kernel = topk_cta_kernel<MODE, NT, NV>;
  const int smem = 4 * NT * NV * 4 * ((MODE == kPlain) ? 1 : 2);
  cudaError_t err = ensure_dynamic_smem(kernel, smem);
  if (err != cudaSuccess) return err;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(a.rows * C), 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, a);
}

template <int MODE>
cudaError_t run_mode(const TopkRowArgs& a0, int num_sms, cudaStream_t s) {
  TopkRowArgs a = a0;
  const int64_t L = a.L;
  if (L <= 256) return run_warp<MODE, 2>(a, num_sms, s);
  if (L <= 512) return run_warp<MODE, 4>(a, num_sms, s);
  if (L <= 768) return run_warp<MODE, 6>(a, num_sms, s);
  if (L <= 1024) return run_warp<MODE, 8>(a, num_sms, s);
  if (L <= 2048) return run_warp<MODE, 16>(a, num_sms, s);
  const bool small = L <= 4096;
  const int64_t scap = small ? 4096 : 8192;
  int64_t C = (L + scap - 1) / scap;
  // Spread short batches over more CTAs while slices stay >= 2048 entries.
  while (a.rows * C < 2 * num_sms && C < 8 && L / (2 * C) >= 2048) C *= 2;
  if (C > 8) return cudaErrorInvalidValue;
  int64_t slice = (L + C - 1) / C;
  slice = (slice + 3) / 4 * 4;
  a.slice = slice;
  if (small) return run_cta<MODE, 128, 8>(a, static_cast<int>(C), s);
  return run_cta<MODE, 256, 8>(a, static_cast<int>(C), s);
}

}  // namespace

cudaError_t launch_topk_rows(int mode, const TopkRowArgs& a, int num_sms, cudaStream_t s) {
  if (a.rows <= 0) return cudaSuccess;
  switch (mode) {
    case kPlain: return run_mode<kPlain>(a, num_sms, s);
    case kEF: return run_mode<kEF>(a, num_sms, s);
    case kDelta: return run_mode<kDelta>(a, num_sms, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace mpc
