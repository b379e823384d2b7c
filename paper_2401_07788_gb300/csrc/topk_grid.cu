// topk_grid.cu -- exact TopK (§2.3), with error feedback (§2.4) or the EF21
// buffer update (§2.4), for rows longer than one thread-block cluster holds
// (up to whole tensors of 2^31-1 entries).  Multi-pass, with the counters and
// candidates in a caller workspace; one row at a time.
//
// Per row, a fixed sequence of launches (each kernel returns at once when the
// device-side state says its step is not needed, so the host never waits):
//   init     clear the row's counters;
//   sample   bin scale from a strided sample of the ranked values;
//   hist     histogram of all entries over bins linear in |x| (error feedback:
//            s = x + err is written back into err, so later passes read s);
//   pick     the bin that holds the k-th largest entry, as a key range;
//   3 x (hist, pick)  refinement rounds with 2048 bins of equal key width over
//            that range, while it holds more candidates than the list takes;
//   count    per 8192-entry chunk: entries above the range (or, once T is
//            known, above / equal to T); entries inside the range are appended
//            to the candidate list;
//   select   T and `need` from the candidate list; candidates above / equal to
//            T join their chunks' counts;
//   scan     per chunk: kept entries and ties before it;
//   write    the payload in ascending index order, and the buffer updates.
#include "common.cuh"
#include "kernels.h"
#include "select.cuh"

namespace mpc {
namespace {

constexpr int kGT = 256;                 // threads per CTA
constexpr int kGPT = 32;                 // entries per thread per chunk
constexpr int64_t kCH = kGT * kGPT;      // entries per chunk (8192)
constexpr int kGNB = 2048;               // histogram bins
constexpr uint32_t kCandCap = 65536;     // candidate list capacity
constexpr int kSamples = 4096;
constexpr int kMaxRounds = 3;            // refinement rounds (11 bits each) reach one key

struct GridMeta {
  float scale;      // |x| bins: nb / sample max (0: integer bins from the start)
  int lo, hi;       // key range that holds T
  int sft;          // integer bins of the current round: (key - lo) >> sft
  int round;        // 0: |x| bins; >= 1: integer bins
  uint32_t kr;      // rank of T within [lo, hi]
  uint32_t m;       // entries in [lo, hi]
  int resolved;     // T and need are known without a candidate list
  int T;
  uint32_t need;
  uint32_t ncand;   // candidates appended by count
  uint32_t nchunks;
};

struct WsLayout {
  GridMeta* meta;
  uint32_t* hist;   // kGNB
  uint32_t* cgt;    // nchunks: entries above (later: kept entries before the chunk)
  uint32_t* ceq;    // nchunks: entries equal to T (later: ties before the chunk)
  int* ckey;        // kCandCap candidate keys
  int64_t* cidx;    // kCandCap candidate positions
};

size_t align256(size_t b) { return (b + 255) / 256 * 256; }

WsLayout layout(void* ws, int64_t nchunks) {
  WsLayout w;
  char* p = static_cast<char*>(ws);
  w.meta = reinterpret_cast<GridMeta*>(p);
  p += align256(sizeof(GridMeta));
  w.hist = reinterpret_cast<uint32_t*>(p);
  p += align256(kGNB * 4);
  w.cgt = reinterpret_cast<uint32_t*>(p);
  p += align256(nchunks * 4);
  w.ceq = reinterpret_cast<uint32_t*>(p);
  p += align256(nchunks * 4);
  w.cidx = reinterpret_cast<int64_t*>(p);
  p += align256(kCandCap * 8);
  w.ckey = reinterpret_cast<int*>(p);
  return w;
}

size_t ws_bytes_for(int64_t L) {
  const int64_t nchunks = (L + kCH - 1) / kCH;
  return align256(sizeof(GridMeta)) + align256(kGNB * 4) + 2 * align256(nchunks * 4) +
         align256(kCandCap * 8) + align256(kCandCap * 4);
}

template <int MODE>
__device__ __forceinline__ float ranked(float x, float a) {
  if (MODE == kEF) return fadd(x, a);
  if (MODE == kDelta) return fsub(x, a);
  return x;
}

// The value a pass ranks: after the first histogram pass of error feedback,
// s = x + err lives in err itself.
template <int MODE>
__device__ __forceinline__ float value_at(const float* xr, const float* ar, int64_t e) {
  if (MODE == kEF) return ar[e];
  if (MODE == kDelta) return fsub(xr[e], ar[e]);
  return xr[e];
}

__device__ __forceinline__ uint32_t block_sum(uint32_t v, uint32_t* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = __reduce_add_sync(kFull, v);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  uint32_t s = 0;
  for (int i = 0; i < static_cast<int>(blockDim.x / 32); ++i) s += red[i];
  __syncthreads();
  return s;
}

__global__ void g_init(GridMeta* meta, uint32_t* hist, int64_t nchunks) {
  pdl_begin();
  for (int i = threadIdx.x; i < kGNB; i += blockDim.x) hist[i] = 0;
  if (threadIdx.x == 0) {
    GridMeta m = {};
    m.lo = 0;
    m.hi = 0x7fffffff;
    m.nchunks = static_cast<uint32_t>(nchunks);
    *meta = m;
  }
}

template <int MODE>
__global__ void __launch_bounds__(kGT) g_sample(const float* xr, const float* ar, int64_t L,
                                                int64_t k, GridMeta* meta) {
  pdl_begin();
  __shared__ uint32_t red[kGT / 32];
  int mx = -1;
  for (int s = threadIdx.x; s < kSamples; s += kGT) {
    const int64_t e = (L / kSamples) * s;
    if (e < L) mx = max(mx, finite_key(mag_key(ranked<MODE>(xr[e], MODE != kPlain ? ar[e] : 0.0f))));
  }
  mx = __reduce_max_sync(kFull, mx);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = static_cast<uint32_t>(mx);
  __syncthreads();
  if (threadIdx.x == 0) {
    int m = -1;
    for (int i = 0; i < kGT / 32; ++i) m = max(m, static_cast<int>(red[i]));
    meta->scale = bucket_scale(m, kGNB);
    meta->kr = static_cast<uint32_t>(k);
    meta->m = static_cast<uint32_t>(L);
    if (k >= L) {  // every entry is kept
      meta->resolved = 1;
      meta->T = -1;
      meta->need = 0;
    }
    if (meta->scale == 0.0f) {
      meta->round = 1;  // integer bins over the whole key range, 2048 of them
      meta->sft = 21 - __clz(0x7fffffff);
    }
  }
}

// Histogram of one chunk into the row histogram.  Round 0: bins linear in |x|
// over every entry (and, for error feedback, s written back into err).
// Later rounds: integer bins over the keys in [lo, hi].
template <int MODE>
__global__ void __launch_bounds__(kGT) g_hist(const float* xr, float* ar, int64_t L,
                                              GridMeta* meta, uint32_t* hist, int first) {
  pdl_begin();
  __shared__ uint32_t sh[kGNB];
  const GridMeta m = *meta;
  const bool bins = !m.resolved && m.m > kCandCap;
  const bool write_s = first && MODE == kEF;  // s = x + err goes back into err once
  if (!bins && !write_s) return;
  for (int i = threadIdx.x; i < kGNB; i += kGT) sh[i] = 0;
  __syncthreads();
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kCH;
  for (int j = 0; j < kGPT; ++j) {
    const int64_t e = c0 + j * kGT + threadIdx.x;
    if (e >= L) break;
    float v;
    if (write_s) {
      v = fadd(xr[e], ar[e]);
      ar[e] = v;
    } else {
      v = value_at<MODE>(xr, ar, e);
    }
    if (!bins) continue;
    const int key = mag_key(v);
    if (m.round == 0) {
      atomicAdd(&sh[bucket_of(key, m.scale, kGNB)], 1u);
    } else if (key >= m.lo && key <= m.hi) {
      atomicAdd(&sh[static_cast<uint32_t>(key - m.lo) >> m.sft], 1u);
    }
  }
  __syncthreads();
  if (!bins) return;
  for (int i = threadIdx.x; i < kGNB; i += kGT)
    if (sh[i]) atomicAdd(&hist[i], sh[i]);
}

// Smallest key whose |x| bin is at least b (bins are monotone in the key).
__device__ int first_key_of_bin(int b, float scale) {
  int lo = 0, hi = 0x7f800000;  // bucket_of(hi) is the top bin
  while (lo < hi) {
    const int mid = lo + (hi - lo) / 2;
    if (bucket_of(mid, scale, kGNB) >= b) hi = mid;
    else lo = mid + 1;
  }
  return lo;
}

// Pick the bin holding the kr-th entry and narrow [lo, hi] to it.
__global__ void __launch_bounds__(kGT) g_pick(GridMeta* meta, uint32_t* hist) {
  pdl_begin();
  __shared__ uint32_t red[kGT / 32];
  __shared__ uint32_t pick_t, pick_excl;
  GridMeta m = *meta;
  if (m.resolved || m.m <= kCandCap) return;
  constexpr int G = kGNB / kGT;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t c[G], total = 0;
  for (int b = 0; b < G; ++b) {
    c[b] = hist[kGNB - 1 - (tid * G + b)];
    total += c[b];
  }
  if (tid == 0) {
    pick_t = 0;
    pick_excl = 0;
  }
  const uint32_t inc = warp_inclusive_scan(total, lane);
  if (lane == 31) red[warp] = inc;
  __syncthreads();
  uint32_t base = 0;
  for (int i = 0; i < warp; ++i) base += red[i];
  const uint32_t excl = base + inc - total;
  if (excl < m.kr && m.kr <= excl + total) {
    pick_t = tid;
    pick_excl = excl;
  }
  __syncthreads();
  if (tid == static_cast<int>(pick_t)) {
    uint32_t run = pick_excl;
    int bin = kGNB - 1 - tid * G;
    uint32_t cnt = 0;
    for (int b = 0; b < G; ++b) {
      bin = kGNB - 1 - (tid * G + b);
      cnt = c[b];
      if (run + cnt >= m.kr) break;
      run += cnt;
    }
    int nlo, nhi;
    if (m.round == 0) {
      nlo = first_key_of_bin(bin, m.scale);
      nhi = (bin == kGNB - 1) ? 0x7fffffff : first_key_of_bin(bin + 1, m.scale) - 1;
    } else {
      nlo = m.lo + (bin << m.sft);
      nhi = static_cast<int>(min(static_cast<uint32_t>(m.hi),
                                 static_cast<uint32_t>(nlo) + ((1u << m.sft) - 1u)));
    }
    m.kr -= run;
    m.m = cnt;
    m.lo = nlo;
    m.hi = nhi;
    if (cnt == m.kr) {  // the whole range is kept
      m.resolved = 1;
      m.T = nlo - 1;
      m.need = 0;
    } else if (nlo >= nhi) {  // one key left: ties at T
      m.resolved = 1;
      m.T = nlo;
      m.need = m.kr;
    } else {
      m.round += 1;
      m.sft = max(0, 21 - __clz(static_cast<uint32_t>(nhi - nlo)));  // at most 2048 bins
    }
    *meta = m;
  }
  __syncthreads();
  for (int i = tid; i < kGNB; i += kGT) hist[i] = 0;  // ready for the next round
}

// Per chunk: entries above (and equal to) T once it is known; otherwise the
// entries above [lo, hi], with the entries inside appended to the list.
template <int MODE>
__global__ void __launch_bounds__(kGT) g_count(const float* xr, const float* ar, int64_t L,
                                               GridMeta* meta, uint32_t* cgt, uint32_t* ceq,
                                               int* ckey, int64_t* cidx) {
  pdl_begin();
  __shared__ uint32_t red[kGT / 32];
  const GridMeta m = *meta;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kCH;
  uint32_t g = 0, q = 0;
  for (int j = 0; j < kGPT; ++j) {
    const int64_t e = c0 + j * kGT + threadIdx.x;
    if (e >= L) break;
    const int key = mag_key(value_at<MODE>(xr, ar, e));
    if (m.resolved) {
      g += key > m.T;
      q += key == m.T;
    } else {
      g += key > m.hi;
      if (key >= m.lo && key <= m.hi) {
        const uint32_t at = atomicAdd(&meta->ncand, 1u);
        if (at < kCandCap) {
          ckey[at] = key;
          cidx[at] = e;
        }
      }
    }
  }
  g = block_sum(g, red);
  q = block_sum(q, red);
  if (threadIdx.x == 0) {
    cgt[blockIdx.x] = g;
    ceq[blockIdx.x] = q;
  }
}

// T and need from the candidate list (one CTA), then the candidates' chunks.
__global__ void __launch_bounds__(1024) g_select(GridMeta* meta, uint32_t* cgt, uint32_t* ceq,
                                                 const int* ckey, const int64_t* cidx) {
  pdl_begin();
  __shared__ uint32_t hist[kRoundBins];
  __shared__ int s_lo, s_hi, s_T;
  __shared__ uint32_t s_kr, s_need, s_done;
  GridMeta m = *meta;
  if (m.resolved) return;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t n = min(m.ncand, kCandCap);
  if (tid == 0) {
    s_lo = m.lo;
    s_hi = m.hi;
    s_kr = m.kr;
    s_done = 0;
  }
  __syncthreads();
  // rounds of 256 bins of equal key width over [lo, hi] until one key is left
  // or a bin is kept whole
  while (!s_done) {
    const int lo = s_lo, hi = s_hi;
    if (lo >= hi) {
      if (tid == 0) {
        s_T = lo;
        s_need = s_kr;
        s_done = 1;
      }
      __syncthreads();
      break;
    }
    const int sft = round_shift(lo, hi);
    for (int i = tid; i < kRoundBins; i += 1024) hist[i] = 0;
    __syncthreads();
    for (uint32_t i = tid; i < n; i += 1024) {
      const int key = ckey[i];
      if (key >= lo && key <= hi) atomicAdd(&hist[static_cast<uint32_t>(key - lo) >> sft], 1u);
    }
    __syncthreads();
    if (warp == 0) {
      const BinPick p = warp_pick_bin(hist, s_kr, lane);
      if (lane == 0) {
        const uint32_t kr = s_kr - p.above;
        const int nlo = lo + (p.bin << sft);
        const int nhi = static_cast<int>(
            min(static_cast<uint32_t>(hi), static_cast<uint32_t>(nlo) + ((1u << sft) - 1u)));
        s_kr = kr;
        if (p.count == kr) {
          s_T = nlo - 1;
          s_need = 0;
          s_done = 1;
        } else {
          s_lo = nlo;
          s_hi = nhi;
        }
      }
    }
    __syncthreads();
  }
  const int T = s_T;
  for (uint32_t i = tid; i < n; i += 1024) {
    const int key = ckey[i];
    const int64_t ch = cidx[i] / kCH;
    if (key > T) atomicAdd(&cgt[ch], 1u);
    else if (key == T) atomicAdd(&ceq[ch], 1u);
  }
  if (tid == 0) {
    meta->T = T;
    meta->need = s_need;
    meta->resolved = 1;
  }
}

// Exclusive scan over the 1024 threads of a CTA; *total gets the sum.
__device__ __forceinline__ uint32_t excl_scan_1024(uint32_t v, uint32_t* red, uint32_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t inc = warp_inclusive_scan(v, lane);
  if (lane == 31) red[warp] = inc;
  __syncthreads();
  uint32_t before = 0, all = 0;
  for (int i = 0; i < 32; ++i) {
    if (i < warp) before += red[i];
    all += red[i];
  }
  __syncthreads();
  *total = all;
  return before + inc - v;
}

// Per chunk: kept entries before it and ties (entries equal to T) before it,
// written in place of the chunk's counts.
__global__ void __launch_bounds__(1024) g_scan(const GridMeta* meta, uint32_t* cgt, uint32_t* ceq,
                                               int64_t nchunks) {
  pdl_begin();
  __shared__ uint32_t red[32];
  const uint32_t need = meta->need;
  uint32_t carry_g = 0, carry_e = 0;  // identical in every thread
  for (int64_t base = 0; base < nchunks; base += 1024) {
    const int64_t c = base + threadIdx.x;
    const uint32_t g = c < nchunks ? cgt[c] : 0u;
    const uint32_t e = c < nchunks ? ceq[c] : 0u;
    uint32_t te, tk;
    const uint32_t eb = carry_e + excl_scan_1024(e, red, &te);
    const uint32_t kept = g + (eb >= need ? 0u : min(e, need - eb));
    const uint32_t kb = carry_g + excl_scan_1024(kept, red, &tk);
    if (c < nchunks) {
      cgt[c] = kb;
      ceq[c] = eb;
    }
    carry_g += tk;
    carry_e += te;
  }
}

// Payload of one chunk in ascending index order, and the buffer updates.
template <int MODE>
__global__ void __launch_bounds__(kGT) g_write(const float* xr, float* ar, int64_t L, int64_t k,
                                               const GridMeta* meta, const uint32_t* cgt,
                                               const uint32_t* ceq, float* vals, int32_t* idx) {
  pdl_begin();
  constexpr int NW = kGT / 32;
  __shared__ uint32_t ug[kGPT * NW], ue[kGPT * NW];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int T = meta->T;
  const uint32_t need = meta->need;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kCH;
  const unsigned lt = lanemask_lt();
  // units of 32 consecutive entries: unit u = j * NW + warp covers
  // [c0 + j * kGT + 32 * warp, +32)
  for (int j = 0; j < kGPT; ++j) {
    const int64_t e = c0 + j * kGT + tid;
    int key = -1;
    if (e < L) key = mag_key(value_at<MODE>(xr, ar, e));
    const unsigned bg = __ballot_sync(kFull, key > T);
    const unsigned be = __ballot_sync(kFull, key == T);
    if (lane == 0) {
      ug[j * NW + warp] = __popc(bg);
      ue[j * NW + warp] = __popc(be);
    }
  }
  __syncthreads();
  if (warp == 0) {  // exclusive scans over the chunk's units
    constexpr int PER = kGPT * NW / 32;
    uint32_t g[PER], q[PER], tg = 0, te = 0;
    for (int i = 0; i < PER; ++i) {
      g[i] = ug[lane * PER + i];
      q[i] = ue[lane * PER + i];
      tg += g[i];
      te += q[i];
    }
    uint32_t xg = warp_inclusive_scan(tg, lane) - tg;
    uint32_t xe = warp_inclusive_scan(te, lane) - te;
    for (int i = 0; i < PER; ++i) {
      ug[lane * PER + i] = xg;
      ue[lane * PER + i] = xe;
      xg += g[i];
      xe += q[i];
    }
  }
  __syncthreads();
  const uint32_t kbase = cgt[blockIdx.x], ebase = ceq[blockIdx.x];
  for (int j = 0; j < kGPT; ++j) {
    const int64_t e = c0 + j * kGT + tid;
    float v = 0.0f;
    int key = -1;
    if (e < L) {
      v = value_at<MODE>(xr, ar, e);
      key = mag_key(v);
    }
    const int u = j * NW + warp;
    const bool eq = key == T;
    const unsigned be = __ballot_sync(kFull, eq);
    const uint32_t erank = ebase + ue[u] + __popc(be & lt);
    const bool kp = key > T || (eq && erank < need);
    const unsigned bk = __ballot_sync(kFull, kp);
    if (kp) {
      // kept before it: the chunk's kept predecessors, entries above T in
      // earlier units, ties taken in earlier units, kept lanes of this unit
      const uint64_t pos = static_cast<uint64_t>(kbase) + ug[u] +
                           min(ebase + ue[u], need) - min(ebase, need) + __popc(bk & lt);
      if (pos < static_cast<uint64_t>(k)) {
        vals[pos] = v;
        idx[pos] = static_cast<int32_t>(e);
      }
      if (MODE == kEF) ar[e] = 0.0f;            // err' = s - C(s): +0 where sent
      if (MODE == kDelta) ar[e] = fadd(ar[e], v);  // g' = g + d where sent
    }
  }
}

template <int MODE>
cudaError_t run_grid(const TopkGridArgs& a, cudaStream_t s) {
  const int64_t L = a.L;
  const int64_t nchunks = (L + kCH - 1) / kCH;
  if (nchunks > 0x7fffffffLL) return cudaErrorInvalidValue;
  const WsLayout w = layout(a.ws, nchunks);
  const unsigned grid = static_cast<unsigned>(nchunks);
  for (int64_t r = 0; r < a.rows; ++r) {
    const float* xr = a.x + r * L;
    float* ar = (MODE != kPlain) ? a.aux + r * L : nullptr;
    float* vr = a.vals + r * a.k;
    int32_t* ir = a.idx + r * a.k;
    g_init<<<1, 256, 0, s>>>(w.meta, w.hist, nchunks);
    g_sample<MODE><<<1, kGT, 0, s>>>(xr, ar, L, a.k, w.meta);
    g_hist<MODE><<<grid, kGT, 0, s>>>(xr, ar, L, w.meta, w.hist, 1);
    g_pick<<<1, kGT, 0, s>>>(w.meta, w.hist);
    for (int i = 0; i < kMaxRounds; ++i) {
      g_hist<MODE><<<grid, kGT, 0, s>>>(xr, ar, L, w.meta, w.hist, 0);
      g_pick<<<1, kGT, 0, s>>>(w.meta, w.hist);
    }
    g_count<MODE><<<grid, kGT, 0, s>>>(xr, ar, L, w.meta, w.cgt, w.ceq, w.ckey, w.cidx);
    g_select<<<1, 1024, 0, s>>>(w.meta, w.cgt, w.ceq, w.ckey, w.cidx);
    g_scan<<<1, 1024, 0, s>>>(w.meta, w.cgt, w.ceq, nchunks);
    g_write<MODE><<<grid, kGT, 0, s>>>(xr, ar, L, a.k, w.meta, w.cgt, w.ceq, vr, ir);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace

size_t topk_grid_workspace_bytes(int64_t rows, int64_t L, int64_t k) {
  (void)rows;
  (void)k;
  return ws_bytes_for(L);
}

cudaError_t launch_topk_grid(int mode, const TopkGridArgs& a, int num_sms, cudaStream_t s) {
  (void)num_sms;
  if (a.rows <= 0) return cudaSuccess;
  switch (mode) {
    case kPlain: return run_grid<kPlain>(a, s);
    case kEF: return run_grid<kEF>(a, s);
    case kDelta: return run_grid<kDelta>(a, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace mpc
