// topk_grid.cu -- exact TopK (§2.3), with error feedback (§2.4) or the EF21
// buffer update (§2.4), for rows longer than the on-chip row kernels take (up
// to whole tensors of 2^31-1 entries), with the counters, lists and per-chunk
// status words in a caller workspace.  Rows go in batches of up to 64 (enough
// for about 2^26 entries a batch): every launch below takes a batch, row
// blockIdx.y of it, each row with a workspace slice of its own, so that a call
// is 23 launches per batch whatever the number of rows.
//
// Per row, the selection by the band path (one read of the row), else by the
// multi-pass path where the band path gave up, then the write: one more read
// of the row, or, in list mode (k up to a thirty-second of the row), the
// payload from the list of every entry >= t_lo that the band path's read made.
// Every kernel returns at once when the device-side state says its step is not
// needed, so the host never waits.
//
// Band path:
//   w_sample, w_spick  1/256 of the row's entries (1024 to 65536) spread
//             over it (one a thread) give a band of keys [t_lo, t_hi) that
//             holds the k-th largest magnitude unless the sample is 4
//             standard deviations off (as in topk_band.cuh);
//   w_pass1   one read of the row by persistent CTAs, 8192-entry chunks staged
//             by double-buffered bulk copies: entries >= t_hi ("sure")
//             counted; band entries (list mode: every entry >= t_lo) listed in
//             the workspace (a region per CTA, each chunk's entries one segment
//             in index order) and the band's counted in a 256-bin histogram of
//             their keys (error feedback: s = x + err written back into err);
//   w_pick1   the histogram bin holding the k-th entry (or: the band missed,
//             and the multi-pass path takes over);
//   w_bin2    the band entries in that bin, listed;
//   w_select2 T and `need` among them by integer rounds.
//
// Multi-pass path:
//   init     clear the row's state (before the band path);
//   sample   bin scale from a strided sample of the ranked values;
//   hist     histogram of all entries over bins linear in |x| (error feedback:
//            s = x + err is written back into err unless the band path did);
//   pick     the bin that holds the k-th largest entry, as a key range;
//   3 x (hist, pick)  refinement rounds with 2048 bins of equal key width over
//            that range, while it holds more candidates than the list takes;
//   count    the entries inside the range appended to the candidate list;
//   select   T and `need` from the candidate list.
//
//   (band path) w_mark: band entries above / equal to T join the counts of
//   their 4096-entry write chunks (pass 1 counted the sure entries there);
//   (multi-pass) count also counts, per write chunk, the entries above the
//   range or, once T is known, above / equal to it; select adds the candidates.
//
// Write (both paths): w_scan1 / w_scan2, the prefix sums of the per-chunk
// counts; g_write3, persistent CTAs over 4096-entry chunks, double-buffered:
// the payload in ascending index order and the buffer updates; or, in list
// mode, g_wlist: the same from the list's segments.
#include "common.cuh"
#include "kernels.h"
#include "launch_util.h"
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
constexpr int kWSamples = 65536;         // band path: sample entries
constexpr int kWSBins = 32768;           // band path: sample bins, key >> 16 (1/128 octave)
constexpr int kWSShift = 16;
constexpr int kFBins = 256;              // band path: bins of the band histogram
constexpr uint32_t kCand2Cap = 1u << 21;  // band path: entries of the chosen bin
constexpr float kWZ = 4.0f;              // band half-width in standard deviations
constexpr int kWT = 128;                 // write kernel: threads
constexpr int64_t kWCH = 32 * kWT;       // write kernel: entries of a chunk (4096)
constexpr uint32_t kWNoSure = 0x7f800001u;  // a t_hi no magnitude reaches (NaN bits)

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
  // band path
  int band;         // 1 while the band path is on
  int s_in_aux;     // error feedback: s = x + err has been written into err
  int counted;      // per-chunk counts are in place (the multi-pass count is skipped)
  int bin2;         // the chosen band bin needs w_bin2 / w_select2
  uint32_t t_lo, t_hi;
  int fsh;          // band histogram: bin = min((key - t_lo) >> fsh, 255)
  uint32_t sure;    // entries with key >= t_hi
  uint32_t nband;   // band entries listed (may exceed the capacity: then the path gives up)
  int b_lo, b_hi;   // the chosen band bin's keys
  uint32_t b_kr;    // rank of T within it
  uint32_t ncand2;
  int lmode;        // list mode: every entry >= t_lo listed (the payload comes from the list)
  int smax;         // largest finite sample key (band path)
};

struct WsLayout {
  GridMeta* meta;
  uint32_t* hist;   // kGNB
  uint32_t* cgt;    // per write chunk (kWCH entries): entries above T; after the scan,
                    // those of the earlier chunks of its block of 1024 chunks
  uint32_t* ceq;    // the same for entries equal to T
  uint32_t* tg;     // per block of 1024 write chunks: entries above T before it
  uint32_t* te;     // and entries equal to T before it
  int* ckey;        // kCandCap candidate keys
  int64_t* cidx;    // kCandCap candidate positions
  uint32_t* fhist;  // kFBins: band histogram
  uint32_t* shist;  // kWSBins: sample histogram
  int* bkey;        // band list: value bits (magnitude key = bits & 0x7fffffff)
  uint32_t* bidx;   //            positions in the row
  uint32_t* seg;    // per pass-1 chunk: start of its entries in its CTA's region
  uint32_t* segn;   //                   and their number
  int* c2key;       // kCand2Cap: keys of the chosen band bin
  uint32_t* nbc;    // kMaxBandCtas: band entries listed by each CTA of w_pass1
  uint32_t bcap;    // band list capacity (G regions of bcap / G entries, G the pass-1 grid)
  uint32_t c2cap;   // c2key capacity: the chosen bin's entries are band-list entries
};

// CTAs of the persistent band-path kernels at most (each lists its band
// entries in a region of its own, the band list split evenly among them).
constexpr int kMaxBandCtas = 4096;

// Band list capacity: a sixteenth of the row and 64K entries (the band of a
// 65536-entry sample at 4 standard deviations is a few percent of the row);
// for k up to a thirty-second of the row, room for list mode too: k, a quarter
// more, a sixty-fourth of the row and 64K entries.  (Beyond that the list costs
// more to build and read back than the second read of the row it saves.)
bool list_eligible(int64_t L, int64_t k) { return k <= L / 32; }
uint32_t band_cap(int64_t L, int64_t k) {
  int64_t c = L / 16 + 65536;
  if (list_eligible(L, k)) c = max64(c, k + k / 4 + L / 64 + 65536);
  return static_cast<uint32_t>(min64(c, 0xffffffffLL));
}

size_t align256(size_t b) { return (b + 255) / 256 * 256; }

uint32_t c2_cap(int64_t L, int64_t k) { return min(kCand2Cap, band_cap(L, k)); }

// Band-path sample entries of a row: 1/256 of it (a multiple of 1024), at least
// 1024 and at most kWSamples, so that the sample reads stay a few percent of
// the row's sectors.
int sample_count(int64_t L) {
  return static_cast<int>(max64(1024, min64(kWSamples, L / 256 / 1024 * 1024)));
}

// Rows of one batch: enough rows for about 2^26 entries, at most 64.  Each row
// of a batch has a workspace slice of its own.
constexpr int64_t kMaxBatch = 64;
int64_t grid_batch(int64_t rows, int64_t L) {
  return max64(1, min64(min64(rows, kMaxBatch), (int64_t(1) << 26) / max64(L, 1)));
}

WsLayout layout(void* ws, int64_t L, int64_t k, int64_t nchunks) {
  WsLayout w;
  char* p = static_cast<char*>(ws);
  w.meta = reinterpret_cast<GridMeta*>(p);
  p += align256(sizeof(GridMeta));
  w.hist = reinterpret_cast<uint32_t*>(p);
  p += align256(kGNB * 4);
  const int64_t nwch = (L + kWCH - 1) / kWCH;
  w.cgt = reinterpret_cast<uint32_t*>(p);
  p += align256(static_cast<size_t>(nwch) * 4);
  w.ceq = reinterpret_cast<uint32_t*>(p);
  p += align256(static_cast<size_t>(nwch) * 4);
  w.tg = reinterpret_cast<uint32_t*>(p);
  p += align256(static_cast<size_t>((nwch + 1023) / 1024) * 4);
  w.te = reinterpret_cast<uint32_t*>(p);
  p += align256(static_cast<size_t>((nwch + 1023) / 1024) * 4);
  w.cidx = reinterpret_cast<int64_t*>(p);
  p += align256(kCandCap * 8);
  w.ckey = reinterpret_cast<int*>(p);
  p += align256(kCandCap * 4);
  w.fhist = reinterpret_cast<uint32_t*>(p);
  p += align256(kFBins * 4);
  w.shist = reinterpret_cast<uint32_t*>(p);
  p += align256(kWSBins * 4);
  w.c2cap = c2_cap(L, k);
  w.c2key = reinterpret_cast<int*>(p);
  p += align256(static_cast<size_t>(w.c2cap) * 4);
  w.nbc = reinterpret_cast<uint32_t*>(p);
  p += align256(kMaxBandCtas * 4);
  w.bcap = band_cap(L, k);
  w.bkey = reinterpret_cast<int*>(p);
  p += align256(static_cast<size_t>(w.bcap) * 4);
  w.bidx = reinterpret_cast<uint32_t*>(p);
  p += align256(static_cast<size_t>(w.bcap) * 4);
  w.seg = reinterpret_cast<uint32_t*>(p);
  p += align256(static_cast<size_t>(nchunks) * 4);
  w.segn = reinterpret_cast<uint32_t*>(p);
  return w;
}

size_t ws_bytes_for(int64_t L, int64_t k) {
  const int64_t nchunks = (L + kCH - 1) / kCH;
  return 2 * align256(static_cast<size_t>(nchunks) * 4) + align256(sizeof(GridMeta)) +
         align256(kGNB * 4) +
         2 * align256(static_cast<size_t>((L + kWCH - 1) / kWCH) * 4) +
         2 * align256(static_cast<size_t>(((L + kWCH - 1) / kWCH + 1023) / 1024) * 4) +
         align256(kCandCap * 8) + align256(kCandCap * 4) + align256(kFBins * 4) +
         align256(kWSBins * 4) +
         align256(static_cast<size_t>(c2_cap(L, k)) * 4) + align256(kMaxBandCtas * 4) +
         2 * align256(static_cast<size_t>(band_cap(L, k)) * 4);
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

// Rows are processed in batches, row blockIdx.y of a batch per launch: its
// slice of the workspace lies wsr bytes after the previous row's.
template <class T>
__device__ __forceinline__ T* row_ws(T* p, size_t wsr) {
  return reinterpret_cast<T*>(reinterpret_cast<uintptr_t>(p) + static_cast<uintptr_t>(blockIdx.y) * wsr);
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

__global__ void g_init(GridMeta* meta, uint32_t* hist, uint32_t* shist, uint32_t* fhist,
                       int64_t nchunks, int64_t L, int64_t k, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  meta = row_ws(meta, wsr);
  hist = row_ws(hist, wsr);
  shist = row_ws(shist, wsr);
  fhist = row_ws(fhist, wsr);
  for (int i = threadIdx.x; i < kGNB; i += blockDim.x) hist[i] = 0;
  for (int i = threadIdx.x; i < kWSBins; i += blockDim.x) shist[i] = 0;
  for (int i = threadIdx.x; i < kFBins; i += blockDim.x) fhist[i] = 0;
  if (threadIdx.x == 0) {
    GridMeta m = {};
    m.lo = 0;
    m.hi = 0x7fffffff;
    m.nchunks = static_cast<uint32_t>(nchunks);
    m.smax = -1;
    if (k >= L) {  // every entry is kept
      m.resolved = 1;
      m.T = -1;
      m.need = 0;
    }
    *meta = m;
  }
}

template <int MODE>
__global__ void __launch_bounds__(kGT) g_sample(const float* xr, const float* ar, int64_t L,
                                                int64_t k, GridMeta* meta, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  xr += static_cast<int64_t>(blockIdx.y) * L;
  if (MODE != kPlain) ar += static_cast<int64_t>(blockIdx.y) * L;
  meta = row_ws(meta, wsr);
  __shared__ uint32_t red[kGT / 32];
  if (meta->resolved) return;  // the band path found T (or every entry is kept)
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
                                              GridMeta* meta, uint32_t* hist, int first,
                                              size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  xr += static_cast<int64_t>(blockIdx.y) * L;
  if (MODE != kPlain) ar += static_cast<int64_t>(blockIdx.y) * L;
  meta = row_ws(meta, wsr);
  hist = row_ws(hist, wsr);
  __shared__ uint32_t sh[kGNB];
  const GridMeta m = *meta;
  const bool bins = !m.resolved && m.m > kCandCap;
  // s = x + err goes back into err once (unless the band path already did)
  const bool write_s = first && MODE == kEF && !m.s_in_aux;
  if (!bins && !write_s) return;
  for (int i = threadIdx.x; i < kGNB; i += kGT) sh[i] = 0;
  __syncthreads();
  // chunks c, c + gridDim.x, ... (a fixed grid, so that a launch with nothing to
  // do costs little)
  for (int64_t c0 = static_cast<int64_t>(blockIdx.x) * kCH; c0 < L;
       c0 += static_cast<int64_t>(gridDim.x) * kCH) {
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
__global__ void __launch_bounds__(kGT) g_pick(GridMeta* meta, uint32_t* hist, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  meta = row_ws(meta, wsr);
  hist = row_ws(hist, wsr);
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

// Per write chunk (kWCH entries): once T is known, the entries above and equal
// to it; otherwise the entries above [lo, hi], with the entries inside appended
// to the candidate list.  A fixed grid strides over the chunks.
template <int MODE>
__global__ void __launch_bounds__(kGT) g_count(const float* xr, const float* ar, int64_t L,
                                               GridMeta* meta, uint32_t* cgt, uint32_t* ceq,
                                               int* ckey, int64_t* cidx, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  xr += static_cast<int64_t>(blockIdx.y) * L;
  if (MODE != kPlain) ar += static_cast<int64_t>(blockIdx.y) * L;
  meta = row_ws(meta, wsr);
  cgt = row_ws(cgt, wsr);
  ceq = row_ws(ceq, wsr);
  ckey = row_ws(ckey, wsr);
  cidx = row_ws(cidx, wsr);
  __shared__ uint32_t red[kGT / 32];
  const GridMeta m = *meta;
  if (m.counted) return;  // the band path has the counts
  for (int64_t c = blockIdx.x; c * kWCH < L; c += gridDim.x) {
    const int64_t c0 = c * kWCH;
    uint32_t g = 0, q = 0;
    for (int j = 0; j < kWCH / kGT; ++j) {
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
      cgt[c] = g;
      ceq[c] = q;
    }
  }
}

// T and need from the candidate list (one CTA), then the candidates' chunks.
__global__ void __launch_bounds__(1024) g_select(GridMeta* meta, uint32_t* cgt, uint32_t* ceq,
                                                 const int* ckey, const int64_t* cidx, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  meta = row_ws(meta, wsr);
  cgt = row_ws(cgt, wsr);
  ceq = row_ws(ceq, wsr);
  ckey = row_ws(ckey, wsr);
  cidx = row_ws(cidx, wsr);
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
    const int64_t ch = cidx[i] / kWCH;
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

// ===========================================================================
// Band path
// ===========================================================================

// The band from a sample of the row.  w_sample: ns = sample_count(L) entries
// spread evenly over the row, one a thread over ns / 1024 CTAs, binned by
// magnitude key into 32768 bins of 1/128 octave (key >> 16), and the largest
// finite sample key.
// w_spick (one CTA): the band reaches 4 standard deviations of the sample count
// on either side of the k-th entry; list mode when the sample's count at or
// above t_lo, scaled to the row with a margin, fits the list.
template <int MODE>
__global__ void __launch_bounds__(1024) w_sample(const float* xr, const float* ar, int64_t L,
                                                 GridMeta* meta, uint32_t* shist, int ns,
                                                 size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  xr += static_cast<int64_t>(blockIdx.y) * L;
  if (MODE != kPlain) ar += static_cast<int64_t>(blockIdx.y) * L;
  meta = row_ws(meta, wsr);
  shist = row_ws(shist, wsr);
  if (meta->resolved) return;  // every entry is kept
  const int64_t s = static_cast<int64_t>(blockIdx.x) * 1024 + threadIdx.x;
  const int64_t e = s * L / ns;
  const int key = mag_key(ranked<MODE>(xr[e], MODE != kPlain ? ar[e] : 0.0f));
  // lanes with the same bin add once
  const uint32_t bin = static_cast<uint32_t>(key) >> kWSShift;
  const unsigned same = __match_any_sync(kFull, bin);
  if ((threadIdx.x & 31) == __ffs(same) - 1) atomicAdd(&shist[bin], static_cast<uint32_t>(__popc(same)));
  const int mx = __reduce_max_sync(kFull, finite_key(key));
  if ((threadIdx.x & 31) == 0 && mx > 0) atomicMax(&meta->smax, mx);
}

__global__ void __launch_bounds__(1024) w_spick(int64_t L, int64_t k, GridMeta* meta,
                                                const uint32_t* shist, int list_ok, uint32_t bcap,
                                                int ns, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  meta = row_ws(meta, wsr);
  shist = row_ws(shist, wsr);
  // bins in rank order (largest keys first): warp w reads ranks [1024 w, 1024 w + 1024),
  // lane l the ranks 1024 w + 32 j + l (coalesced)
  constexpr int J = kWSBins / 1024;
  __shared__ uint32_t wsum[32];
  __shared__ int pick[2];
  __shared__ uint32_t s_ge;  // sample entries in the bins down to t_lo's
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (meta->resolved) return;
  const int smax = meta->smax;
  if (smax <= 0) return;  // no finite non-zero magnitude in the sample: multi-pass path
  if (tid < 2) pick[tid] = -1;
  if (tid == 0) s_ge = ns;
  const float mu = __fdividef(static_cast<float>(k) * static_cast<float>(ns),
                              static_cast<float>(L));
  const float sd = mu * rsqrtf(mu);
  const int r_hi = static_cast<int>(floorf(mu - kWZ * sd));
  const int r_lo = static_cast<int>(ceilf(mu + kWZ * sd)) + 1;
  uint32_t v[J], s = 0;
#pragma unroll
  for (int j = 0; j < J; ++j) {
    v[j] = shist[kWSBins - 1 - (1024 * warp + 32 * j + lane)];
    s += v[j];
  }
  s = __reduce_add_sync(kFull, s);
  if (lane == 0) wsum[warp] = s;
  __syncthreads();
  uint32_t before = 0;  // sample entries in the warps' blocks before this one
  for (int w = 0; w < warp; ++w) before += wsum[w];
  const int rs[2] = {r_hi, r_lo};
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int r = rs[q];
    if (r >= 1 && r <= ns && before < static_cast<uint32_t>(r) &&
        static_cast<uint32_t>(r) <= before + s) {
      // this warp's block holds the r-th largest: 32 bins at a time
      uint32_t run = before;
      for (int j = 0; j < J; ++j) {
        const uint32_t incl = run + warp_inclusive_scan(v[j], lane);
        const bool hit = incl >= static_cast<uint32_t>(r) && incl - v[j] < static_cast<uint32_t>(r);
        const unsigned who = __ballot_sync(kFull, hit);
        if (who) {
          if (lane == __ffs(who) - 1) {
            pick[q] = kWSBins - 1 - (1024 * warp + 32 * j + lane);
            if (q == 1) s_ge = incl;
          }
          break;
        }
        run = __shfl_sync(kFull, incl, 31);
      }
    }
  }
  __syncthreads();
  if (tid == 0) {
    uint32_t t_lo = 0, t_hi = kWNoSure;
    if (pick[0] >= 0 && pick[0] < kWSBins - 1)
      t_hi = min(static_cast<uint32_t>(pick[0] + 1) << kWSShift, kWNoSure);
    if (pick[1] > 0) t_lo = static_cast<uint32_t>(pick[1]) << kWSShift;
    if (t_lo > t_hi) t_lo = t_hi;
    // the band histogram spans [t_lo, t_hi), or, with nothing sure, up to one
    // octave above the sample's largest magnitude (larger keys share the top bin)
    const uint32_t fhi = t_hi != kWNoSure ? t_hi - 1u
                                          : min(static_cast<uint32_t>(smax) + (1u << 23), 0x7f7fffffu);
    meta->t_lo = t_lo;
    meta->t_hi = t_hi;
    meta->fsh = max(0, 24 - __clz(max(fhi, t_lo) - t_lo));  // (key - t_lo) >> fsh < 256
    meta->sure = 0;
    meta->nband = 0;
    meta->ncand2 = 0;
    meta->bin2 = 0;
    meta->band = 1;
    const float est = static_cast<float>(pick[1] > 0 ? s_ge : ns) *
                      (static_cast<float>(L) / static_cast<float>(ns));
    meta->lmode = list_ok && pick[1] > 0 && est * 1.25f + 65536.0f <= static_cast<float>(bcap);
  }
}

// The chunk loader of the persistent band-path kernels: chunk c's entries of
// src into buf by bulk copies, part w (1024 entries) completing on bars[w];
// issued by the first NW lanes of warp 0.  fence.proxy.async first: the buffer
// was last written by generic stores two chunks before.
template <int NW, int64_t CH>
__device__ __forceinline__ void issue_chunk(float* buf, const float* src, const float* pre,
                                            int64_t L, int64_t c, uint64_t* bars, int lane) {
  const int64_t c0 = c * CH;
  const int n = static_cast<int>(min64(CH, L - c0));
  const int p0 = 1024 * lane;
  if (lane >= NW || p0 >= n) return;
  const uint32_t bytes = static_cast<uint32_t>(min(1024, n - p0)) * 4u;
  fence_proxy_async_smem();
  if (pre != nullptr) bulk_prefetch_l2(pre + c0 + p0, bytes);
  mbar_arrive_expect_tx(&bars[lane], bytes);
  bulk_g2s(buf + p0, src + c0 + p0, bytes, &bars[lane]);
}

// L2 prefetch of chunk c of src, part w (1024 entries) by lane w of warp 0: the
// chunk after the one whose bulk copies were just issued, so that each CTA has
// two chunks on the way from HBM.
template <int NW, int64_t CH>
__device__ __forceinline__ void prefetch_chunk(const float* src, int64_t L, int64_t c, int lane) {
  const int64_t c0 = c * CH;
  if (c0 >= L) return;
  const int n = static_cast<int>(min64(CH, L - c0));
  const int p0 = 1024 * lane;
  if (lane >= NW || p0 >= n) return;
  const uint32_t bytes = static_cast<uint32_t>(min(1024, n - p0)) * 4u;
  bulk_prefetch_l2(src + c0 + p0, bytes);
}

// One read of the row.  Persistent CTAs take chunks c, c + G, ... (G = the grid),
// double-buffered: the next chunk's bulk copies are in flight while this one
// is classified.  Thread t owns the 32 consecutive entries [32t, 32t + 32) of a
// chunk (within its warp's part, so that a warp needs no other warp's data):
// per entry |x| >= t_hi ("sure") and |x| >= t_lo as bit words.  The sure
// entries of each write chunk (half a chunk here) go to cgt; the band entries
// go to this CTA's region of the band list (rcap entries), in index order
// within each warp's run, and into the CTA's histogram of band keys, added to
// the row's once at the end.
template <int MODE>
__global__ void __launch_bounds__(kGT) w_pass1(const float* xr, float* ar, int64_t L,
                                               int64_t nchunks, int aligned, GridMeta* meta,
                                               uint32_t* cgt, uint32_t* ceq, int* bkey,
                                               uint32_t* bidx, uint32_t rcap, uint32_t* nbc,
                                               uint32_t* seg, uint32_t* segn, uint32_t* fhist,
                                               uint32_t spin_limit, unsigned* status, size_t wsr) {
  pdl_begin();
  xr += static_cast<int64_t>(blockIdx.y) * L;
  if (MODE != kPlain) ar += static_cast<int64_t>(blockIdx.y) * L;
  meta = row_ws(meta, wsr);
  cgt = row_ws(cgt, wsr);
  ceq = row_ws(ceq, wsr);
  bkey = row_ws(bkey, wsr);
  bidx = row_ws(bidx, wsr);
  nbc = row_ws(nbc, wsr);
  seg = row_ws(seg, wsr);
  segn = row_ws(segn, wsr);
  fhist = row_ws(fhist, wsr);
  constexpr int NW = kGT / 32;
  extern __shared__ __align__(16) float wbuf[];  // 2 x kCH
  __shared__ uint32_t fh[kFBins];
  __shared__ uint32_t rs[2][NW];  // sure entries per warp, by buffer
  __shared__ uint32_t wl[NW];     // listed entries per warp of the current chunk
  __shared__ uint32_t s_fail;
  __shared__ uint64_t bars[2][NW];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (!meta->band || meta->resolved) return;
  const uint32_t t_lo = meta->t_lo, t_hi = meta->t_hi;
  const int fsh = meta->fsh;
  const bool lmode = meta->lmode != 0;
  const float f_lo = __uint_as_float(t_lo), f_hi = __uint_as_float(t_hi);
  for (int i = tid; i < kFBins; i += kGT) fh[i] = 0;
  if (tid == 0) s_fail = 0;
  uint32_t cnt = 0;  // entries this CTA listed (the same in every thread)
  if (aligned && warp == 0 && lane < NW) {
    mbar_init(&bars[0][lane], 1);
    mbar_init(&bars[1][lane], 1);
    fence_mbar_init();
  }
  __syncthreads();
  const uint32_t rbase = blockIdx.x * rcap;  // this CTA's region of the band list
  const float* pre = MODE != kPlain ? ar : nullptr;
  int64_t c = blockIdx.x;
  if (aligned && warp == 0 && c < nchunks) issue_chunk<NW, kCH>(wbuf, xr, pre, L, c, bars[0], lane);
  uint32_t par = 0;  // bit b: parity of buffer b's next phase
  uint32_t sure_w = 0;  // sure entries seen by this warp
  int64_t prev = -1;
  int b = 0;
  // the sure counts of chunk c's two write chunks, from the warps' sums in rs[bb]
  auto put_sure = [&](int64_t cc, int bb) {
    constexpr int H = NW / 2;  // warps of a write chunk
    for (int h = 0; h < 2; ++h) {
      const int64_t wc = 2 * cc + h;
      if (wc * kWCH >= L) break;
      uint32_t s = 0;
#pragma unroll
      for (int w = 0; w < H; ++w) s += rs[bb][h * H + w];
      cgt[wc] = lmode ? 0u : s;  // list mode: the sure entries are counted from the list
      ceq[wc] = 0;
    }
  };
  static_assert(kCH == 2 * kWCH, "a pass-1 chunk is two write chunks");
  for (; c < nchunks; c += gridDim.x, b ^= 1) {
    const int64_t cn = c + gridDim.x;
    if (aligned && warp == 0 && cn < nchunks) {
      issue_chunk<NW, kCH>(wbuf + (b ^ 1) * kCH, xr, pre, L, cn, bars[b ^ 1], lane);
      // plain TopK only (measured: with the err row as well, and in the write
      // pass, the deeper prefetch is slower)
      if (MODE == kPlain) prefetch_chunk<NW, kCH>(xr, L, cn + gridDim.x, lane);
    }
    if (tid == 0 && prev >= 0) put_sure(prev, b ^ 1);
    const int64_t c0 = c * kCH;
    const int n = static_cast<int>(min64(kCH, L - c0));
    float* cb = wbuf + b * kCH;
    const int pb = 1024 * warp;
    if (pb < n) {
      if (aligned) {
        if (!mbar_wait_bounded(&bars[b][warp], (par >> b) & 1u, spin_limit, status)) {
          mbar_wait_bounded(&bars[b][warp], (par >> b) & 1u, kDrainPolls, nullptr);
          s_fail = 1;
        }
        if (MODE != kPlain) {
          const int nq = min(1024, n - pb) / 4;
          float4* c4 = reinterpret_cast<float4*>(cb + pb);
          float4* a4 = reinterpret_cast<float4*>(ar + c0 + pb);
          for (int q = lane; q < nq; q += 32) {
            const float4 xv = c4[q];
            const float4 av = a4[q];
            const float4 sv = make_float4(ranked<MODE>(xv.x, av.x), ranked<MODE>(xv.y, av.y),
                                          ranked<MODE>(xv.z, av.z), ranked<MODE>(xv.w, av.w));
            c4[q] = sv;
            if (MODE == kEF) a4[q] = sv;  // s = x + err into err
          }
          fence_proxy_async_smem();  // these stores before the buffer's next bulk copy
        }
      } else {
        for (int e = pb + lane; e < min(pb + 1024, n); e += 32) {
          const float v = ranked<MODE>(xr[c0 + e], MODE != kPlain ? ar[c0 + e] : 0.0f);
          cb[e] = v;
          if (MODE == kEF) ar[c0 + e] = v;
        }
      }
      __syncwarp();
    }
    par ^= 1u << b;
    // classification of this thread's 32 entries
    const int e0 = 32 * tid;
    const int nv = max(0, min(32, n - e0));
    const uint32_t vmask = nv >= 32 ? 0xffffffffu : ((1u << nv) - 1u);
    uint32_t hw = 0, gw = 0;
    if (nv > 0) {
      const float4* my4 = reinterpret_cast<const float4*>(cb + e0);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float4 v = my4[(u + lane) & 7];  // 8 consecutive lanes on 8 bank groups
        or_if_ge(hw, v.x, f_hi, 1u << (4 * u + 0));
        or_if_ge(hw, v.y, f_hi, 1u << (4 * u + 1));
        or_if_ge(hw, v.z, f_hi, 1u << (4 * u + 2));
        or_if_ge(hw, v.w, f_hi, 1u << (4 * u + 3));
        or_if_ge(gw, v.x, f_lo, 1u << (4 * u + 0));
        or_if_ge(gw, v.y, f_lo, 1u << (4 * u + 1));
        or_if_ge(gw, v.z, f_lo, 1u << (4 * u + 2));
        or_if_ge(gw, v.w, f_lo, 1u << (4 * u + 3));
      }
      const uint32_t rot = 4u * static_cast<uint32_t>(lane & 7);
      hw = __funnelshift_l(hw, hw, rot) & vmask;
      gw = __funnelshift_l(gw, gw, rot) & vmask;
    }
    // the listed entries (the band; list mode: every entry >= t_lo) of this chunk
    // as one segment of the CTA's region, in index order
    const uint32_t bw = gw & ~hw;
    const uint32_t lw = lmode ? gw : bw;
    const uint32_t nlw = __popc(lw);
    const uint32_t bi = warp_inclusive_scan(nlw, lane);
    if (lane == 31) wl[warp] = bi;
    __syncthreads();
    uint32_t wb = 0, ctot = 0;
#pragma unroll
    for (int w2 = 0; w2 < NW; ++w2) {
      wb += w2 < warp ? wl[w2] : 0u;
      ctot += wl[w2];
    }
    if (tid == 0) {
      seg[c] = cnt;
      segn[c] = ctot;
    }
    uint32_t pos = cnt + wb + bi - nlw;
    cnt += ctot;
    uint32_t w = lw;
    while (w) {
      const int j = __ffs(w) - 1;
      w &= w - 1;
      const int e = e0 + j;
      const int bits = __float_as_int(cb[e]);
      if ((bw >> j) & 1u)
        atomicAdd(&fh[min(static_cast<uint32_t>((bits & 0x7fffffff) - static_cast<int>(t_lo)) >> fsh,
                          kFBins - 1u)],
                  1u);
      if (pos < rcap) {
        bkey[rbase + pos] = bits;
        bidx[rbase + pos] = static_cast<uint32_t>(c0 + e);
      }
      ++pos;
    }
    const uint32_t ws = __reduce_add_sync(kFull, static_cast<uint32_t>(__popc(hw)));
    sure_w += ws;
    if (lane == 0) rs[b][warp] = ws;
    __syncthreads();  // buffer b free for the chunk after next; rs[b] complete
    prev = c;
  }
  if (lane == 0 && sure_w) atomicAdd(&meta->sure, sure_w);
  if (tid == 0) {
    if (prev >= 0) put_sure(prev, b ^ 1);
    nbc[blockIdx.x] = min(cnt, rcap);
    if (cnt) atomicAdd(&meta->nband, cnt);
    // a full region, or a timed-out copy: the multi-pass path takes over
    if (cnt > rcap || s_fail) meta->band = 0;
    if (MODE == kEF && blockIdx.x == 0) meta->s_in_aux = 1;
  }
  for (int i = tid; i < kFBins; i += kGT)
    if (fh[i]) atomicAdd(&fhist[i], fh[i]);
}

// The band bin holding the k-th entry, or the band path gives up (one warp).
__global__ void __launch_bounds__(32) w_pick1(GridMeta* meta, const uint32_t* fhist, int64_t k,
                                              size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  meta = row_ws(meta, wsr);
  fhist = row_ws(fhist, wsr);
  const GridMeta m = *meta;
  if (!m.band || m.resolved) return;
  const int lane = threadIdx.x & 31;
  const int64_t ge = m.lmode ? static_cast<int64_t>(m.nband) : static_cast<int64_t>(m.sure) + m.nband;
  if (!(static_cast<int64_t>(m.sure) < k && k <= ge)) {
    if (lane == 0) meta->band = 0;  // the multi-pass path takes over
    return;
  }
  const uint32_t kr = static_cast<uint32_t>(k - m.sure);
  const BinPick p = warp_pick_bin(fhist, kr, lane);
  if (lane == 0) {
    const int bl = static_cast<int>(m.t_lo) + (p.bin << m.fsh);
    // the top bin also takes every larger band key (none reaches t_hi; the
    // list of list mode holds the sure entries too)
    int bh = p.bin == kFBins - 1
                 ? 0x7fffffff
                 : static_cast<int>(min(static_cast<uint32_t>(bl) + ((1u << m.fsh) - 1u), 0x7fffffffu));
    if (m.t_hi != kWNoSure) bh = min(bh, static_cast<int>(m.t_hi) - 1);
    const uint32_t kr2 = kr - p.above;
    if (p.count == kr2) {  // the bin is kept whole
      meta->T = bl - 1;
      meta->need = 0;
      meta->counted = 1;
      meta->resolved = 1;
    } else {
      meta->b_lo = bl;
      meta->b_hi = bh;
      meta->b_kr = kr2;
      meta->bin2 = 1;
    }
  }
}

// The band entries of the chosen bin, listed: CTA r reads region r of the band
// list (four loads in flight a thread; one atomic a warp).
__global__ void __launch_bounds__(256) w_bin2(GridMeta* meta, const int* bkey, const uint32_t* nbc,
                                              uint32_t rcap, int* c2key, uint32_t c2cap,
                                              size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  meta = row_ws(meta, wsr);
  bkey = row_ws(bkey, wsr);
  nbc = row_ws(nbc, wsr);
  c2key = row_ws(c2key, wsr);
  const GridMeta m = *meta;
  if (!m.band || !m.bin2) return;
  const int lane = threadIdx.x & 31;
  const unsigned lt = lanemask_lt();
  const uint32_t nr = nbc[blockIdx.x];
  const int* rk = bkey + static_cast<size_t>(blockIdx.x) * rcap;
  for (uint32_t i0 = (threadIdx.x & ~31u) * 4u; i0 < nr; i0 += 256u * 4u) {
    int key[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t i = i0 + 32u * q + lane;
      key[q] = i < nr ? (rk[i] & 0x7fffffff) : -1;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const bool in = key[q] >= m.b_lo && key[q] <= m.b_hi;
      const unsigned bb = __ballot_sync(kFull, in);
      if (!bb) continue;
      uint32_t base = 0;
      if (lane == 0) base = atomicAdd(&meta->ncand2, static_cast<uint32_t>(__popc(bb)));
      base = __shfl_sync(kFull, base, 0);
      const uint32_t slot = base + __popc(bb & lt);
      if (in && slot < c2cap) c2key[slot] = key[q];
    }
  }
}

// T and need among the chosen bin's entries, by integer rounds (one CTA).
__global__ void __launch_bounds__(1024) w_select2(GridMeta* meta, const int* c2key, uint32_t c2cap,
                                                  size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  meta = row_ws(meta, wsr);
  c2key = row_ws(c2key, wsr);
  __shared__ uint32_t hist[kRoundBins];
  __shared__ int s_lo, s_hi, s_T;
  __shared__ uint32_t s_kr, s_need, s_done;
  const GridMeta m = *meta;
  if (!m.band || !m.bin2) return;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (m.ncand2 > c2cap) {
    if (tid == 0) meta->band = 0;  // too crowded: the multi-pass path takes over
    return;
  }
  const uint32_t n = m.ncand2;
  if (tid == 0) {
    s_lo = m.b_lo;
    s_hi = m.b_hi;
    s_kr = m.b_kr;
    s_done = 0;
  }
  __syncthreads();
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
      const int key = c2key[i];
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
  if (tid == 0) {
    meta->T = s_T;
    meta->need = s_need;
    meta->counted = 1;
    meta->resolved = 1;
  }
}

// Band entries above T, and equal to it, join their write chunks' counts: CTA r
// reads region r of the band list; lanes of a warp on the same chunk add once.
__global__ void __launch_bounds__(256) w_mark(const GridMeta* meta, const int* bkey,
                                              const uint32_t* bidx, const uint32_t* nbc,
                                              uint32_t rcap, uint32_t* cgt, uint32_t* ceq, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  meta = row_ws(meta, wsr);
  bkey = row_ws(bkey, wsr);
  bidx = row_ws(bidx, wsr);
  nbc = row_ws(nbc, wsr);
  cgt = row_ws(cgt, wsr);
  ceq = row_ws(ceq, wsr);
  const GridMeta m = *meta;
  if (!m.band || !m.resolved) return;
  const int lane = threadIdx.x & 31;
  const uint32_t nr = nbc[blockIdx.x];
  const size_t rb = static_cast<size_t>(blockIdx.x) * rcap;
  const int T = m.T;
  for (uint32_t i0 = (threadIdx.x & ~31u) * 4u; i0 < nr; i0 += 256u * 4u) {
    int key[4];
    uint32_t ch[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t i = i0 + 32u * q + lane;
      key[q] = i < nr ? (bkey[rb + i] & 0x7fffffff) : -1;
      ch[q] = i < nr ? static_cast<uint32_t>(bidx[rb + i] / kWCH) : 0xffffffffu;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const unsigned same = __match_any_sync(kFull, ch[q]);
      const unsigned bg = __ballot_sync(kFull, key[q] > T) & same;
      const unsigned be = __ballot_sync(kFull, key[q] == T) & same;
      if (ch[q] != 0xffffffffu && lane == __ffs(same) - 1) {
        if (bg) atomicAdd(&cgt[ch[q]], static_cast<uint32_t>(__popc(bg)));
        if (be) atomicAdd(&ceq[ch[q]], static_cast<uint32_t>(__popc(be)));
      }
    }
  }
}

// Exclusive prefix sums of the per-write-chunk counts, in two steps: each CTA
// of w_scan1 scans 1024 chunks' counts in place and writes their totals; w_scan2
// (one CTA) scans the totals.  The counts before chunk c are then
// cgt[c] + tg[c / 1024] (and ceq[c] + te[c / 1024]).
__global__ void __launch_bounds__(1024) w_scan1(uint32_t* cgt, uint32_t* ceq, uint32_t* tg,
                                                uint32_t* te, int64_t nwch, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  cgt = row_ws(cgt, wsr);
  ceq = row_ws(ceq, wsr);
  tg = row_ws(tg, wsr);
  te = row_ws(te, wsr);
  __shared__ uint32_t red[32];
  const int64_t c = static_cast<int64_t>(blockIdx.x) * 1024 + threadIdx.x;
  const uint32_t g = c < nwch ? cgt[c] : 0u, q = c < nwch ? ceq[c] : 0u;
  uint32_t sg, sq;
  const uint32_t xg = excl_scan_1024(g, red, &sg);
  const uint32_t xq = excl_scan_1024(q, red, &sq);
  if (c < nwch) {
    cgt[c] = xg;
    ceq[c] = xq;
  }
  if (threadIdx.x == 0) {
    tg[blockIdx.x] = sg;
    te[blockIdx.x] = sq;
  }
}

__global__ void __launch_bounds__(1024) w_scan2(uint32_t* tg, uint32_t* te, int nblocks, size_t wsr) {
  pdl_begin();
  pdl_end();  // light work: the next grid may be scheduled now
  tg = row_ws(tg, wsr);
  te = row_ws(te, wsr);
  __shared__ uint32_t red[32];
  uint32_t carry_g = 0, carry_q = 0;
  for (int b0 = 0; b0 < nblocks; b0 += 1024) {
    const int b = b0 + threadIdx.x;
    const uint32_t g = b < nblocks ? tg[b] : 0u, q = b < nblocks ? te[b] : 0u;
    uint32_t sg, sq;
    const uint32_t xg = excl_scan_1024(g, red, &sg);
    const uint32_t xq = excl_scan_1024(q, red, &sq);
    if (b < nblocks) {
      tg[b] = carry_g + xg;
      te[b] = carry_q + xq;
    }
    carry_g += sg;
    carry_q += sq;
  }
}

// w |= bit when a > b, or when a == b (one compare and one predicated OR).
__device__ __forceinline__ void or_if_gt(uint32_t& w, int a, int b, uint32_t bit) {
  asm("{\n .reg .pred p;\n setp.gt.s32 p, %1, %2;\n @p or.b32 %0, %0, %3;\n}"
      : "+r"(w)
      : "r"(a), "r"(b), "r"(bit));
}
__device__ __forceinline__ void or_if_eq(uint32_t& w, int a, int b, uint32_t bit) {
  asm("{\n .reg .pred p;\n setp.eq.s32 p, %1, %2;\n @p or.b32 %0, %0, %3;\n}"
      : "+r"(w)
      : "r"(a), "r"(b), "r"(bit));
}

// The payload in ascending index order, and the buffer updates, once T and
// need are known and the scan has the counts before each write chunk: one read
// of the row (x, s from err for error feedback, or x with d = x - g formed here
// for EF21).  Persistent CTAs over chunks of kWCH entries, double-buffered.
// Thread t's 32 entries give its words of entries above T and equal to T; ties
// are kept in index order while their rank in the row is below need; a block
// scan gives the positions, the kept columns are staged at them, and the
// payload leaves with coalesced stores.
template <int MODE>
__global__ void __launch_bounds__(kWT) g_write3(const float* xr, float* ar, int64_t L,
                                                int64_t nwch, int64_t k, int aligned,
                                                const GridMeta* meta, const uint32_t* cgt,
                                                const uint32_t* ceq, const uint32_t* tg,
                                                const uint32_t* te, float* vals, int32_t* idx,
                                                uint32_t spin_limit, unsigned* status, size_t wsr) {
  pdl_begin();
  xr += static_cast<int64_t>(blockIdx.y) * L;
  if (MODE != kPlain) ar += static_cast<int64_t>(blockIdx.y) * L;
  meta = row_ws(meta, wsr);
  cgt = row_ws(cgt, wsr);
  ceq = row_ws(ceq, wsr);
  tg = row_ws(tg, wsr);
  te = row_ws(te, wsr);
  vals += static_cast<int64_t>(blockIdx.y) * k;
  idx += static_cast<int64_t>(blockIdx.y) * k;
  constexpr int NW = kWT / 32;
  extern __shared__ __align__(16) float wbuf[];  // 2 x kWCH values, then kWCH staged columns
  uint16_t* cols = reinterpret_cast<uint16_t*>(wbuf + 2 * kWCH);
  __shared__ uint32_t rg[NW], re[NW];
  __shared__ uint64_t bars[2][NW];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (meta->band && meta->lmode) return;  // g_wlist writes the payload from the list
  const int T = meta->T;
  const uint32_t need = meta->need;
  if (aligned && warp == 0 && lane < NW) {
    mbar_init(&bars[0][lane], 1);
    mbar_init(&bars[1][lane], 1);
    fence_mbar_init();
  }
  __syncthreads();
  // the values ranked: s lives in err for error feedback
  const float* src = MODE == kEF ? ar : xr;
  const float* pre = MODE == kDelta ? ar : nullptr;
  int64_t c = blockIdx.x;
  if (aligned && warp == 0 && c < nwch) issue_chunk<NW, kWCH>(wbuf, src, pre, L, c, bars[0], lane);
  uint32_t par = 0;
  int b = 0;
  for (; c < nwch; c += gridDim.x, b ^= 1) {
    const int64_t cn = c + gridDim.x;
    if (aligned && warp == 0 && cn < nwch)
      issue_chunk<NW, kWCH>(wbuf + (b ^ 1) * kWCH, src, pre, L, cn, bars[b ^ 1], lane);
    const int64_t c0 = c * kWCH;
    const int n = static_cast<int>(min64(kWCH, L - c0));
    float* cb = wbuf + b * kWCH;
    const int pb = 1024 * warp;
    if (pb < n) {
      if (aligned) {
        if (!mbar_wait_bounded(&bars[b][warp], (par >> b) & 1u, spin_limit, status))
          mbar_wait_bounded(&bars[b][warp], (par >> b) & 1u, kDrainPolls, nullptr);
        if (MODE == kDelta) {
          const int nq = min(1024, n - pb) / 4;
          float4* c4 = reinterpret_cast<float4*>(cb + pb);
          const float4* a4 = reinterpret_cast<const float4*>(ar + c0 + pb);
          for (int q = lane; q < nq; q += 32) {
            const float4 xv = c4[q];
            const float4 av = a4[q];
            c4[q] = make_float4(fsub(xv.x, av.x), fsub(xv.y, av.y), fsub(xv.z, av.z),
                                fsub(xv.w, av.w));
          }
          fence_proxy_async_smem();  // these stores before the buffer's next bulk copy
        }
      } else {
        for (int e = pb + lane; e < min(pb + 1024, n); e += 32)
          cb[e] = value_at<MODE>(xr, ar, c0 + e);
      }
      __syncwarp();
    }
    par ^= 1u << b;
    // words of this thread's 32 entries: above T, and equal to T
    const int e0 = 32 * tid;
    const int nv = max(0, min(32, n - e0));
    const uint32_t vmask = nv >= 32 ? 0xffffffffu : ((1u << nv) - 1u);
    uint32_t gw = 0, ew = 0;
    if (nv > 0) {
      const float4* my4 = reinterpret_cast<const float4*>(cb + e0);
      if (need == 0) {
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const float4 v = my4[(u + lane) & 7];  // 8 consecutive lanes on 8 bank groups
          or_if_gt(gw, mag_key(v.x), T, 1u << (4 * u + 0));
          or_if_gt(gw, mag_key(v.y), T, 1u << (4 * u + 1));
          or_if_gt(gw, mag_key(v.z), T, 1u << (4 * u + 2));
          or_if_gt(gw, mag_key(v.w), T, 1u << (4 * u + 3));
        }
      } else {
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const float4 v = my4[(u + lane) & 7];
          const int k0 = mag_key(v.x), k1 = mag_key(v.y), k2 = mag_key(v.z), k3 = mag_key(v.w);
          or_if_gt(gw, k0, T, 1u << (4 * u + 0));
          or_if_gt(gw, k1, T, 1u << (4 * u + 1));
          or_if_gt(gw, k2, T, 1u << (4 * u + 2));
          or_if_gt(gw, k3, T, 1u << (4 * u + 3));
          or_if_eq(ew, k0, T, 1u << (4 * u + 0));
          or_if_eq(ew, k1, T, 1u << (4 * u + 1));
          or_if_eq(ew, k2, T, 1u << (4 * u + 2));
          or_if_eq(ew, k3, T, 1u << (4 * u + 3));
        }
      }
      const uint32_t rot = 4u * static_cast<uint32_t>(lane & 7);
      gw = __funnelshift_l(gw, gw, rot) & vmask;
      ew = __funnelshift_l(ew, ew, rot) & vmask;
    }
    const uint32_t ng = __popc(gw), ne = __popc(ew);
    const uint32_t gi = warp_inclusive_scan(ng, lane);
    const uint32_t ei = warp_inclusive_scan(ne, lane);
    if (lane == 31) {
      rg[warp] = gi;
      re[warp] = ei;
    }
    __syncthreads();
    uint32_t gp = gi - ng, ep = ei - ne, G = 0, E = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      gp += (w < warp) ? rg[w] : 0u;
      ep += (w < warp) ? re[w] : 0u;
      G += rg[w];
      E += re[w];
    }
    // entries above T and equal to T before this chunk
    const uint32_t gb = cgt[c] + tg[c >> 10], eb = ceq[c] + te[c >> 10];
    // ties kept: those whose rank among the row's ties is below need
    const uint32_t room = need > eb ? need - eb : 0u;  // ties this chunk may still take
    uint32_t kw = gw;
    if (ne && room > ep) {
      uint32_t take = min(room - ep, ne);
      uint32_t w = ew;
      while (take--) {
        kw |= w & (~w + 1u);
        w &= w - 1;
      }
    }
    // positions: kept entries before this chunk, then before this thread in it
    const uint64_t base = static_cast<uint64_t>(gb) + min(eb, need);
    uint32_t p = gp + min(ep, room);
    const uint32_t total = G + min(E, room);
    while (kw) {
      const int j = __ffs(kw) - 1;
      kw &= kw - 1;
      cols[p++] = static_cast<uint16_t>(e0 + j);
    }
    __syncthreads();
    // four kept entries a thread at a time: the state loads of EF21 go out
    // together (the kept columns are distinct, so no store aliases a load)
    for (uint32_t i0 = tid; i0 < total; i0 += 4 * kWT) {
      int e[4];
      float v[4], g[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t i = i0 + q * kWT;
        e[q] = i < total ? cols[i] : 0;
        v[q] = cb[e[q]];
        g[q] = (MODE == kDelta && i < total) ? ar[c0 + e[q]] : 0.0f;
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t i = i0 + q * kWT;
        if (i >= total) break;
        const uint64_t pos = base + i;
        if (pos < static_cast<uint64_t>(k)) {
          vals[pos] = v[q];
          idx[pos] = static_cast<int32_t>(c0 + e[q]);
        }
        if (MODE == kEF) ar[c0 + e[q]] = 0.0f;               // err' = s - C(s): +0 where sent
        if (MODE == kDelta) ar[c0 + e[q]] = fadd(g[q], v[q]);  // g' = g + d where sent
      }
    }
    __syncthreads();  // buffer b, the staged columns and rg / re free again
  }
}

// List mode: the payload from the list instead of a second read of the row.
// Warp w takes pass-1 chunks c = w, w + W, ...; chunk c's entries (every entry
// >= t_lo, in index order) are the segment of region c % G1 that pass 1
// recorded.  Kept: above T, and ties while their rank among the row's ties is
// below need; positions from the scanned per-write-chunk counts (a pass-1 chunk
// is write chunks 2c and 2c + 1).  Error feedback: +0 into err at the kept
// entries (err holds s); EF21: state + d there.
template <int MODE>
__global__ void __launch_bounds__(256) g_wlist(float* ar, int64_t nchunks, uint32_t g1,
                                               uint32_t rcap, int64_t k, const GridMeta* meta,
                                               const int* bkey, const uint32_t* bidx,
                                               const uint32_t* seg, const uint32_t* segn,
                                               const uint32_t* cgt, const uint32_t* ceq,
                                               const uint32_t* tg, const uint32_t* te,
                                               float* vals, int32_t* idx, int64_t L, size_t wsr) {
  pdl_begin();
  if (MODE != kPlain) ar += static_cast<int64_t>(blockIdx.y) * L;
  meta = row_ws(meta, wsr);
  bkey = row_ws(bkey, wsr);
  bidx = row_ws(bidx, wsr);
  seg = row_ws(seg, wsr);
  segn = row_ws(segn, wsr);
  cgt = row_ws(cgt, wsr);
  ceq = row_ws(ceq, wsr);
  tg = row_ws(tg, wsr);
  te = row_ws(te, wsr);
  vals += static_cast<int64_t>(blockIdx.y) * k;
  idx += static_cast<int64_t>(blockIdx.y) * k;
  if (!(meta->band && meta->lmode)) return;
  const int T = meta->T;
  const uint32_t need = meta->need;
  const int lane = threadIdx.x & 31;
  const unsigned lt = lanemask_lt();
  const int64_t nw = static_cast<int64_t>(gridDim.x) * (blockDim.x / 32);
  for (int64_t c = static_cast<int64_t>(blockIdx.x) * (blockDim.x / 32) + (threadIdx.x >> 5);
       c < nchunks; c += nw) {
    const int64_t wc = 2 * c;
    const uint32_t gb = cgt[wc] + tg[wc >> 10], eb = ceq[wc] + te[wc >> 10];
    uint64_t pos = static_cast<uint64_t>(gb) + min(eb, need);
    uint32_t eq_seen = eb;
    const size_t rb = static_cast<size_t>(c % g1) * rcap + seg[c];
    const uint32_t n = segn[c];
    for (uint32_t i0 = 0; i0 < n; i0 += 32) {
      const uint32_t i = i0 + lane;
      const bool in = i < n;
      const int bits = in ? bkey[rb + i] : 0;
      const uint32_t col = in ? bidx[rb + i] : 0u;
      const int key = bits & 0x7fffffff;
      const bool eq = in && key == T;
      const unsigned be = __ballot_sync(kFull, eq);
      const bool kp = (in && key > T) || (eq && eq_seen + __popc(be & lt) < need);
      eq_seen += __popc(be);
      const unsigned bk = __ballot_sync(kFull, kp);
      if (kp) {
        const uint64_t p = pos + __popc(bk & lt);
        const float v = __int_as_float(bits);
        if (p < static_cast<uint64_t>(k)) {
          vals[p] = v;
          idx[p] = static_cast<int32_t>(col);
        }
        if (MODE == kEF) ar[col] = 0.0f;                   // err' = s - C(s): +0 where sent
        if (MODE == kDelta) ar[col] = fadd(ar[col], v);   // g' = g + d where sent
      }
      pos += __popc(bk);
    }
  }
}

// Persistent grids: the CTAs that fit on the GPU (and no more than the band
// list has regions).
template <class K>
unsigned persistent_grid(K kernel, int threads, int smem, int num_sms, int64_t nchunks, int64_t batch) {
  const int occ = resident_blocks(kernel, threads, smem);
  const int64_t fit = (static_cast<int64_t>(num_sms) * occ + batch - 1) / batch;  // per row
  const int64_t g = min64(min64(fit, kMaxBandCtas), nchunks);
  return static_cast<unsigned>(max64(g, 1));
}

template <int MODE>
cudaError_t run_grid(const TopkGridArgs& a, int num_sms, cudaStream_t s) {
  const int64_t L = a.L;
  const int64_t nchunks = (L + kCH - 1) / kCH;
  const int64_t nwch = (L + kWCH - 1) / kWCH;
  const int nblk = static_cast<int>((nwch + 1023) / 1024);
  if (nchunks > 0x7fffffffLL) return cudaErrorInvalidValue;
  const int64_t B = grid_batch(a.rows, L);
  const size_t wsr = align256(ws_bytes_for(L, a.k));  // one row's workspace slice
  const WsLayout w = layout(a.ws, L, a.k, nchunks);     // the first row's
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  const int aligned = (L % 4 == 0) && al16(a.x) && (MODE == kPlain || al16(a.aux));
  constexpr int kP1Smem = 2 * kCH * 4;             // two chunk buffers
  constexpr int kWSmem = 2 * kWCH * 4 + kWCH * 2;  // two chunk buffers and the staged columns
  auto p1 = w_pass1<MODE>;
  auto wr = g_write3<MODE>;
  cudaError_t err = ensure_dynamic_smem(p1, kP1Smem);
  if (err == cudaSuccess) err = ensure_dynamic_smem(wr, kWSmem);
  if (err != cudaSuccess) return err;
  // grids per row (the launches below take B rows, blockIdx.y the row)
  const unsigned g1 = persistent_grid(p1, kGT, kP1Smem, num_sms, nchunks, B);
  const unsigned gw = persistent_grid(wr, kWT, kWSmem, num_sms, nwch, B);
  const uint32_t rcap = w.bcap / g1;  // band-list region of one pass-1 CTA
  const int ns = sample_count(L);
  // the list-mode write: a warp per pass-1 chunk
  const unsigned gl = static_cast<unsigned>(
      max64(1, min64((nchunks + 7) / 8, (static_cast<int64_t>(num_sms) * 8 + B - 1) / B)));
  // the multi-pass kernels: a fixed grid striding over the chunks
  const unsigned gm = static_cast<unsigned>(
      max64(1, min64(nwch, (static_cast<int64_t>(num_sms) * 8 + B - 1) / B)));
  // launches with programmatic dependent launch (the light kernels let the next
  // grid be scheduled as soon as they start); the first error ends the call
  auto go = [&](auto kernel, dim3 grid, int threads, int smem, auto... args) {
    if (err == cudaSuccess) err = launch_kernel(kernel, grid, dim3(threads), smem, s, 0u, args...);
  };
  for (int64_t r0 = 0; r0 < a.rows && err == cudaSuccess; r0 += B) {
    const unsigned nb = static_cast<unsigned>(min64(B, a.rows - r0));
    const float* xr = a.x + r0 * L;
    float* ar = (MODE != kPlain) ? a.aux + r0 * L : nullptr;
    float* vr = a.vals + r0 * a.k;
    int32_t* ir = a.idx + r0 * a.k;
    auto G = [nb](unsigned x) { return dim3(x, nb); };
    go(g_init, G(1), 1024, 0, w.meta, w.hist, w.shist, w.fhist, nchunks, L, a.k, wsr);
    // the band path
    go(w_sample<MODE>, G(static_cast<unsigned>(ns / 1024)), 1024, 0, xr, ar, L, w.meta, w.shist, ns, wsr);
    go(w_spick, G(1), 1024, 0, L, a.k, w.meta, w.shist, list_eligible(L, a.k) ? 1 : 0, w.bcap, ns, wsr);
    go(p1, G(g1), kGT, kP1Smem, xr, ar, L, nchunks, aligned, w.meta, w.cgt, w.ceq, w.bkey, w.bidx,
       rcap, w.nbc, w.seg, w.segn, w.fhist, a.spin_limit, a.status, wsr);
    go(w_pick1, G(1), 32, 0, w.meta, w.fhist, a.k, wsr);
    go(w_bin2, G(g1), 256, 0, w.meta, w.bkey, w.nbc, rcap, w.c2key, w.c2cap, wsr);
    go(w_select2, G(1), 1024, 0, w.meta, w.c2key, w.c2cap, wsr);
    go(w_mark, G(g1), 256, 0, w.meta, w.bkey, w.bidx, w.nbc, rcap, w.cgt, w.ceq, wsr);
    // the multi-pass path (each kernel returns at once when the band path resolved)
    go(g_sample<MODE>, G(1), kGT, 0, xr, ar, L, a.k, w.meta, wsr);
    go(g_hist<MODE>, G(gm), kGT, 0, xr, ar, L, w.meta, w.hist, 1, wsr);
    go(g_pick, G(1), kGT, 0, w.meta, w.hist, wsr);
    for (int i = 0; i < kMaxRounds; ++i) {
      go(g_hist<MODE>, G(gm), kGT, 0, xr, ar, L, w.meta, w.hist, 0, wsr);
      go(g_pick, G(1), kGT, 0, w.meta, w.hist, wsr);
    }
    go(g_count<MODE>, G(gm), kGT, 0, xr, ar, L, w.meta, w.cgt, w.ceq, w.ckey, w.cidx, wsr);
    go(g_select, G(1), 1024, 0, w.meta, w.cgt, w.ceq, w.ckey, w.cidx, wsr);
    // both paths: positions per write chunk, then the payload (the second read)
    go(w_scan1, G(static_cast<unsigned>(nblk)), 1024, 0, w.cgt, w.ceq, w.tg, w.te, nwch, wsr);
    go(w_scan2, G(1), 1024, 0, w.tg, w.te, nblk, wsr);
    go(wr, G(gw), kWT, kWSmem, xr, ar, L, nwch, a.k, aligned, w.meta, w.cgt, w.ceq, w.tg, w.te, vr,
       ir, a.spin_limit, a.status, wsr);
    go(g_wlist<MODE>, G(gl), 256, 0, ar, nchunks, g1, rcap, a.k, w.meta, w.bkey, w.bidx, w.seg,
       w.segn, w.cgt, w.ceq, w.tg, w.te, vr, ir, L, wsr);
  }
  return err;
}

}  // namespace

size_t topk_grid_workspace_bytes(int64_t rows, int64_t L, int64_t k) {
  return static_cast<size_t>(grid_batch(rows, L)) * align256(ws_bytes_for(L, k));
}

cudaError_t launch_topk_grid(int mode, const TopkGridArgs& a, int num_sms, cudaStream_t s) {
  if (a.rows <= 0) return cudaSuccess;
  switch (mode) {
    case kPlain: return run_grid<kPlain>(a, num_sms, s);
    case kEF: return run_grid<kEF>(a, num_sms, s);
    case kDelta: return run_grid<kDelta>(a, num_sms, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace mpc
